"""Pins for the oracle's attention (Eq. 1 / Eq. 3 form) and the final sparse
step of Algorithm 1 (gather K[mu0], V[mu0], append the generation rows)."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F


def rng(seed):
    return np.random.default_rng(seed)


def test_attention_matches_torch_sdpa(orc):
    r = rng(0)
    Q = r.standard_normal((7, 16))
    K = r.standard_normal((50, 16))
    V = r.standard_normal((50, 16))
    ref = F.scaled_dot_product_attention(torch.from_numpy(Q)[None], torch.from_numpy(K)[None],
                                         torch.from_numpy(V)[None])[0].numpy()
    assert np.abs(orc.attention(Q, K, V) - ref).max() <= 1e-13


def test_single_key_returns_its_value(orc):
    r = rng(1)
    Q = r.standard_normal((3, 8))
    V = r.standard_normal((1, 8))
    O = orc.attention(Q, r.standard_normal((1, 8)), V)
    assert np.abs(O - V).max() <= 1e-15


def test_equal_keys_average_values(orc):
    r = rng(2)
    Q = r.standard_normal((3, 8))
    K = np.tile(r.standard_normal(8), (5, 1))
    V = r.standard_normal((5, 8))
    assert np.abs(orc.attention(Q, K, V) - V.mean(0)).max() <= 1e-14


def test_full_selection_is_dense_attention(orc):
    # k = n: the sparse set is the whole prompt cache plus the generation rows,
    # i.e. the dense cached attention of Eq. 3 over [K; K_g].
    r = rng(3)
    n, ng, d = 40, 6, 8
    Q = r.standard_normal((4, d))
    K, V = r.standard_normal((n, d)), r.standard_normal((n, d))
    Kg, Vg = r.standard_normal((ng, d)), r.standard_normal((ng, d))
    O = orc.sparse_attn(Q, K, V, np.arange(n), Kg, Vg)
    ref = F.scaled_dot_product_attention(torch.from_numpy(Q)[None], torch.from_numpy(np.vstack([K, Kg]))[None],
                                         torch.from_numpy(np.vstack([V, Vg]))[None])[0].numpy()
    assert np.abs(O - ref).max() <= 1e-13


def test_sparse_gather_and_order(orc):
    # The sparse step attends exactly to K[mu0] and the generation rows; the
    # order of the gathered rows does not matter.
    r = rng(4)
    n, d = 64, 8
    Q = r.standard_normal((4, d))
    K, V = r.standard_normal((n, d)), r.standard_normal((n, d))
    Kg, Vg = r.standard_normal((3, d)), r.standard_normal((3, d))
    mu0 = np.array([3, 4, 17, 40, 41, 63])
    O = orc.sparse_attn(Q, K, V, mu0, Kg, Vg)
    ref = F.scaled_dot_product_attention(torch.from_numpy(Q)[None], torch.from_numpy(np.vstack([K[mu0], Kg]))[None],
                                         torch.from_numpy(np.vstack([V[mu0], Vg]))[None])[0].numpy()
    assert np.abs(O - ref).max() <= 1e-13
    O2 = orc.sparse_attn(Q, K, V, mu0[::-1].copy(), Kg, Vg)
    assert np.abs(O - O2).max() <= 1e-14
    # No generation rows.
    O3 = orc.sparse_attn(Q, K, V, mu0)
    ref3 = F.scaled_dot_product_attention(torch.from_numpy(Q)[None], torch.from_numpy(K[mu0])[None],
                                          torch.from_numpy(V[mu0])[None])[0].numpy()
    assert np.abs(O3 - ref3).max() <= 1e-13


def test_bad_arguments_raise(orc):
    with pytest.raises(ValueError):
        orc.sparse_attn(np.zeros((1, 4)), np.zeros((4, 4)), np.zeros((4, 4)), np.zeros(0, dtype=np.int32))
