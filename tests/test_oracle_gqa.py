"""Pins for the oracle's grouped-query (GQA) filtering and attention: the KV
head's importance is the sum of Eq. 8 over its group's query heads, checked
against an independent numpy softmax, exhaustive search, the single-head
case, head-order invariance, a planted answer on the Dream-shaped workload,
and torch's dense grouped-query attention when everything is kept."""
import itertools
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2606_00724_gb300 import synth


def _softmax_weights(Qg, rows):
    # Eq. 7 row softmax of one head's queries, Eq. 8 column sum (numpy, fp64).
    s = Qg @ rows.T / math.sqrt(Qg.shape[1])
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p /= p.sum(axis=1, keepdims=True)
    return p.sum(axis=0)


def test_group_weights_are_the_sum_over_heads():
    r = np.random.default_rng(3)
    G, q, d, m = 3, 4, 16, 9
    Qh = r.standard_normal((G, q, d))
    rows = r.standard_normal((m, d))
    W = oracle.skim_weights(Qh.reshape(-1, d), rows)
    want = sum(_softmax_weights(Qh[g], rows) for g in range(G))
    assert np.allclose(W, want, rtol=0, atol=1e-12)
    assert abs(W.sum() - G * q) < 1e-12          # every query row's softmax sums to 1


def _brute_force_sets(Qh, pyr, n, L, keep):
    # Exhaustive search per scale: the kept set is the keep[b]-subset of the
    # candidates with the largest total group weight.
    d = Qh.shape[2]
    sets = {}
    cand = np.arange(n >> L)
    for b in range(L, 0, -1):
        rows = oracle.level(pyr, n, b)[cand]
        W = sum(_softmax_weights(Qh[g], rows) for g in range(Qh.shape[0]))
        best = max(itertools.combinations(range(cand.size), int(keep[b])), key=lambda s: W[list(s)].sum())
        sets[b] = np.sort(cand[list(best)])
        cand = np.stack([2 * sets[b], 2 * sets[b] + 1], 1).reshape(-1)
    return sets, cand


@pytest.mark.parametrize("seed", range(4))
def test_group_filter_brute_force(seed):
    r = np.random.default_rng(10 + seed)
    G, q, d, n, L = 3, 2, 8, 32, 2
    keep = np.array([6, 3, 4], dtype=np.int32)  # keep[0] = 2 keep[1]: no trim
    Qh = r.standard_normal((G, q, d))
    K = r.standard_normal((n, d))
    pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), L, False).astype(np.float64)
    mu0, sets = oracle.filter_gqa(Qh, pyr, K, n, L, keep, want_sets=True)
    want, cand = _brute_force_sets(Qh, pyr, n, L, keep)
    for b in range(L, 0, -1):
        assert np.array_equal(sets[b], want[b]), b
    assert np.array_equal(mu0, np.sort(cand))


def test_group_of_one_is_the_single_head_filter():
    r = np.random.default_rng(7)
    q, d, n, L = 8, 32, 256, 3
    keep = oracle.default_schedule(n, L, 40)
    Q = r.standard_normal((q, d))
    K = r.standard_normal((n, d))
    pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), L, False)
    a = oracle.filter_gqa(Q[None], pyr, K, n, L, keep, want_sets=True)
    b = oracle.filter(Q, pyr, K, n, L, keep, want_sets=True)
    assert np.array_equal(a[0], b[0])
    for lev in range(L + 1):
        assert np.array_equal(a[1][lev], b[1][lev])


def test_head_order_does_not_matter():
    r = np.random.default_rng(8)
    G, q, d, n, L = 4, 3, 32, 512, 3
    keep = oracle.default_schedule(n, L, 51)
    Qh = r.standard_normal((G, q, d))
    K = r.standard_normal((n, d))
    pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), L, False)
    a = oracle.filter_gqa(Qh, pyr, K, n, L, keep)
    b = oracle.filter_gqa(Qh[::-1, ::-1].copy(), pyr, K, n, L, keep)
    assert np.array_equal(a, b)


def test_planted_ladder_dream_shape():
    # Dream-7B head layout (7 query heads per KV head): the planted answer
    # is what the group filter finds at every scale.
    w = synth.WORKLOADS["g1"]
    dt = synth.storage_dtype(w)
    u = synth.make_unit(w, 1, w.heads - 1, planted=True, cfg="g1")
    assert u.Q.shape == (w.group * w.q, w.head_dim)
    Qh = u.Q.to(dt).float().numpy().reshape(w.group, w.q, w.head_dim)
    K = u.K.to(dt).float().numpy()
    pyr = oracle.haar_pyramid_spec32(K, w.levels, True)
    mu0, sets = oracle.filter_gqa(Qh, pyr, K, w.n, w.levels, np.array(w.keep), want_sets=True)
    for b, tgt in u.targets.items():
        assert np.array_equal(sets[b], tgt.numpy()), b
    assert np.array_equal(mu0, u.targets[0].numpy())


def test_keep_everything_is_dense_grouped_attention():
    r = np.random.default_rng(9)
    G, q, d, n, ng = 3, 5, 32, 64, 4
    Qh = r.standard_normal((G, q, d))
    K, V = r.standard_normal((n, d)), r.standard_normal((n, d))
    Kg, Vg = r.standard_normal((ng, d)), r.standard_normal((ng, d))
    O = oracle.sparse_attn_gqa(Qh, K, V, np.arange(n, dtype=np.int32), Kg, Vg)
    Kall = torch.from_numpy(np.concatenate([K, Kg]))[None, None]
    Vall = torch.from_numpy(np.concatenate([V, Vg]))[None, None]
    want = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(Qh)[None], Kall, Vall,
                                                            enable_gqa=True)[0].numpy()
    assert np.allclose(O, want, rtol=0, atol=1e-12)
