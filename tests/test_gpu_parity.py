"""GPU parity: libwf (through its C ABI) against the fp64 CPU oracle on the
same seeded inputs.

Bars: stored pyramid bit-exact; selected indices (every scale) bit-exact on
planted-ladder inputs; outputs within fp32 max-abs 1e-5, or bf16 max-abs 2e-2
and rel-L2 1e-2.  Unplanted inputs (where near-ties may make several answers
correct) are checked for a valid Top-K at every scale instead.
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import LibRun, assert_close_out, eps_valid, f64, make_layer, oracle_unit
from paper_2606_00724_gb300 import synth

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)


def _check_units(w, batch, run, units):
    bf16 = w.dtype == "bf16"
    for u in units:
        b, h = divmod(u, w.heads)
        Q, K, V, Kg, Vg = (f64(t[b, h]) for t in (batch.Q, batch.K, batch.V, batch.Kg, batch.Vg))
        pyr, mu0, sets, O = oracle_unit(Q, K, V, Kg, Vg, w.levels, w.keep, bf16)
        assert np.array_equal(run.pyramid(u), pyr.astype(np.float64)), f"pyramid unit {u}"
        gsets = run.level_sets(u)
        for lev in range(w.levels, -1, -1):
            assert np.array_equal(gsets[lev], sets[lev]), f"unit {u} scale {lev}"
        tgt = batch.targets[u]
        if tgt is not None:
            assert np.array_equal(run.idx[u].cpu().numpy(), tgt[0].cpu().numpy())
        assert np.array_equal(run.idx[u].cpu().numpy(), mu0)
        assert_close_out(f64(run.O[b, h]), O, batch.Q.dtype)


@pytest.mark.parametrize("cfg", ["c1", "c2"])
def test_small_configs_all_units(cfg):
    w, batch = make_layer(cfg)
    run = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).run()
    torch.cuda.synchronize()
    _check_units(w, batch, run, range(w.units))


@pytest.mark.parametrize("cfg", ["c3", "c4", "c5"])
def test_full_size_sampled_units(cfg):
    # Full-size layer through the per-stage kernels (wf_dwt_build, wf_filter,
    # wf_sparse_attn; the fused kernel that the benchmark times is checked in
    # test_gpu_step.py); the oracle checks a few units (first, last, one in
    # between).
    w = synth.WORKLOADS[cfg]
    units = [0, w.units // 2 + 3, w.units - 1]
    w, batch = make_layer(cfg, units=None)
    run = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).run()
    torch.cuda.synchronize()
    _check_units(w, batch, run, units)
    # Every unit's planted answer (no oracle needed).
    idx = run.idx.cpu().numpy()
    for u in range(w.units):
        assert np.array_equal(idx[u], batch.targets[u][0].cpu().numpy()), f"unit {u}"


def _rand_case(seed, B, H, n, d, q, ng, dtype, bshd=False, device="cuda"):
    g = torch.Generator(device="cpu").manual_seed(seed)
    def r(rows):
        x = torch.randn(B, rows, H, d, generator=g) if bshd else torch.randn(B, H, rows, d, generator=g)
        x = x.to(dtype).to(device)
        return x.transpose(1, 2) if bshd else x
    return r(q), r(n), r(n), r(ng) if ng else None, r(ng) if ng else None


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("n,d,q,ng,L,keep,bshd", [
    (256, 64, 5, 3, 3, [37, 19, 20, 24], False),       # ragged tiles, odd final k (trim)
    (512, 128, 32, 0, 2, [60, 30, 77], True),           # BSHD strides, no generation rows
    (96, 64, 1, 1, 1, [17, 9], False),                 # single query, L = 1, trim
    (2048, 128, 64, 32, 4, [256, 128, 128, 128, 128], False),  # 64 query rows
    (128, 64, 7, 2, 3, [128, 64, 32, 16], False),      # keep everything (k = n)
    (64, 128, 3, 0, 6, [1, 1, 1, 1, 1, 1, 1], False),  # deepest pyramid, k = 1
    (65536, 128, 32, 32, 3, [3000, 4000, 5000, 6000], False),  # lists of 8192 / 12000 / 10000 / 8000: the
                                                               # Top-K's register and memory paths
])
def test_random_shapes(dtype, n, d, q, ng, L, keep, bshd):
    B, H = 2, 3
    Q, K, V, Kg, Vg = _rand_case(n + d + q + L, B, H, n, d, q, ng, dtype, bshd)
    run = LibRun(Q, K, V, Kg, Vg, L, keep).run()
    torch.cuda.synchronize()
    for u in range(B * H):
        b, h = divmod(u, H)
        Qn, Kn, Vn = f64(Q[b, h]), f64(K[b, h]), f64(V[b, h])
        Kgn = f64(Kg[b, h]) if ng else None
        Vgn = f64(Vg[b, h]) if ng else None
        pyr = oracle.haar_pyramid_spec32(Kn.astype(np.float32), L, dtype == torch.bfloat16)
        assert np.array_equal(run.pyramid(u), pyr.astype(np.float64))
        gsets = run.level_sets(u)
        eps_valid(Qn, pyr.astype(np.float64), Kn, n, L, keep, gsets)
        idx = run.idx[u].cpu().numpy()
        assert np.all(np.diff(idx) > 0) and idx.min() >= 0 and idx.max() < n
        # Attention on the GPU's own selection (independent of near-ties).
        O = oracle.sparse_attn(Qn, Kn, Vn, idx, Kgn, Vgn)
        assert_close_out(f64(run.O[b, h]), O, dtype)
        if keep[0] == n:
            assert np.array_equal(idx, np.arange(n))


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_attention_full_selection_is_dense(dtype):
    # k = n: the sparse attention equals dense cached attention over [K; Kg].
    B, H, n, d, q, ng = 1, 2, 192, 128, 16, 8
    Q, K, V, Kg, Vg = _rand_case(7, B, H, n, d, q, ng, dtype)
    run = LibRun(Q, K, V, Kg, Vg, 1, [n, n // 2])
    idx = torch.arange(n, dtype=torch.int32, device="cuda").repeat(B * H, 1)
    run.attn(idx)
    torch.cuda.synchronize()
    for h in range(H):
        want = oracle.attention(f64(Q[0, h]), np.vstack([f64(K[0, h]), f64(Kg[0, h])]),
                                np.vstack([f64(V[0, h]), f64(Vg[0, h])]))
        assert_close_out(f64(run.O[0, h]), want, dtype)


def test_attention_unsorted_indices_and_scale():
    B, H, n, d, q, ng = 1, 1, 300, 64, 4, 0
    Q, K, V, _, _ = _rand_case(8, B, H, n, d, q, ng, torch.float32)
    run = LibRun(Q, K, V, None, None, 1, [10, 5])
    sel = torch.tensor([[299, 3, 150, 7, 8, 42, 0]], dtype=torch.int32, device="cuda")
    run.attn(sel, scale=0.3)
    torch.cuda.synchronize()
    Qn = f64(Q[0, 0]) * 0.3 * np.sqrt(d)  # oracle uses 1/sqrt(d): fold the scale into Q
    want = oracle.sparse_attn(Qn, f64(K[0, 0]), f64(V[0, 0]), sel[0].cpu().numpy())
    assert_close_out(f64(run.O[0, 0]), want, torch.float32)


def test_step_matches_separate_calls():
    from paper_2606_00724_gb300 import wf
    w, batch = make_layer("c2")
    a = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).run()
    idx = torch.empty_like(a.idx)
    O = torch.empty_like(a.O)
    coeffs = torch.empty_like(a.coeffs)
    ws = torch.zeros(wf.wf_step_workspace_bytes(batch.Q, batch.K, w.levels, w.keep, w.ng), dtype=torch.uint8,
                     device="cuda")
    wf.wf_step(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, coeffs, True, w.levels, w.keep, idx, O, ws)
    torch.cuda.synchronize()
    assert torch.equal(coeffs, a.coeffs)
    assert torch.equal(idx, a.idx)
    # wf_step runs the fused kernel (bf16 P on the tensor cores): same
    # indices, outputs within the bf16 tolerance of the per-stage kernels.
    assert_close_out(f64(O), f64(a.O), torch.bfloat16)
    # Second step re-using the cached pyramid (no refresh) gives the same answer.
    O2 = torch.empty_like(O)
    wf.wf_step(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, coeffs, False, w.levels, w.keep, idx, O2, ws)
    torch.cuda.synchronize()
    assert torch.equal(O2, O)
