"""GPU parity of the generic-basis path (Eq. 6 / Eq. 11 with Haar or db2,
periodized): wf_wavelet_approx against the oracle's fp32 storage rule bit
for bit (whole prompt and gathered candidate blocks), the Haar case against
the stored pyramid and wf_filter, and wf_filter_wavelet's indices against
the oracle's literal filter on planted inputs (every scale, bit-exact), and
wf_step_wavelet's indices and output against the oracle.  For bf16 keys with
head_dim 128 and one query head per key head both calls run the fused
kernel once per scale."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from helpers import LibRun, assert_close_out, f64
from paper_2606_00724_gb300 import synth, wf

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)

BASES = {"haar": (wf.WF_WAVELET_HAAR, oracle.HAAR), "db2": (wf.WF_WAVELET_DB2, oracle.DB2)}


def _keys(seed, B, H, n, d, dtype, bshd):
    g = torch.Generator(device="cpu").manual_seed(seed)
    if bshd:
        return torch.randn(B, n, H, d, generator=g).to(dtype).cuda().transpose(1, 2)
    return torch.randn(B, H, n, d, generator=g).to(dtype).cuda()


def _unit_keys(K, u):
    B, H = K.shape[:2]
    return K[u // H, u % H].float().cpu().numpy()


@pytest.mark.parametrize("basis", ["haar", "db2"])
@pytest.mark.parametrize("dtype,d,n,level,bshd", [
    (torch.bfloat16, 128, 4096, 4, False),
    (torch.bfloat16, 128, 2048, 1, True),
    (torch.float32, 64, 1024, 3, False),
    (torch.bfloat16, 64, 8192, 6, False),
    (torch.float32, 128, 256, 8, True),
])
def test_approx_whole_prompt(basis, dtype, d, n, level, bshd):
    wv, ov = BASES[basis]
    B, H = 2, 3
    K = _keys(n + level, B, H, n, d, dtype, bshd)
    m = n >> level
    out = torch.empty(B, H, m, d, dtype=dtype, device="cuda")
    wf.wf_wavelet_approx(K, level, wv, out)
    torch.cuda.synchronize()
    for u in (0, B * H - 1):
        want = oracle.wavelet_approx_spec32(_unit_keys(K, u), ov, level, dtype == torch.bfloat16)
        got = out[u // H, u % H].float().cpu().numpy()
        assert np.array_equal(got, want), f"unit {u}"


@pytest.mark.parametrize("basis", ["haar", "db2"])
@pytest.mark.parametrize("dtype,level,m", [(torch.bfloat16, 3, 100), (torch.float32, 2, 7), (torch.bfloat16, 1, 1),
                                          (torch.bfloat16, 5, 64)])
def test_approx_gathered_blocks(basis, dtype, level, m):
    # Eq. 11: the transform of the concatenated blocks of a candidate list
    # (periodic over the gathered sequence, not the prompt).
    wv, ov = BASES[basis]
    B, H, n, d = 1, 4, 4096, 128
    K = _keys(7 * m + level, B, H, n, d, dtype, False)
    r = np.random.default_rng(m + level)
    cand = np.stack([np.sort(r.choice(n >> level, m, replace=False)) for _ in range(B * H)]).astype(np.int32)
    cand_t = torch.from_numpy(cand).cuda()
    out = torch.empty(B, H, m, d, dtype=dtype, device="cuda")
    wf.wf_wavelet_approx(K, level, wv, out, cand=cand_t)
    torch.cuda.synchronize()
    for u in range(B * H):
        toks = np.concatenate([np.arange(c << level, (c + 1) << level) for c in cand[u]])
        want = oracle.wavelet_approx_spec32(_unit_keys(K, u)[toks], ov, level, dtype == torch.bfloat16)
        assert np.array_equal(out[u // H, u % H].float().cpu().numpy(), want), f"unit {u}"


def test_haar_whole_prompt_is_the_pyramid_level():
    B, H, n, d, L = 2, 4, 8192, 128, 4
    K = _keys(11, B, H, n, d, torch.bfloat16, False)
    out = torch.empty(B, H, n >> L, d, dtype=torch.bfloat16, device="cuda")
    wf.wf_wavelet_approx(K, L, wf.WF_WAVELET_HAAR, out)
    coeffs = torch.empty(wf.wf_coeffs_bytes(K, L), dtype=torch.uint8, device="cuda")
    wf.wf_dwt_build(K, L, coeffs)
    torch.cuda.synchronize()
    pyr = coeffs.view(torch.bfloat16).view(B, H, n - (n >> L), d)
    assert torch.equal(out, pyr[:, :, n - (n >> (L - 1)):])


def _filter_wavelet(batch, w, wv):
    Q, K = batch.Q, batch.K
    B, H = K.shape[:2]
    top = torch.empty(B, H, w.n >> w.levels, w.head_dim, dtype=K.dtype, device="cuda")
    wf.wf_wavelet_approx(K, w.levels, wv, top)
    ws = torch.zeros(wf.wf_filter_wavelet_workspace_bytes(Q, K, w.levels, w.keep, wv), dtype=torch.uint8,
                     device="cuda")
    idx = torch.empty(B * H, w.k, dtype=torch.int32, device="cuda")
    sets = torch.empty(B * H, sum(w.keep), dtype=torch.int32, device="cuda")
    wf.wf_filter_wavelet(Q, top, K, w.levels, w.keep, wv, idx, ws, level_sets=sets)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    return idx, sets


@pytest.mark.parametrize("cfg", ["c2", "c3"])
def test_filter_wavelet_haar_equals_filter(cfg):
    w = synth.WORKLOADS[cfg]
    batch = synth.make_batch(w, planted=True, device="cuda", cfg=cfg, units=[0, 5, w.units - 1])
    idx, sets = _filter_wavelet(batch, w, wf.WF_WAVELET_HAAR)
    ref = LibRun(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, w.levels, w.keep).dwt().filter()
    torch.cuda.synchronize()
    assert torch.equal(idx, ref.idx)
    assert torch.equal(sets, ref.sets)


@pytest.mark.parametrize("cfg,units", [("c1", None), ("c2", [0, 31]), ("c3", [0, 63]), ("c4", [31])])
def test_filter_wavelet_db2_matches_oracle(cfg, units):
    w = synth.WORKLOADS[cfg]
    batch = synth.make_batch(w, planted=True, device="cuda", cfg=cfg, units=units)
    idx, sets = _filter_wavelet(batch, w, wf.WF_WAVELET_DB2)
    for u in (units if units is not None else range(w.units)):
        b, h = divmod(u, w.heads)
        Q, K = f64(batch.Q[b, h]), f64(batch.K[b, h])
        mu0, osets = oracle.filter_wavelet(Q, K, w.levels, np.array(w.keep), oracle.DB2, spec32=True,
                                           store_bf16=w.dtype == "bf16", want_sets=True)
        gsets = oracle.split_level_sets(sets[u].cpu().numpy(), w.levels, w.keep)
        for lev in range(w.levels, -1, -1):
            assert np.array_equal(gsets[lev], osets[lev]), f"unit {u} scale {lev}"
        assert np.array_equal(idx[u].cpu().numpy(), mu0)


@pytest.mark.parametrize("cfg,units", [("c2", [0, 31]), ("c3", [0, 63]), ("c4", [31])])
def test_step_wavelet_db2_matches_oracle(cfg, units):
    # The literal step: indices and level sets of the planted units against the
    # oracle's literal filter, every unit's output against the oracle attention
    # on the GPU's own indices, and the filter-only call agreeing bit for bit.
    w = synth.WORKLOADS[cfg]
    batch = synth.make_batch(w, planted=True, device="cuda", cfg=cfg, units=units)
    Q, K, V = batch.Q, batch.K, batch.V
    B, H = K.shape[:2]
    wv = wf.WF_WAVELET_DB2
    top = torch.empty(B, H, w.n >> w.levels, w.head_dim, dtype=K.dtype, device="cuda")
    wf.wf_wavelet_approx(K, w.levels, wv, top)
    ws = torch.zeros(wf.wf_step_wavelet_workspace_bytes(Q, K, w.levels, w.keep, wv, w.ng), dtype=torch.uint8,
                     device="cuda")
    idx = torch.empty(B * H, w.k, dtype=torch.int32, device="cuda")
    sets = torch.empty(B * H, sum(w.keep), dtype=torch.int32, device="cuda")
    O = torch.empty_like(Q)
    wf.wf_step_wavelet(Q, top, K, V, batch.Kg, batch.Vg, w.levels, w.keep, wv, idx, O, ws, level_sets=sets)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    idx_f, sets_f = _filter_wavelet(batch, w, wv)
    assert torch.equal(idx, idx_f) and torch.equal(sets, sets_f)
    for u in units:
        b, h = divmod(u, w.heads)
        Qu, Ku = f64(Q[b, h]), f64(K[b, h])
        mu0, osets = oracle.filter_wavelet(Qu, Ku, w.levels, np.array(w.keep), oracle.DB2, spec32=True,
                                           store_bf16=True, want_sets=True)
        gsets = oracle.split_level_sets(sets[u].cpu().numpy(), w.levels, w.keep)
        for lev in range(w.levels, -1, -1):
            assert np.array_equal(gsets[lev], osets[lev]), f"unit {u} scale {lev}"
        assert np.array_equal(idx[u].cpu().numpy(), mu0)
    idx_h = idx.cpu().numpy()
    for u in range(w.units):
        b, h = divmod(u, w.heads)
        ref = oracle.sparse_attn(f64(Q[b, h]), f64(K[b, h]), f64(V[b, h]), idx_h[u], f64(batch.Kg[b, h]),
                                 f64(batch.Vg[b, h]))
        assert_close_out(f64(O[b, h]), ref, torch.bfloat16)


@pytest.mark.parametrize("basis", ["db2", "haar"])
def test_step_wavelet_odd_units_no_generation_rows(basis):
    # Three units (a two-unit cluster plan leaves its last cluster one unit)
    # and no generation rows: every unit against the oracle's literal filter
    # (indices at every scale) and attention over the selected rows only.
    wv, ov = BASES[basis]
    w = dataclasses.replace(synth.WORKLOADS["c3"], name="odd_units", batch=1, heads=3, n=4096, levels=3, ng=0,
                            keep=tuple(int(x) for x in oracle.default_schedule(4096, 3, 512)))
    batch = synth.make_batch(w, planted=True, device="cuda", cfg="c3")
    Q, K, V = batch.Q, batch.K, batch.V
    B, H = K.shape[:2]
    top = torch.empty(B, H, w.n >> w.levels, w.head_dim, dtype=K.dtype, device="cuda")
    wf.wf_wavelet_approx(K, w.levels, wv, top)
    ws = torch.zeros(wf.wf_step_wavelet_workspace_bytes(Q, K, w.levels, w.keep, wv, 0), dtype=torch.uint8,
                     device="cuda")
    idx = torch.empty(B * H, w.k, dtype=torch.int32, device="cuda")
    sets = torch.empty(B * H, sum(w.keep), dtype=torch.int32, device="cuda")
    O = torch.empty_like(Q)
    wf.wf_step_wavelet(Q, top, K, V, None, None, w.levels, w.keep, wv, idx, O, ws, level_sets=sets)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    for u in range(w.units):
        b, h = divmod(u, w.heads)
        Qu, Ku, Vu = f64(Q[b, h]), f64(K[b, h]), f64(V[b, h])
        mu0, osets = oracle.filter_wavelet(Qu, Ku, w.levels, np.array(w.keep), ov, spec32=True, store_bf16=True,
                                           want_sets=True)
        gsets = oracle.split_level_sets(sets[u].cpu().numpy(), w.levels, w.keep)
        for lev in range(w.levels, -1, -1):
            assert np.array_equal(gsets[lev], osets[lev]), f"unit {u} scale {lev}"
        assert np.array_equal(idx[u].cpu().numpy(), mu0), f"unit {u}"
        assert_close_out(f64(O[b, h]), oracle.sparse_attn(Qu, Ku, Vu, mu0), torch.bfloat16)
