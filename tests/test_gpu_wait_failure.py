"""The failure path of the tensor-core kernels' bounded waits, driven through
the test-only control of include/wf_testing.h: the first wait of every CTA
waits on a barrier that nothing completes, with a short bound, so it gives
up.  The call must report WF_ERR_TIMEOUT through the workspace status word,
write nothing outside its outputs, and leave the context usable: the next
normal call matches the oracle.  Small layers only (four units)."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from helpers import assert_close_out, f64
from paper_2606_00724_gb300 import synth, wf

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)

WF_ERR_TIMEOUT = -7
GUARD = 64          # guard rows / words on each side of an output
SENTINEL = -12288.0  # exact in bf16


def _small_layer(n=4096, levels=3, k=512):
    w = dataclasses.replace(synth.WORKLOADS["c3"], name=f"wait_failure_n{n}", batch=1, heads=4, n=n, levels=levels,
                            keep=tuple(int(x) for x in oracle.default_schedule(n, levels, k)))
    b = synth.make_batch(w, planted=True, device="cpu", cfg="c3")
    return w, dataclasses.replace(b, Q=b.Q.cuda(), K=b.K.cuda(), V=b.V.cuda(), Kg=b.Kg.cuda(), Vg=b.Vg.cuda())


def _guarded_out(Q):
    """O as a view into a buffer with GUARD sentinel rows before and after
    each head's rows."""
    B, H, q, d = Q.shape
    full = torch.full((B, H, q + 2 * GUARD, d), SENTINEL, dtype=Q.dtype, device=Q.device)
    return full, full[:, :, GUARD:GUARD + q, :]


def _guarded_idx(units, k, device):
    full = torch.full((units * k + 2 * GUARD,), -7, dtype=torch.int32, device=device)
    return full, full[GUARD:GUARD + units * k].view(units, k)


def _guards_intact(O_full, idx_full):
    g = O_full[:, :, :GUARD].float(), O_full[:, :, -GUARD:].float()
    assert torch.all(g[0] == SENTINEL) and torch.all(g[1] == SENTINEL), "write outside O"
    assert torch.all(idx_full[:GUARD] == -7) and torch.all(idx_full[-GUARD:] == -7), "write outside idx"


def _oracle_unit(w, batch, u):
    b, h = divmod(u, w.heads)
    Q, K, V, Kg, Vg = (f64(t[b, h]) for t in (batch.Q, batch.K, batch.V, batch.Kg, batch.Vg))
    pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), w.levels, True)
    mu0 = oracle.filter(Q, pyr, K, w.n, w.levels, np.array(w.keep))
    return mu0, oracle.sparse_attn(Q, K, V, mu0, Kg, Vg)


# 4K tokens: two units per cluster; 32K tokens (lists of 2048): one unit per
# cluster served by both compute warpgroups.
@pytest.mark.parametrize("n,levels,k,check", [(4096, 3, 512, 4), (32768, 4, 2048, 2)])
def test_fused_step_wait_gives_up_then_recovers(n, levels, k, check):
    w, batch = _small_layer(n, levels, k)
    keep = list(w.keep)
    coeffs = torch.empty(wf.wf_coeffs_bytes(batch.K, w.levels), dtype=torch.uint8, device="cuda")
    ws = torch.zeros(wf.wf_step_workspace_bytes(batch.Q, batch.K, w.levels, keep, w.ng), dtype=torch.uint8,
                     device="cuda")
    O_full, O = _guarded_out(batch.Q)
    idx_full, idx = _guarded_idx(w.units, w.k, "cuda")
    wf.wf_dwt_build(batch.K, w.levels, coeffs)
    try:
        wf.wf_testing_set_wait_failure(True, 100_000)  # ~50 us at 2 GHz
        wf.wf_step(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, coeffs, False, w.levels, keep, idx, O, ws)
        with pytest.raises(wf.WfError) as ei:
            wf.wf_workspace_status(ws)
        assert ei.value.status == WF_ERR_TIMEOUT
    finally:
        wf.wf_testing_set_wait_failure(False, 0)
    torch.cuda.synchronize()
    _guards_intact(O_full, idx_full)
    # The status word was cleared by the report; a normal call is exact.
    wf.wf_step(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, coeffs, False, w.levels, keep, idx, O, ws)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    _guards_intact(O_full, idx_full)
    for u in range(check):
        mu0, O_ref = _oracle_unit(w, batch, u)
        assert np.array_equal(idx[u].cpu().numpy(), mu0), f"unit {u}"
        assert_close_out(f64(O[0, u]), O_ref, torch.bfloat16)


def test_tensor_core_attention_wait_gives_up_then_recovers():
    w, batch = _small_layer()
    g = torch.Generator(device="cpu").manual_seed(5)
    idx_list = torch.stack([torch.randperm(w.n, generator=g)[: w.k].sort().values for _ in range(w.units)])
    idx_list = idx_list.to(torch.int32).cuda()
    ws = torch.zeros(wf.wf_attn_workspace_bytes(batch.Q, w.k, w.ng), dtype=torch.uint8, device="cuda")
    O_full, O = _guarded_out(batch.Q)
    try:
        wf.wf_testing_set_wait_failure(True, 100_000)
        wf.wf_sparse_attn(batch.Q, batch.K, batch.V, idx_list, w.k, batch.Kg, batch.Vg, O, ws)
        with pytest.raises(wf.WfError) as ei:
            wf.wf_workspace_status(ws)
        assert ei.value.status == WF_ERR_TIMEOUT
    finally:
        wf.wf_testing_set_wait_failure(False, 0)
    torch.cuda.synchronize()
    g0, g1 = O_full[:, :, :GUARD].float(), O_full[:, :, -GUARD:].float()
    assert torch.all(g0 == SENTINEL) and torch.all(g1 == SENTINEL), "write outside O"
    wf.wf_sparse_attn(batch.Q, batch.K, batch.V, idx_list, w.k, batch.Kg, batch.Vg, O, ws)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    for u in range(w.units):
        b, h = divmod(u, w.heads)
        Q, K, V, Kg, Vg = (f64(t[b, h]) for t in (batch.Q, batch.K, batch.V, batch.Kg, batch.Vg))
        ref = oracle.sparse_attn(Q, K, V, idx_list[u].cpu().numpy(), Kg, Vg)
        assert_close_out(f64(O[b, h]), ref, torch.bfloat16)



def test_grouped_filter_wait_gives_up_then_recovers():
    # wf_step on grouped query heads (the grouped filter kernel, then the
    # tensor-core attention) under the same stalled first wait: the status
    # word reports WF_ERR_TIMEOUT, nothing is written outside idx and O, and
    # the next normal call matches the oracle.
    n, levels, k = 4096, 3, 512
    w = dataclasses.replace(synth.WORKLOADS["g1"], name="wait_failure_gqa", batch=1, heads=2, n=n, levels=levels,
                            keep=tuple(int(x) for x in oracle.default_schedule(n, levels, k)))
    b = synth.make_batch(w, planted=True, device="cpu", cfg="g1")
    batch = dataclasses.replace(b, Q=b.Q.cuda(), K=b.K.cuda(), V=b.V.cuda(), Kg=b.Kg.cuda(), Vg=b.Vg.cuda())
    keep = list(w.keep)
    G = w.group
    coeffs = torch.empty(wf.wf_coeffs_bytes(batch.K, w.levels), dtype=torch.uint8, device="cuda")
    ws = torch.zeros(wf.wf_step_workspace_bytes(batch.Q, batch.K, w.levels, keep, w.ng), dtype=torch.uint8,
                     device="cuda")
    O_full, O = _guarded_out(batch.Q)
    idx_full, idx = _guarded_idx(w.units, w.k, "cuda")
    wf.wf_dwt_build(batch.K, w.levels, coeffs)
    try:
        wf.wf_testing_set_wait_failure(True, 100_000)
        wf.wf_step(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, coeffs, False, w.levels, keep, idx, O, ws)
        with pytest.raises(wf.WfError) as ei:
            wf.wf_workspace_status(ws)
        assert ei.value.status == WF_ERR_TIMEOUT
    finally:
        wf.wf_testing_set_wait_failure(False, 0)
    torch.cuda.synchronize()
    _guards_intact(O_full, idx_full)
    wf.wf_step(batch.Q, batch.K, batch.V, batch.Kg, batch.Vg, coeffs, False, w.levels, keep, idx, O, ws)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    _guards_intact(O_full, idx_full)
    for u in range(w.units):
        bb, h = divmod(u, w.heads)
        Qh = f64(batch.Q[bb, h * G:(h + 1) * G])
        K, V, Kg, Vg = (f64(t[bb, h]) for t in (batch.K, batch.V, batch.Kg, batch.Vg))
        pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), w.levels, True)
        mu0 = oracle.filter_gqa(Qh, pyr, K, w.n, w.levels, np.array(w.keep))
        assert np.array_equal(idx[u].cpu().numpy(), mu0), f"unit {u}"
        assert_close_out(f64(O[bb, h * G:(h + 1) * G]), oracle.sparse_attn_gqa(Qh, K, V, mu0, Kg, Vg), torch.bfloat16)
