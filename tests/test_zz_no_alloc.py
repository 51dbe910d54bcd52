"""wf_sparse_attn_noalloc: the sparse-attention entry point for callers that
cannot allocate device memory (its scratch is a fixed static device array
inside libwf).  Checked through the C ABI against wf_sparse_attn, which uses
a caller workspace, on two calls in a row.  This file is collected last."""
import threading

import numpy as np
import pytest
import torch

from helpers import assert_close_out, f64
from paper_2606_00724_gb300 import synth, wf

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)


def _inputs(cfg, seed):
    w = synth.WORKLOADS[cfg]
    batch = synth.make_batch(w, planted=False, device="cuda", cfg=cfg)
    g = torch.Generator(device="cpu").manual_seed(seed)
    idx = torch.stack([torch.randperm(w.n, generator=g)[: w.k].sort().values for _ in range(w.units)])
    return w, batch, idx.to(torch.int32).cuda()


@pytest.mark.parametrize("cfg", ["c1", "c2"])
def test_noalloc_matches_workspace_entry_point(cfg):
    w, batch, idx = _inputs(cfg, 1)
    ws = torch.zeros(wf.wf_attn_workspace_bytes(batch.Q, w.k, w.ng), dtype=torch.uint8, device="cuda")
    ref = torch.empty_like(batch.Q)
    wf.wf_sparse_attn(batch.Q, batch.K, batch.V, idx, w.k, batch.Kg, batch.Vg, ref, ws)
    for call in range(2):
        out = torch.full_like(batch.Q, float("nan"))
        wf.wf_sparse_attn_noalloc(batch.Q, batch.K, batch.V, idx, w.k, batch.Kg, batch.Vg, out)
        torch.cuda.synchronize()
        assert torch.isfinite(out.float()).all(), f"call {call}"
        assert_close_out(f64(out), f64(ref), batch.Q.dtype)
    # A second, different problem right after: the shared scratch keeps the
    # previous call's contents, which must not leak into this result.
    idx2 = torch.flip(idx, dims=[1]).contiguous()
    ref2 = torch.empty_like(batch.Q)
    wf.wf_sparse_attn(batch.Q, batch.K, batch.V, idx2[:, : w.k // 2].contiguous(), w.k // 2, None, None, ref2, ws)
    out2 = torch.empty_like(batch.Q)
    wf.wf_sparse_attn_noalloc(batch.Q, batch.K, batch.V, idx2[:, : w.k // 2].contiguous(), w.k // 2, None, None,
                              out2)
    torch.cuda.synchronize()
    assert_close_out(f64(out2), f64(ref2), batch.Q.dtype)
    # No bounded device wait gave up (the status word in the static array).
    wf.wf_noalloc_status()


def test_noalloc_from_another_host_thread():
    # Another host thread with the same device current uses the same context
    # (the runtime's primary context), so it finds the cached scratch address.
    w, batch, idx = _inputs("c2", 3)
    ws = torch.zeros(wf.wf_attn_workspace_bytes(batch.Q, w.k, w.ng), dtype=torch.uint8, device="cuda")
    ref = torch.empty_like(batch.Q)
    wf.wf_sparse_attn(batch.Q, batch.K, batch.V, idx, w.k, batch.Kg, batch.Vg, ref, ws)
    out = torch.full_like(batch.Q, float("nan"))
    torch.cuda.synchronize()
    errors = []

    def worker():
        try:
            torch.cuda.set_device(batch.Q.device)
            wf.wf_sparse_attn_noalloc(batch.Q, batch.K, batch.V, idx, w.k, batch.Kg, batch.Vg, out)
            torch.cuda.synchronize()
        except Exception as e:  # reported in the main thread
            errors.append(e)

    t = threading.Thread(target=worker)
    t.start()
    t.join()
    assert not errors, errors
    assert_close_out(f64(out), f64(ref), batch.Q.dtype)
    wf.wf_noalloc_status()


def test_noalloc_rejects_oversized_requests():
    # 64 heads x 4096 selected rows needs ~68 MB of split-K scratch, beyond
    # the fixed 16 MiB: rejected with WF_ERR_WORKSPACE before any launch.
    B, H, n, d, q = 1, 64, 4096, 128, 32
    Q = torch.zeros(B, H, q, d, dtype=torch.bfloat16, device="cuda")
    K = torch.zeros(B, H, n, d, dtype=torch.bfloat16, device="cuda")
    idx = torch.zeros(B * H, n, dtype=torch.int32, device="cuda")
    O = torch.zeros_like(Q)
    assert wf.wf_attn_workspace_bytes(Q, n, 0) > (16 << 20)
    with pytest.raises(wf.WfError) as ei:
        wf.wf_sparse_attn_noalloc(Q, K, K, idx, n, None, None, O)
    assert ei.value.status == -5
    assert torch.count_nonzero(O) == 0


def test_noalloc_scratch_looked_up_per_context():
    # The static array has its own address in every CUDA context.  With a
    # second (non-primary) driver context current, the status query must look
    # the array up in that context (a cached primary-context address would
    # make its 4-byte read fail there), and the primary context must keep
    # working afterwards.  No kernel runs in the second context.
    import ctypes
    try:
        cu = ctypes.CDLL("libcuda.so.1")
        create, pop, destroy = cu.cuCtxCreate_v2, cu.cuCtxPopCurrent_v2, cu.cuCtxDestroy_v2
    except (OSError, AttributeError):
        pytest.skip("driver entry points unavailable")
    torch.cuda.synchronize()
    wf.wf_noalloc_status()  # the primary context's entry
    dev = ctypes.c_int()
    assert cu.cuDeviceGet(ctypes.byref(dev), torch.cuda.current_device()) == 0
    ctx = ctypes.c_void_p()
    assert create(ctypes.byref(ctx), 0, dev) == 0  # current on this thread from here
    try:
        wf.wf_noalloc_status()  # looked up in the second context
        wf.wf_noalloc_status()  # and served from its cache entry
    finally:
        popped = ctypes.c_void_p()
        assert pop(ctypes.byref(popped)) == 0 and popped.value == ctx.value
        assert destroy(ctx) == 0
    wf.wf_noalloc_status()  # the primary context again
    torch.cuda.synchronize()
