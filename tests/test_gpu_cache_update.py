"""GPU parity of wf_cache_update: new key/value rows written into the caches
and the touched pyramid blocks refreshed in the same kernel.

Bars: the caches hold exactly the new rows in the window and are unchanged
elsewhere; the refreshed pyramid equals a full wf_dwt_build of the updated
keys and the oracle's spec-fp32 pyramid bit for bit (every coefficient)."""
import numpy as np
import pytest
import torch

import oracle
from helpers import f64
from paper_2606_00724_gb300 import wf

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)


def _cache(seed, B, H, n, d, dtype, bshd):
    g = torch.Generator(device="cpu").manual_seed(seed)

    def r(rows):
        if bshd:
            return torch.randn(B, rows, H, d, generator=g).to(dtype).cuda().transpose(1, 2)
        return torch.randn(B, H, rows, d, generator=g).to(dtype).cuda()
    return r


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("n,d,L,pos,count,bshd,values", [
    (1024, 128, 3, 37, 50, False, True),      # window across several 8-token blocks
    (1024, 128, 3, 0, 1, False, True),        # one row at the start
    (1024, 64, 4, 1023, 1, False, False),     # one row at the end, keys only
    (512, 128, 5, 0, 512, True, True),        # the whole cache, BSHD strides
    (2048, 128, 4, 992, 32, False, True),     # one aligned query block
    (256, 64, 1, 101, 7, True, True),         # L = 1
])
def test_cache_update(dtype, n, d, L, pos, count, bshd, values):
    B, H = 2, 3
    r = _cache(n + L + pos, B, H, n, d, dtype, bshd)
    K, V = r(n), r(n)
    Kn, Vn = r(count), r(count)
    coeffs = torch.empty(wf.wf_coeffs_bytes(K, L), dtype=torch.uint8, device="cuda")
    wf.wf_dwt_build(K, L, coeffs)
    K0, V0 = K.clone(), V.clone()
    wf.wf_cache_update(Kn, Vn if values else None, K, V if values else None, pos, L, coeffs)
    full = torch.empty_like(coeffs)
    wf.wf_dwt_build(K, L, full)
    torch.cuda.synchronize()
    sl = slice(pos, pos + count)
    assert torch.equal(K[:, :, sl], Kn)
    assert torch.equal(K[:, :, :pos], K0[:, :, :pos]) and torch.equal(K[:, :, pos + count:], K0[:, :, pos + count:])
    if values:
        assert torch.equal(V[:, :, sl], Vn)
        assert torch.equal(V[:, :, :pos], V0[:, :, :pos])
        assert torch.equal(V[:, :, pos + count:], V0[:, :, pos + count:])
    else:
        assert torch.equal(V, V0)
    assert torch.equal(coeffs, full)
    # One unit against the oracle's spec-fp32 pyramid of the updated keys.
    rows = n - (n >> L)
    c = coeffs.view(dtype).view(B, H, rows, d)
    want = oracle.haar_pyramid_spec32(f64(K[1, 2]).astype(np.float32), L, dtype == torch.bfloat16)
    assert np.array_equal(f64(c[1, 2]), want.astype(np.float64))


def test_cache_update_then_step_matches_rebuild():
    # A fused step on the incrementally refreshed pyramid selects exactly what
    # it selects on a rebuilt one.
    B, H, n, d, q, L = 1, 4, 4096, 128, 32, 3
    keep = wf.wf_default_schedule(n, L, 512)
    r = _cache(5, B, H, n, d, torch.bfloat16, False)
    K, V, Q, Kg, Vg = r(n), r(n), r(q), r(32), r(32)
    Kn, Vn = r(64), r(64)
    coeffs = torch.empty(wf.wf_coeffs_bytes(K, L), dtype=torch.uint8, device="cuda")
    wf.wf_dwt_build(K, L, coeffs)
    wf.wf_cache_update(Kn, Vn, K, V, 1000, L, coeffs)
    ws = torch.zeros(wf.wf_step_workspace_bytes(Q, K, L, keep, 32), dtype=torch.uint8, device="cuda")
    idx_a = torch.empty(B * H, keep[0], dtype=torch.int32, device="cuda")
    idx_b = torch.empty_like(idx_a)
    O_a, O_b = torch.empty_like(Q), torch.empty_like(Q)
    wf.wf_step(Q, K, V, Kg, Vg, coeffs, False, L, keep, idx_a, O_a, ws)
    wf.wf_step(Q, K, V, Kg, Vg, coeffs.clone(), True, L, keep, idx_b, O_b, ws)
    wf.wf_workspace_status(ws)
    torch.cuda.synchronize()
    assert torch.equal(idx_a, idx_b)
    assert torch.equal(O_a, O_b)
