"""Thin ctypes binding of libwf (include/wf.h), same names as the C ABI.

Argument marshalling only: torch tensors are turned into device pointers and
wf_tensor descriptors, the current CUDA stream is passed through, and a
negative status raises WfError.  Every step of the path runs in libwf's CUDA
kernels; if libwf.so is missing this module raises on import of the library
(there is no fallback).

Tensors are [B, H, rows, d] views whose last axis is contiguous (BHSD or
BSHD strides both work); idx / level_sets are int32.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libwf.so")

WF_F32, WF_BF16 = 0, 1
_DTYPES = {torch.float32: WF_F32, torch.bfloat16: WF_BF16}


class WfError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {status_str(status)} ({status})")
        self.status = status


class wf_tensor(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("heads", ctypes.c_int32), ("seq", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("stride_b", ctypes.c_int64), ("stride_h", ctypes.c_int64),
                ("stride_s", ctypes.c_int64), ("dtype", ctypes.c_int32)]


_lib = None

# Every symbol declared in include/wf.h, with its ctypes signature.
_P, _I, _I64, _SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_size_t
_T = ctypes.POINTER(wf_tensor)
SIGNATURES = {
    "wf_status_str": (ctypes.c_char_p, [_I]),
    "wf_coeffs_bytes": (_SZ, [_T, _I]),
    "wf_dwt_build": (_I, [_P, _P, _T, _I, _P, _SZ, _P]),
    "wf_default_schedule": (_I, [_I64, _I, _I64, _P]),
    "wf_level0_schedule": (_I, [_I64, _I, _I64, _P]),
    "wf_cache_update": (_I, [_P, _P, _T, _P, _P, _T, _I64, _I, _P, _SZ, _P]),
    "wf_schedule_from_proportions": (_I, [_I64, _I, _P, _P]),
    "wf_filter_workspace_bytes": (_SZ, [_T, _T, _I, _P]),
    "wf_filter": (_I, [_P, _T, _P, _P, _T, _I, _P, _P, _P, _P, _SZ, _P]),
    "wf_wavelet_approx": (_I, [_P, _T, _P, _I, _I, _I, _P, _SZ, _P]),
    "wf_filter_wavelet_workspace_bytes": (_SZ, [_T, _T, _I, _P, _I]),
    "wf_filter_wavelet": (_I, [_P, _T, _P, _P, _T, _I, _P, _I, _P, _P, _P, _SZ, _P]),
    "wf_attn_workspace_bytes": (_SZ, [_T, _I, _I]),
    "wf_sparse_attn": (_I, [_P, _T, _P, _P, _T, _P, _I, _P, _P, _T, _P, _T, ctypes.c_float, _P, _SZ, _P]),
    "wf_step_workspace_bytes": (_SZ, [_T, _T, _I, _P, _I]),
    "wf_sparse_attn_noalloc": (_I, [_P, _T, _P, _P, _T, _P, _I, _P, _P, _T, _P, _T, ctypes.c_float, _P]),
    "wf_noalloc_status": (_I, [_P]),
    "wf_step": (_I, [_P, _T, _P, _P, _T, _P, _P, _T, _P, _SZ, _I, _I, _P, _P, _P, _P, _T, _P, _SZ, _P]),
    "wf_step_wavelet_workspace_bytes": (_SZ, [_T, _T, _I, _P, _I, _I]),
    "wf_step_wavelet": (_I, [_P, _T, _P, _P, _P, _T, _P, _P, _T, _I, _P, _I, _P, _P, _P, _T, _P, _SZ, _P]),
    "wf_workspace_status": (_I, [_P, _P]),
    # include/wf_testing.h (test-only)
    "wf_testing_set_wait_failure": (_I, [_I, ctypes.c_longlong]),
}


def lib():
    """Load libwf.so (built by __graft_entry__.build() / build.py)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libwf.so not built at {LIB_PATH}; run paper_2606_00724_gb300/build.py")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def status_str(status: int) -> str:
    return lib().wf_status_str(status).decode()


def _check(status: int, what: str):
    if status != 0:
        raise WfError(status, what)


def desc(t: torch.Tensor) -> wf_tensor:
    """wf_tensor for a [B, H, rows, d] tensor with a contiguous last axis."""
    if t.dim() != 4:
        raise ValueError("expected a [B, H, rows, d] tensor")
    if t.dtype not in _DTYPES:
        raise ValueError(f"unsupported dtype {t.dtype}")
    if t.shape[3] > 1 and t.stride(3) != 1:
        raise ValueError("head_dim axis must be contiguous")
    B, H, S, D = t.shape
    return wf_tensor(B, H, S, D, t.stride(0), t.stride(1), t.stride(2), _DTYPES[t.dtype])


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _keep_arr(keep):
    arr = (ctypes.c_int32 * len(keep))(*[int(x) for x in keep])
    return arr


def wf_coeffs_bytes(K: torch.Tensor, levels: int) -> int:
    d = desc(K)
    return int(lib().wf_coeffs_bytes(ctypes.byref(d), levels))


def wf_dwt_build(K: torch.Tensor, levels: int, coeffs: torch.Tensor, stream=None):
    d = desc(K)
    _check(lib().wf_dwt_build(_ptr(K), None, ctypes.byref(d), levels, _ptr(coeffs),
                              coeffs.numel() * coeffs.element_size(), _stream(stream)), "wf_dwt_build")


def wf_cache_update(Knew: torch.Tensor, Vnew, K: torch.Tensor, V, pos: int, levels: int, coeffs: torch.Tensor,
                    stream=None) -> None:
    """Write Knew (and Vnew) into the caches at [pos, pos + count) and refresh
    the touched pyramid blocks (see the C header)."""
    dn, dk = desc(Knew), desc(K)
    _check(lib().wf_cache_update(_ptr(Knew), _ptr(Vnew) if Vnew is not None else None, ctypes.byref(dn), _ptr(K),
                                 _ptr(V) if V is not None else None, ctypes.byref(dk), pos, levels, _ptr(coeffs),
                                 coeffs.numel() * coeffs.element_size(), _stream(stream)), "wf_cache_update")


def wf_default_schedule(n: int, levels: int, k: int) -> list[int]:
    keep = (ctypes.c_int32 * (levels + 1))()
    _check(lib().wf_default_schedule(n, levels, k, keep), "wf_default_schedule")
    return list(keep)


def wf_level0_schedule(n: int, levels: int, k: int) -> list[int]:
    keep = (ctypes.c_int32 * (levels + 1))()
    _check(lib().wf_level0_schedule(n, levels, k, keep), "wf_level0_schedule")
    return list(keep)


def wf_schedule_from_proportions(n: int, levels: int, m) -> list[int]:
    arr = (ctypes.c_double * (levels + 1))(*[float(x) for x in m])
    keep = (ctypes.c_int32 * (levels + 1))()
    _check(lib().wf_schedule_from_proportions(n, levels, arr, keep), "wf_schedule_from_proportions")
    return list(keep)


def wf_filter_workspace_bytes(Q: torch.Tensor, K: torch.Tensor, levels: int, keep) -> int:
    dq, dk = desc(Q), desc(K)
    return int(lib().wf_filter_workspace_bytes(ctypes.byref(dq), ctypes.byref(dk), levels, _keep_arr(keep)))


def wf_filter(Q: torch.Tensor, coeffs: torch.Tensor, K: torch.Tensor, levels: int, keep, idx: torch.Tensor,
              ws: torch.Tensor, level_sets: torch.Tensor | None = None, stream=None):
    dq, dk = desc(Q), desc(K)
    _check(lib().wf_filter(_ptr(Q), ctypes.byref(dq), _ptr(coeffs), _ptr(K), ctypes.byref(dk), levels,
                           _keep_arr(keep), _ptr(idx), _ptr(level_sets), _ptr(ws), ws.numel() * ws.element_size(),
                           _stream(stream)), "wf_filter")


WF_WAVELET_HAAR, WF_WAVELET_DB2 = 0, 1


def wf_wavelet_approx(K: torch.Tensor, level: int, wavelet: int, out: torch.Tensor, cand=None, m=None,
                      stream=None):
    """Level-`level` approximation rows of the gathered blocks of `cand`
    ([B*H][m] int32, or None for the whole prompt) into out ([B, H, m, d])."""
    dk = desc(K)
    if m is None:
        m = cand.shape[1] if cand is not None else K.shape[2] >> level
    _check(lib().wf_wavelet_approx(_ptr(K), ctypes.byref(dk), _ptr(cand), int(m), level, wavelet, _ptr(out),
                                   out.numel() * out.element_size(), _stream(stream)), "wf_wavelet_approx")


def wf_filter_wavelet_workspace_bytes(Q: torch.Tensor, K: torch.Tensor, levels: int, keep, wavelet: int) -> int:
    dq, dk = desc(Q), desc(K)
    return int(lib().wf_filter_wavelet_workspace_bytes(ctypes.byref(dq), ctypes.byref(dk), levels, _keep_arr(keep),
                                                       wavelet))


def wf_filter_wavelet(Q: torch.Tensor, top: torch.Tensor, K: torch.Tensor, levels: int, keep, wavelet: int,
                      idx: torch.Tensor, ws: torch.Tensor, level_sets: torch.Tensor | None = None, stream=None):
    dq, dk = desc(Q), desc(K)
    _check(lib().wf_filter_wavelet(_ptr(Q), ctypes.byref(dq), _ptr(top), _ptr(K), ctypes.byref(dk), levels,
                                   _keep_arr(keep), wavelet, _ptr(idx), _ptr(level_sets), _ptr(ws),
                                   ws.numel() * ws.element_size(), _stream(stream)), "wf_filter_wavelet")


def wf_attn_workspace_bytes(Q: torch.Tensor, k: int, n_g: int) -> int:
    dq = desc(Q)
    return int(lib().wf_attn_workspace_bytes(ctypes.byref(dq), k, n_g))


def wf_sparse_attn(Q, K, V, idx, k: int, Kg, Vg, O, ws, scale: float = 0.0, stream=None):
    dq, dk, do = desc(Q), desc(K), desc(O)
    dg = desc(Kg) if Kg is not None else None
    if Vg is not None and Kg is not None and (Vg.stride() != Kg.stride() or Vg.shape != Kg.shape):
        raise ValueError("Kg and Vg must share shape and strides")
    if V.stride() != K.stride() or V.shape != K.shape:
        raise ValueError("K and V must share shape and strides")
    _check(lib().wf_sparse_attn(_ptr(Q), ctypes.byref(dq), _ptr(K), _ptr(V), ctypes.byref(dk), _ptr(idx), k,
                                _ptr(Kg), _ptr(Vg), ctypes.byref(dg) if dg is not None else None, _ptr(O),
                                ctypes.byref(do), float(scale), _ptr(ws), ws.numel() * ws.element_size(),
                                _stream(stream)), "wf_sparse_attn")


def wf_sparse_attn_noalloc(Q, K, V, idx, k: int, Kg, Vg, O, scale: float = 0.0, stream=None):
    """wf_sparse_attn for callers that cannot allocate device memory: the
    scratch comes from libwf's fixed static device array
    (WF_NOALLOC_SCRATCH_BYTES = 16 MiB), shared by every call in a CUDA
    context."""
    dq, dk, do = desc(Q), desc(K), desc(O)
    dg = desc(Kg) if Kg is not None else None
    if Vg is not None and Kg is not None and (Vg.stride() != Kg.stride() or Vg.shape != Kg.shape):
        raise ValueError("Kg and Vg must share shape and strides")
    if V.stride() != K.stride() or V.shape != K.shape:
        raise ValueError("K and V must share shape and strides")
    _check(lib().wf_sparse_attn_noalloc(_ptr(Q), ctypes.byref(dq), _ptr(K), _ptr(V), ctypes.byref(dk), _ptr(idx),
                                        k, _ptr(Kg), _ptr(Vg), ctypes.byref(dg) if dg is not None else None,
                                        _ptr(O), ctypes.byref(do), float(scale), _stream(stream)),
           "wf_sparse_attn_noalloc")


def wf_noalloc_status(stream=None):
    """Raise WfError(WF_ERR_TIMEOUT) if a bounded device wait of the
    allocation-free attention gave up since the last check (synchronising)."""
    _check(lib().wf_noalloc_status(_stream(stream)), "wf_noalloc_status")


def wf_step_workspace_bytes(Q: torch.Tensor, K: torch.Tensor, levels: int, keep, n_g: int) -> int:
    dq, dk = desc(Q), desc(K)
    return int(lib().wf_step_workspace_bytes(ctypes.byref(dq), ctypes.byref(dk), levels, _keep_arr(keep), n_g))


def wf_step(Q, K, V, Kg, Vg, coeffs, refresh: bool, levels: int, keep, idx, O, ws, stream=None,
            level_sets=None):
    dq, dk, do = desc(Q), desc(K), desc(O)
    dg = desc(Kg) if Kg is not None else None
    if V.stride() != K.stride() or V.shape != K.shape:
        raise ValueError("K and V must share shape and strides")
    _check(lib().wf_step(_ptr(Q), ctypes.byref(dq), _ptr(K), _ptr(V), ctypes.byref(dk), _ptr(Kg), _ptr(Vg),
                         ctypes.byref(dg) if dg is not None else None, _ptr(coeffs),
                         coeffs.numel() * coeffs.element_size(), int(bool(refresh)), levels, _keep_arr(keep),
                         _ptr(idx), _ptr(level_sets), _ptr(O), ctypes.byref(do), _ptr(ws),
                         ws.numel() * ws.element_size(), _stream(stream)), "wf_step")


def wf_step_wavelet_workspace_bytes(Q: torch.Tensor, K: torch.Tensor, levels: int, keep, wavelet: int,
                                    n_g: int) -> int:
    dq, dk = desc(Q), desc(K)
    return int(lib().wf_step_wavelet_workspace_bytes(ctypes.byref(dq), ctypes.byref(dk), levels, _keep_arr(keep),
                                                     wavelet, n_g))


def wf_step_wavelet(Q, top, K, V, Kg, Vg, levels: int, keep, wavelet: int, idx, O, ws, stream=None,
                    level_sets=None):
    dq, dk, do = desc(Q), desc(K), desc(O)
    dg = desc(Kg) if Kg is not None else None
    if V.stride() != K.stride() or V.shape != K.shape:
        raise ValueError("K and V must share shape and strides")
    _check(lib().wf_step_wavelet(_ptr(Q), ctypes.byref(dq), _ptr(top), _ptr(K), _ptr(V), ctypes.byref(dk),
                                 _ptr(Kg), _ptr(Vg), ctypes.byref(dg) if dg is not None else None, levels,
                                 _keep_arr(keep), wavelet, _ptr(idx), _ptr(level_sets), _ptr(O), ctypes.byref(do),
                                 _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)), "wf_step_wavelet")


def wf_workspace_status(ws: torch.Tensor, stream=None):
    """Raise WfError(WF_ERR_TIMEOUT) if a bounded device wait of the fused
    step kernel gave up since the last check (synchronising)."""
    _check(lib().wf_workspace_status(_ptr(ws), _stream(stream)), "wf_workspace_status")


def wf_testing_set_wait_failure(stall: bool, wait_limit_cycles: int = 0):
    """Test-only (include/wf_testing.h): make the tensor-core kernels' first
    wait stall (a barrier nothing completes) and bound the waits that can give
    up by wait_limit_cycles (0: the default bound).  Reset with (False, 0)."""
    _check(lib().wf_testing_set_wait_failure(int(bool(stall)), int(wait_limit_cycles)),
           "wf_testing_set_wait_failure")
