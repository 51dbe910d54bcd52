"""WaveFilter CPU oracle — TEST INFRASTRUCTURE ONLY.

ctypes wrapper over ``oracle/wf_oracle.c`` (plain single-threaded C, fp64
unless stated), written from the paper's Section 3 (Eq. 5-11) and
Algorithm 1.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py`` may import this package; the product library never does.
It shares no code with the CUDA path.

Every function works on one (batch, head) unit with numpy arrays:
``[rows, d]`` row-major matrices, int32 index vectors.  ``keep`` is the kept
count vector: ``keep[b]`` for scale b = 1..L and ``keep[0]`` = final k.

Every function here is pinned by ``-m "not gpu"`` tests against facts that do
not come from the oracle itself: perfect reconstruction, Parseval and the
closed forms of the Haar and db2 transforms, a hand-worked Haar example and
Daubechies' published db2 taps (``tests/golden/``), brute-force search over
all k-subsets for the Top-K, the two-candidate logistic closed form and torch
softmax for the skim weights, torch's fp64 attention for the sparse
attention, and Table 3's proportion range for the schedules.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "wf_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no implicit multiply-add contraction, no fast-math)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < max(
        os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "wf_oracle.h"))
    ):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
             "-o", tmp, _SRC, "-lm"]
        )
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    P = ctypes.c_void_p
    I64 = ctypes.c_int64
    I = ctypes.c_int
    sigs = {
        "orc_pyramid_row_offset": (I64, [I64, I]),
        "orc_pyramid_rows": (I64, [I64, I]),
        "orc_haar_analysis_f64": (I, [P, I64, I, I, P, P]),
        "orc_haar_synthesis_f64": (I, [P, P, I64, I, I, P]),
        "orc_haar_pyramid_spec32": (I, [P, I64, I, I, I, P]),
        "orc_round_bf16": (ctypes.c_float, [ctypes.c_float]),
        "orc_skim_weights_f64": (I, [P, I, I, P, I64, P]),
        "orc_default_schedule": (I, [I64, I, I64, P]),
        "orc_level0_schedule": (I, [I64, I, I64, P]),
        "orc_schedule_from_proportions": (I, [I64, I, P, P]),
        "orc_filter_f64": (I, [P, I, I, P, P, I64, I, P, P, P, P]),
        "orc_filter_literal_f64": (I, [P, I, I, P, I64, I, P, P, P]),
        "orc_wavelet_taps": (I, [I, P, P]),
        "orc_wavelet_analysis_f64": (I, [P, I64, I, I, I, P, P]),
        "orc_wavelet_synthesis_f64": (I, [P, P, I64, I, I, I, P]),
        "orc_wavelet_approx_spec32": (I, [P, I64, I, I, I, I, P]),
        "orc_filter_wavelet_f64": (I, [P, I, I, P, I64, I, I, P, I, I, P, P]),
        "orc_attention_f64": (I, [P, I, I, P, P, I64, P]),
        "orc_sparse_attn_f64": (I, [P, I, I, P, P, P, I64, P, P, I64, P]),
    }
    for name, (res, args) in sigs.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _check(rc: int, what: str):
    if rc != 0:
        raise ValueError(f"oracle {what}: invalid arguments (rc={rc})")


def pyramid_row_offset(n: int, b: int) -> int:
    return int(_load().orc_pyramid_row_offset(n, b))


def pyramid_rows(n: int, L: int) -> int:
    return int(_load().orc_pyramid_rows(n, L))


def haar_analysis(x, L: int):
    """fp64 pyramid (Eq. 5 applied L times): returns (A, D), pyramid layout."""
    x = _f64(x)
    n, d = x.shape
    rows = pyramid_rows(n, L)
    A = np.zeros((rows, d))
    D = np.zeros((rows, d))
    _check(_load().orc_haar_analysis_f64(_p(x), n, d, L, _p(A), _p(D)), "haar_analysis")
    return A, D


def haar_synthesis(A, D, n: int, L: int):
    A = _f64(A)
    D = _f64(D)
    d = A.shape[1]
    x = np.zeros((n, d))
    _check(_load().orc_haar_synthesis_f64(_p(A), _p(D), n, d, L, _p(x)), "haar_synthesis")
    return x


def level(pyr: np.ndarray, n: int, b: int) -> np.ndarray:
    """Rows of scale b inside a pyramid array."""
    off = pyramid_row_offset(n, b)
    return pyr[off: off + (n >> b)]


def haar_pyramid_spec32(x, L: int, store_bf16: bool):
    """The stored pyramid: fp32 cascade, rounded to bf16 if asked (as float32)."""
    x = _f32(x)
    n, d = x.shape
    A = np.zeros((pyramid_rows(n, L), d), dtype=np.float32)
    _check(_load().orc_haar_pyramid_spec32(_p(x), n, d, L, int(bool(store_bf16)), _p(A)), "pyramid_spec32")
    return A


def round_bf16(f: float) -> float:
    return float(_load().orc_round_bf16(ctypes.c_float(f)))


def skim_weights(Q, rows):
    """Eq. 7-8 on an explicit candidate row set: W[j] over the rows."""
    Q = _f64(Q)
    rows = _f64(rows)
    q, d = Q.shape
    m = rows.shape[0]
    W = np.zeros(m)
    _check(_load().orc_skim_weights_f64(_p(Q), q, d, _p(rows), m, _p(W)), "skim_weights")
    return W


def default_schedule(n: int, L: int, k: int) -> np.ndarray:
    keep = np.zeros(L + 1, dtype=np.int32)
    _check(_load().orc_default_schedule(n, L, k, _p(keep)), "default_schedule")
    return keep


def level0_schedule(n: int, L: int, k: int) -> np.ndarray:
    """The token level as its own selection step (m = (k/n)^(1/(L+1)))."""
    keep = np.zeros(L + 1, dtype=np.int32)
    _check(_load().orc_level0_schedule(n, L, k, _p(keep)), "level0_schedule")
    return keep


def schedule_from_proportions(n: int, L: int, m) -> np.ndarray:
    """m[b] for b = 1..L (index 0 unused)."""
    m = _f64(m)
    assert m.shape[0] == L + 1
    keep = np.zeros(L + 1, dtype=np.int32)
    _check(_load().orc_schedule_from_proportions(n, L, _p(m), _p(keep)), "schedule_from_proportions")
    return keep


def _level_w_len(n: int, L: int, keep) -> int:
    tot = n >> L
    for b in range(L - 1, 0, -1):
        tot += 2 * int(keep[b + 1])
    if int(keep[0]) < 2 * int(keep[1]):
        tot += 2 * int(keep[1])
    return tot


def split_level_sets(flat: np.ndarray, L: int, keep):
    """Split the back-to-back level sets into {b: J_b} (b = L..1) and mu0 (key 0)."""
    out = {}
    pos = 0
    for b in range(L, -1, -1):
        kb = int(keep[b])
        out[b] = flat[pos: pos + kb]
        pos += kb
    return out


def filter(Q, pyr, K, n: int, L: int, keep, want_sets: bool = False, want_w: bool = False):
    """Multi-scale recursive filtering on the stored pyramid (fp64 scoring).

    Returns mu0 (int32, ascending), plus {b: J_b} and the flat W vector when asked.
    """
    Q = _f64(Q)
    pyr = _f64(pyr)
    K = _f64(K)
    keep = _i32(keep)
    q, d = Q.shape
    mu0 = np.zeros(int(keep[0]), dtype=np.int32)
    sets = np.zeros(int(keep.sum()), dtype=np.int32) if want_sets else None
    W = np.zeros(_level_w_len(n, L, keep)) if want_w else None
    _check(_load().orc_filter_f64(_p(Q), q, d, _p(pyr), _p(K), n, L, _p(keep), _p(mu0),
                                  _p(sets) if sets is not None else None,
                                  _p(W) if W is not None else None), "filter")
    res = [mu0]
    if want_sets:
        res.append(split_level_sets(sets, L, keep))
    if want_w:
        res.append(W)
    return res[0] if len(res) == 1 else tuple(res)


def filter_literal(Q, K, L: int, keep, want_sets: bool = False):
    """Algorithm 1 taken literally (Eq. 11 DWT of the gathered tokens per scale)."""
    Q = _f64(Q)
    K = _f64(K)
    keep = _i32(keep)
    q, d = Q.shape
    n = K.shape[0]
    mu0 = np.zeros(int(keep[0]), dtype=np.int32)
    sets = np.zeros(int(keep.sum()), dtype=np.int32) if want_sets else None
    _check(_load().orc_filter_literal_f64(_p(Q), q, d, _p(K), n, L, _p(keep), _p(mu0),
                                          _p(sets) if sets is not None else None), "filter_literal")
    if want_sets:
        return mu0, split_level_sets(sets, L, keep)
    return mu0


def attention(Q, Ks, Vs):
    Q = _f64(Q)
    Ks = _f64(Ks)
    Vs = _f64(Vs)
    q, d = Q.shape
    O = np.zeros((q, Vs.shape[1]))
    _check(_load().orc_attention_f64(_p(Q), q, d, _p(Ks), _p(Vs), Ks.shape[0], _p(O)), "attention")
    return O


def sparse_attn(Q, K, V, mu0, Kg=None, Vg=None):
    Q = _f64(Q)
    K = _f64(K)
    V = _f64(V)
    mu0 = _i32(mu0)
    q, d = Q.shape
    if Kg is None:
        Kg = np.zeros((0, d))
        Vg = np.zeros((0, d))
    Kg = _f64(Kg)
    Vg = _f64(Vg)
    O = np.zeros((q, d))
    _check(_load().orc_sparse_attn_f64(_p(Q), q, d, _p(K), _p(V), _p(mu0), mu0.shape[0],
                                       _p(Kg) if Kg.shape[0] else None, _p(Vg) if Vg.shape[0] else None,
                                       Kg.shape[0], _p(O)), "sparse_attn")
    return O


def filter_gqa(Qh, pyr, K, n: int, L: int, keep, want_sets: bool = False, want_w: bool = False):
    """Filtering for one KV head shared by G query heads (grouped-query
    attention, as in the Dream base model the paper evaluates, Section 4.1).

    Eq. 7's softmax is taken for every query row of every head of the group,
    and Eq. 8's column sum runs over all of those rows: the KV head's
    importance W is the sum of its heads' W.  Qh is [G, q, d] (head after
    head) or already [G*q, d]; the rows are stacked and filtered as one query
    block, which is that sum.  Same outputs as ``filter``.
    """
    Qh = _f64(Qh)
    Qs = np.ascontiguousarray(Qh.reshape(-1, Qh.shape[-1]))
    return filter(Qs, pyr, K, n, L, keep, want_sets=want_sets, want_w=want_w)


def sparse_attn_gqa(Qh, K, V, mu0, Kg=None, Vg=None):
    """Final attention of each query head of a group over the rows its KV head
    kept (Algorithm 1, final step, once per query head).  Qh: [G, q, d];
    returns [G, q, d]."""
    Qh = _f64(Qh)
    return np.stack([sparse_attn(Qh[g], K, V, mu0, Kg, Vg) for g in range(Qh.shape[0])])


# Other wavelet bases (Eq. 6 / Eq. 11 with a generic psi), periodized.
HAAR, DB2 = 0, 1


def wavelet_taps(wavelet: int):
    """(h, g) of the orthogonal filter bank: Haar or db2."""
    h = np.zeros(4)
    g = np.zeros(4)
    taps = _load().orc_wavelet_taps(wavelet, _p(h), _p(g))
    if taps < 0:
        raise ValueError(f"unknown wavelet {wavelet}")
    return h[:taps].copy(), g[:taps].copy()


def wavelet_analysis(x, wavelet: int, L: int):
    """L periodized analysis levels: (A, D) in the pyramid layout."""
    x = _f64(x)
    n, d = x.shape
    rows = pyramid_rows(n, L)
    A = np.zeros((rows, d))
    D = np.zeros((rows, d))
    _check(_load().orc_wavelet_analysis_f64(_p(x), n, d, wavelet, L, _p(A), _p(D)), "wavelet_analysis")
    return A, D


def wavelet_synthesis(A, D, n: int, wavelet: int, L: int):
    A = _f64(A)
    D = _f64(D)
    d = A.shape[1]
    x = np.zeros((n, d))
    _check(_load().orc_wavelet_synthesis_f64(_p(A), _p(D), n, d, wavelet, L, _p(x)), "wavelet_synthesis")
    return x


def wavelet_approx_spec32(x, wavelet: int, level: int, store_bf16: bool):
    """Level-`level` approximation rows of x under the library's fp32 storage rule."""
    x = _f32(x)
    n, d = x.shape
    out = np.zeros((n >> level, d), dtype=np.float32)
    _check(_load().orc_wavelet_approx_spec32(_p(x), n, d, wavelet, level, int(store_bf16), _p(out)),
           "wavelet_approx_spec32")
    return out


def filter_wavelet(Q, K, L: int, keep, wavelet: int, spec32: bool = True, store_bf16: bool = False,
                   want_sets: bool = False):
    """Algorithm 1 with a generic psi, literally (Eq. 11's transform of the
    gathered keys at every scale).  Returns mu0 (and {b: J_b})."""
    Q = _f64(Q)
    K = _f64(K)
    keep = _i32(keep)
    q, d = Q.shape
    n = K.shape[0]
    mu0 = np.zeros(int(keep[0]), dtype=np.int32)
    sets = np.zeros(int(keep.sum()), dtype=np.int32) if want_sets else None
    _check(_load().orc_filter_wavelet_f64(_p(Q), q, d, _p(K), n, L, wavelet, _p(keep), int(spec32),
                                          int(store_bf16), _p(mu0), _p(sets) if sets is not None else None),
           "filter_wavelet")
    if want_sets:
        return mu0, split_level_sets(sets, L, keep)
    return mu0
