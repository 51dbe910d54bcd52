"""C-ABI checks that need no GPU: libwf builds and loads, exports every
function include/wf.h declares, and its host-side logic (schedules, sizes,
argument validation) behaves as documented.  Nothing here launches a kernel.
"""
import ctypes
import os
import re

import numpy as np
import pytest
import torch

import oracle
from paper_2606_00724_gb300 import build as wf_build
from paper_2606_00724_gb300 import synth, wf

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h")]


@pytest.fixture(scope="module")
def lib():
    wf_build.build()
    return wf.lib()


def declared_functions():
    names = set()
    for h in HEADERS:
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names |= set(re.findall(r"\b(wf_\w+)\s*\(", text))
    return names


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert "wf_filter" in names and "wf_step" in names
    for name in names:
        assert hasattr(lib, name), f"{name} declared in include/ but not exported"
    # The binding covers exactly the declared API.
    assert names == set(wf.SIGNATURES)


def test_status_strings(lib):
    for code in range(0, -10, -1):
        assert wf.status_str(code).startswith("WF_")


@pytest.mark.parametrize("n,L,k", [(1024, 2, 128), (8192, 3, 819), (32768, 4, 2048), (131072, 5, 4096),
                                   (32768, 4, 1638), (64, 6, 1), (4096, 1, 4096), (1000, 3, 77), (96, 5, 3)])
def test_default_schedule_matches_oracle(lib, n, L, k):
    assert wf.wf_default_schedule(n, L, k) == oracle.default_schedule(n, L, k).tolist()


def test_schedule_from_proportions_matches_oracle(lib):
    r = np.random.default_rng(0)
    for _ in range(50):
        L = int(r.integers(1, 6))
        n = int(r.integers(1, 64)) << L
        m = [0.0] + list(r.uniform(0.05, 1.0, L))
        assert wf.wf_schedule_from_proportions(n, L, m) == oracle.schedule_from_proportions(n, L, m).tolist()
    with pytest.raises(wf.WfError):
        wf.wf_schedule_from_proportions(64, 2, [0, 0.5, 1.5])


def test_level0_schedule_matches_oracle(lib):
    r = np.random.default_rng(1)
    for _ in range(60):
        L = int(r.integers(1, 7))
        n = int(r.integers(1, 256)) << L
        k = int(r.integers(1, n + 1))
        try:
            want = oracle.level0_schedule(n, L, k).tolist()
        except ValueError:
            with pytest.raises(wf.WfError):
                wf.wf_level0_schedule(n, L, k)
            continue
        assert wf.wf_level0_schedule(n, L, k) == want
    for w in synth.WORKLOADS.values():
        assert wf.wf_level0_schedule(w.n, w.levels, w.k) == oracle.level0_schedule(w.n, w.levels, w.k).tolist()


def test_workload_schedules(lib):
    for w in synth.WORKLOADS.values():
        assert wf.wf_default_schedule(w.n, w.levels, w.k) == list(w.keep)


def _meta(shape, dtype=torch.bfloat16):
    return torch.empty(shape, dtype=dtype, device="meta")


def test_sizes(lib):
    K = _meta((2, 32, 32768, 128))
    assert wf.wf_coeffs_bytes(K, 4) == 2 * 32 * (32768 - 2048) * 128 * 2
    assert wf.wf_coeffs_bytes(_meta((1, 1, 100, 128)), 3) == 0    # 100 % 8 != 0
    assert wf.wf_coeffs_bytes(_meta((1, 1, 64, 96)), 2) == 0      # head_dim 96 unsupported
    Q = _meta((2, 32, 32, 128))
    keep = [2048, 1024, 1024, 1024, 1024]
    assert wf.wf_filter_workspace_bytes(Q, K, 4, keep) > 0
    assert wf.wf_filter_workspace_bytes(Q, K, 4, [2049, 1024, 1024, 1024, 1024]) == 0  # infeasible
    assert wf.wf_filter_workspace_bytes(_meta((2, 32, 65, 128)), K, 4, keep) == 0       # > 64 query rows
    assert wf.wf_attn_workspace_bytes(Q, 2048, 32) > 0
    # Grouped query heads: 7 per key head (224 rows) fit, 9 (288 rows) do not.
    assert wf.wf_filter_workspace_bytes(_meta((2, 224, 32, 128)), K, 4, keep) > 0
    assert wf.wf_filter_workspace_bytes(_meta((2, 288, 32, 128)), K, 4, keep) == 0
    assert wf.wf_filter_workspace_bytes(_meta((2, 48, 32, 128)), K, 4, keep) == 0   # 48 % 32 != 0


# Argument validation returns before any CUDA call.  The pointers below are
# placeholders that are never dereferenced; these cases run only where no GPU
# is visible, so a validation bug could not turn into a device access.
no_gpu = pytest.mark.skipif(torch.cuda.is_available(), reason="placeholder pointers: host-only check")


def _desc(B, H, S, D, dtype=wf.WF_BF16, sb=None, sh=None, ss=None):
    ss = D if ss is None else ss
    sh = S * ss if sh is None else sh
    sb = H * sh if sb is None else sb
    return wf.wf_tensor(B, H, S, D, sb, sh, ss, dtype)


FAKE = ctypes.c_void_p(0x10000)
FAKE2 = ctypes.c_void_p(0x20000)


@no_gpu
def test_dwt_build_rejects(lib):
    d = _desc(1, 2, 64, 128)
    call = lambda K, V, desc, L, C, nbytes: lib.wf_dwt_build(K, V, ctypes.byref(desc), L, C, nbytes, None)
    need = lib.wf_coeffs_bytes(ctypes.byref(d), 2)
    assert call(FAKE, None, d, 2, FAKE2, need - 1) == -5
    assert call(FAKE, FAKE2, d, 2, FAKE2, need) == -1           # V must be NULL
    assert call(None, None, d, 2, FAKE2, need) == -1
    assert call(ctypes.c_void_p(0x10008), None, d, 2, FAKE2, need) == -4   # misaligned K
    assert call(FAKE, None, d, 0, FAKE2, need) == -8            # levels out of range
    assert call(FAKE, None, _desc(1, 2, 62, 128), 2, FAKE2, need) == -2   # 62 % 4 != 0
    assert call(FAKE, None, _desc(1, 2, 64, 128, dtype=7), 2, FAKE2, need) == -3
    assert call(FAKE, None, _desc(1, 2, 64, 128, ss=129), 2, FAKE2, 10 ** 9) == -4     # 258-byte rows


@no_gpu
def test_cache_update_rejects(lib):
    kv = _desc(1, 2, 64, 128)
    nt = _desc(1, 2, 8, 128)
    need = lib.wf_coeffs_bytes(ctypes.byref(kv), 2)
    F3 = ctypes.c_void_p(0x30000)

    def call(Kn, Vn, n_desc, K, V, pos, L=2, nbytes=need, kv_desc=kv):
        return lib.wf_cache_update(Kn, Vn, ctypes.byref(n_desc), K, V, ctypes.byref(kv_desc), pos, L, F3, nbytes,
                                   None)
    assert call(FAKE, None, nt, FAKE2, None, 57) == -1                     # window past the end
    assert call(FAKE, None, nt, FAKE2, None, -1) == -1
    assert call(FAKE, FAKE, nt, FAKE2, None, 0) == -1                      # Vnew without V
    assert call(None, None, nt, FAKE2, None, 0) == -1
    assert call(FAKE, None, _desc(1, 3, 8, 128), FAKE2, None, 0) == -2     # other heads
    assert call(FAKE, None, _desc(1, 2, 8, 128, dtype=wf.WF_F32), FAKE2, None, 0) == -3
    assert call(ctypes.c_void_p(0x10008), None, nt, FAKE2, None, 0) == -4  # misaligned rows
    assert call(FAKE, None, nt, FAKE2, None, 0, nbytes=need - 1) == -5
    assert call(FAKE, None, nt, FAKE2, None, 0, L=0) == -8


@no_gpu
def test_filter_rejects(lib):
    q = _desc(1, 2, 32, 128)
    kv = _desc(1, 2, 1024, 128)
    keep = (ctypes.c_int32 * 3)(128, 64, 91)
    ws_need = lib.wf_filter_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep)
    def call(q=q, kv=kv, L=2, keep=keep, ws=ctypes.c_void_p(0x100000), ws_bytes=ws_need, idx=FAKE2):
        return lib.wf_filter(FAKE, ctypes.byref(q), FAKE2, FAKE, ctypes.byref(kv), L, keep, idx, None, ws,
                             ws_bytes, None)
    assert call(ws_bytes=ws_need - 1) == -5
    assert call(ws=ctypes.c_void_p(0x100010)) == -4              # workspace not 256-byte aligned
    assert call(keep=(ctypes.c_int32 * 3)(129, 64, 91)) == -9    # k > 2 keep[1]
    assert call(keep=(ctypes.c_int32 * 3)(128, 64, 257)) == -9   # keep[2] > n/4
    assert call(q=_desc(1, 3, 32, 128)) == -2                     # heads disagree
    assert call(q=_desc(1, 18, 32, 128)) == -8                    # 9 heads x 32 rows per key head > 256
    assert call(q=_desc(2, 4, 32, 128)) == -2                     # batch disagrees
    assert call(q=_desc(1, 2, 32, 128, dtype=wf.WF_F32)) == -3    # dtypes disagree
    assert call(q=_desc(1, 2, 65, 128)) == -8                     # too many query rows
    assert call(L=11) == -8
    assert call(idx=None) == -1


@no_gpu
def test_attn_rejects(lib):
    q = _desc(1, 2, 32, 128)
    kv = _desc(1, 2, 1024, 128)
    g = _desc(1, 2, 32, 128)
    need = lib.wf_attn_workspace_bytes(ctypes.byref(q), 128, 32)
    def call(k=128, g=g, Kg=FAKE, o=q, ws_bytes=need, scale=0.0):
        return lib.wf_sparse_attn(FAKE, ctypes.byref(q), FAKE, FAKE, ctypes.byref(kv), FAKE2, k, Kg, FAKE,
                                  ctypes.byref(g) if g is not None else None, FAKE2, ctypes.byref(o), scale,
                                  ctypes.c_void_p(0x100000), ws_bytes, None)
    assert call(ws_bytes=need - 1) == -5
    assert call(k=0) == -1
    assert call(k=1025) == -1
    assert call(Kg=None) == -1                                    # n_g > 0 needs Kg
    assert call(o=_desc(1, 2, 31, 128)) == -2
    assert call(scale=-1.0) == -1


@no_gpu
def test_wavelet_rejects(lib):
    kv = _desc(1, 2, 64, 128)
    need = 1 * 2 * 16 * 128 * 2
    call = lambda K=FAKE, cand=None, m=16, level=2, wv=1, out=FAKE2, nb=need: lib.wf_wavelet_approx(
        K, ctypes.byref(kv), cand, m, level, wv, out, nb, None)
    assert call(wv=7) == -8                        # unknown basis
    assert call(level=9) == -8                     # db2 deeper than 8 levels
    assert call(m=15) == -1                        # whole prompt: m must be n >> level
    assert call(nb=need - 1) == -5
    assert call(K=ctypes.c_void_p(0x10008)) == -4
    assert call(cand=ctypes.c_void_p(0x30002), m=3) == -4
    q = _desc(1, 2, 32, 128)
    keep = (ctypes.c_int32 * 3)(16, 8, 8)
    assert lib.wf_filter_wavelet_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep, 1) > \
        lib.wf_filter_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep)
    assert lib.wf_filter_wavelet_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep, 5) == 0
    # The literal step: the filter's workspace (or the attention's) after the status block.
    step_need = lib.wf_step_wavelet_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep, 1, 4)
    assert step_need >= 256 + lib.wf_filter_wavelet_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep, 1)
    assert step_need >= 256 + lib.wf_attn_workspace_bytes(ctypes.byref(q), 16, 4)
    assert lib.wf_step_wavelet_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep, 5, 4) == 0
    assert lib.wf_step_wavelet_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep, 1, -1) == 0


@no_gpu
def test_step_wavelet_rejects(lib):
    kv = _desc(1, 2, 64, 128)
    q = _desc(1, 2, 32, 128)
    g = _desc(1, 2, 4, 128)
    keep = (ctypes.c_int32 * 3)(16, 8, 8)
    need = lib.wf_step_wavelet_workspace_bytes(ctypes.byref(q), ctypes.byref(kv), 2, keep, 1, 4)
    ws = ctypes.c_void_p(0x40000)

    def call(top=FAKE, V=FAKE2, wv=1, Kg=FAKE, ws=ws, ws_bytes=need, idx=ctypes.c_void_p(0x50000), levels=2):
        return lib.wf_step_wavelet(FAKE, ctypes.byref(q), top, FAKE, V, ctypes.byref(kv), Kg, FAKE2,
                                   ctypes.byref(g), levels, keep, wv, idx, None, FAKE2, ctypes.byref(q), ws,
                                   ws_bytes, None)
    assert call(wv=7) == -8                       # unknown basis
    assert call(top=None) == -1
    assert call(V=None) == -1
    assert call(Kg=None) == -1                    # n_g > 0 needs Kg
    assert call(top=ctypes.c_void_p(0x10008)) == -4
    assert call(ws=ctypes.c_void_p(0x40010)) == -4  # ws 256-byte aligned
    assert call(idx=ctypes.c_void_p(0x50002)) == -4
    assert call(ws_bytes=need - 1) == -5


def test_wait_failure_control(lib):
    # Test-only control (include/wf_testing.h): host-side only, no launch.
    assert lib.wf_testing_set_wait_failure(0, -1) == -1  # WF_ERR_INVALID_ARG
    assert lib.wf_testing_set_wait_failure(1, 1000) == 0
    assert lib.wf_testing_set_wait_failure(0, 0) == 0


def test_attn_workspace_sized_by_query_rows(lib):
    # A split's partials take the query rows rounded up to 32, so 32 heads at
    # d 128 fit the allocation-free array (16 MiB) with k + n_g <= 1984 sparse
    # rows for query blocks of up to 32 rows, and <= 960 for 33-64 rows.
    lim = 16 << 20
    for q, rows in ((32, 1984), (17, 1984), (64, 960), (40, 960)):
        d = _desc(1, 32, q, 128)
        assert lib.wf_attn_workspace_bytes(ctypes.byref(d), rows - 32, 32) <= lim, (q, rows)
        assert lib.wf_attn_workspace_bytes(ctypes.byref(d), rows - 31, 32) > lim, (q, rows)
