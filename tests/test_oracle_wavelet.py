"""Pins for the oracle's generic (non-Haar) wavelet path: the db2 taps
against the published table, filter-bank orthogonality and vanishing
moments, a hand-derived periodized impulse response, perfect reconstruction
and Parseval, constants and ramps, the Haar special case against the Haar
oracle, the fp32 storage rule, and the literal filter against exhaustive
search on tiny inputs."""
import itertools
import math
import os

import numpy as np
import pytest

import oracle
from paper_2606_00724_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden():
    taps, imp = {}, []
    for ln in open(os.path.join(GOLDEN, "db2_periodized.txt")):
        if ln.startswith("#") or not ln.strip():
            continue
        f = ln.split()
        if f[0] == "h":
            taps[int(f[1])] = float(f[2])
        else:
            imp.append((int(f[1]), f[2], int(f[3]), f[4]))
    return [taps[k] for k in range(4)], imp


def test_db2_taps_match_published_table():
    h_pub, _ = _golden()
    h, g = oracle.wavelet_taps(oracle.DB2)
    assert np.allclose(h, h_pub, rtol=0, atol=1e-15)


@pytest.mark.parametrize("wavelet", [oracle.HAAR, oracle.DB2])
def test_filter_bank_is_orthonormal(wavelet):
    h, g = oracle.wavelet_taps(wavelet)
    n = len(h)
    shift = lambda a, s: sum(a[k] * a[k + s] for k in range(n - s)) if s < n else 0.0
    assert abs(sum(h) - math.sqrt(2)) < 1e-15 and abs(sum(g)) < 1e-15
    assert abs(shift(h, 0) - 1) < 1e-15 and abs(shift(g, 0) - 1) < 1e-15
    for s in range(2, n, 2):                    # orthogonal to even shifts of itself
        assert abs(shift(h, s)) < 1e-15 and abs(shift(g, s)) < 1e-15
    for s in range(0, n, 2):                    # low- and high-pass orthogonal at every even shift
        assert abs(sum(h[k] * g[k + s] for k in range(n - s))) < 1e-15
        assert abs(sum(g[k] * h[k + s] for k in range(n - s))) < 1e-15
    if wavelet == oracle.DB2:                   # two vanishing moments
        assert abs(sum(k * g[k] for k in range(n))) < 1e-14


def test_db2_periodized_impulse_responses():
    _, imp = _golden()
    h, g = oracle.wavelet_taps(oracle.DB2)
    names = {f"h{k}": h[k] for k in range(4)}
    names.update({f"-h{k}": -h[k] for k in range(4)})
    for pos in (0, 1):
        x = np.zeros((8, 1))
        x[pos] = 1.0
        A, D = oracle.wavelet_analysis(x, oracle.DB2, 1)
        want = {"a": np.zeros(4), "d": np.zeros(4)}
        for p, band, j, name in imp:
            if p == pos:
                want[band][j] = names[name]
        assert np.allclose(A[:4, 0], want["a"], rtol=0, atol=1e-15)
        assert np.allclose(D[:4, 0], want["d"], rtol=0, atol=1e-15)


def _analysis_matrix(n, wavelet):
    # The one-level periodized analysis as an explicit n x n matrix.
    h, g = oracle.wavelet_taps(wavelet)
    M = np.zeros((n, n))
    for j in range(n // 2):
        for k in range(len(h)):
            M[j, (2 * j + k) % n] += h[k]
            M[n // 2 + j, (2 * j + k) % n] += g[k]
    return M


@pytest.mark.parametrize("n", [4, 8, 32])
def test_periodized_level_is_an_orthogonal_map(n):
    M = _analysis_matrix(n, oracle.DB2)
    assert np.allclose(M @ M.T, np.eye(n), rtol=0, atol=1e-14)
    x = np.random.default_rng(n).standard_normal((n, 3))
    A, D = oracle.wavelet_analysis(x, oracle.DB2, 1)
    assert np.allclose(np.vstack([A[: n // 2], D[: n // 2]]), M @ x, rtol=0, atol=1e-14)


@pytest.mark.parametrize("wavelet,L", [(oracle.DB2, 1), (oracle.DB2, 3), (oracle.DB2, 5), (oracle.HAAR, 4)])
def test_perfect_reconstruction_and_parseval(wavelet, L):
    n, d = 64, 5
    x = np.random.default_rng(L).standard_normal((n, d))
    A, D = oracle.wavelet_analysis(x, wavelet, L)
    xr = oracle.wavelet_synthesis(A, D, n, wavelet, L)
    assert np.abs(xr - x).max() < 1e-12
    top = A[oracle.pyramid_row_offset(n, L):]
    energy = (top ** 2).sum() + sum((oracle.level(D, n, b) ** 2).sum() for b in range(1, L + 1))
    assert abs(energy - (x ** 2).sum()) < 1e-10 * (x ** 2).sum()


def test_db2_constants_and_ramps():
    n, L = 64, 3
    c = np.full((n, 2), 1.5)
    A, D = oracle.wavelet_analysis(c, oracle.DB2, L)
    for b in range(1, L + 1):
        assert np.abs(oracle.level(D, n, b)).max() < 1e-13
        assert np.allclose(oracle.level(A, n, b), 1.5 * 2 ** (b / 2), rtol=0, atol=1e-13)
    ramp = np.arange(n, dtype=np.float64)[:, None]
    A, D = oracle.wavelet_analysis(ramp, oracle.DB2, 1)
    det = D[: n // 2, 0]
    # Two vanishing moments: every detail whose support does not wrap is zero.
    assert np.abs(det[:-1]).max() < 1e-12
    assert abs(det[-1]) > 1.0                  # the wrapped one sees the jump n-1 -> 0


def test_haar_through_the_generic_bank():
    x = np.random.default_rng(4).standard_normal((32, 6))
    A, D = oracle.wavelet_analysis(x, oracle.HAAR, 3)
    Ah, Dh = oracle.haar_analysis(x, 3)
    assert np.allclose(A, Ah, rtol=0, atol=1e-15) and np.allclose(D, Dh, rtol=0, atol=1e-15)
    x32 = x.astype(np.float32)
    for bf16 in (False, True):
        pyr = oracle.haar_pyramid_spec32(x32, 3, bf16)
        for b in (1, 2, 3):
            got = oracle.wavelet_approx_spec32(x32, oracle.HAAR, b, bf16)
            assert np.array_equal(got, oracle.level(pyr, 32, b))


def test_spec32_rule_tracks_the_f64_transform():
    x = np.random.default_rng(5).standard_normal((256, 16)).astype(np.float32)
    for b in (1, 3, 5):
        A, _ = oracle.wavelet_analysis(x.astype(np.float64), oracle.DB2, b)
        want = oracle.level(A, 256, b)
        got = oracle.wavelet_approx_spec32(x, oracle.DB2, b, False)
        assert np.abs(got - want).max() <= 1e-5 * np.abs(want).max()
        got16 = oracle.wavelet_approx_spec32(x, oracle.DB2, b, True)
        assert np.array_equal(got16, got16.astype(np.float64).astype(np.float32))
        assert np.abs(got16 - want).max() <= 2 ** -8 * np.abs(want).max()


def test_haar_literal_filter_through_the_generic_path():
    r = np.random.default_rng(6)
    n, d, q, L = 512, 16, 4, 3
    keep = oracle.default_schedule(n, L, 51)
    Q, K = r.standard_normal((q, d)), r.standard_normal((n, d))
    a = oracle.filter_wavelet(Q, K, L, keep, oracle.HAAR, spec32=False, want_sets=True)
    b = oracle.filter_literal(Q, K, L, keep, want_sets=True)
    assert np.array_equal(a[0], b[0])
    for lev in range(L + 1):
        assert np.array_equal(a[1][lev], b[1][lev])


def _softmax_w(Q, rows):
    s = Q @ rows.T / math.sqrt(Q.shape[1])
    p = np.exp(s - s.max(axis=1, keepdims=True))
    return (p / p.sum(axis=1, keepdims=True)).sum(axis=0)


@pytest.mark.parametrize("seed", range(3))
def test_db2_filter_against_exhaustive_search(seed):
    # Each scale: transform the gathered blocks of the previous choice
    # (Eq. 10-11), then the best keep[b]-subset by summed weight.
    r = np.random.default_rng(20 + seed)
    n, d, q, L = 32, 6, 3, 2
    keep = np.array([6, 3, 4], dtype=np.int32)
    Q, K = r.standard_normal((q, d)), r.standard_normal((n, d))
    mu0, sets = oracle.filter_wavelet(Q, K, L, keep, oracle.DB2, spec32=False, want_sets=True)
    cand = np.arange(n >> L)
    for b in range(L, 0, -1):
        toks = np.concatenate([np.arange(c << b, (c + 1) << b) for c in cand])
        A, _ = oracle.wavelet_analysis(K[toks], oracle.DB2, b)
        W = _softmax_w(Q, oracle.level(A, toks.size, b))
        best = max(itertools.combinations(range(cand.size), int(keep[b])), key=lambda s: W[list(s)].sum())
        want = np.sort(cand[list(best)])
        assert np.array_equal(sets[b], want), b
        cand = np.stack([2 * want, 2 * want + 1], 1).reshape(-1)
    assert np.array_equal(mu0, cand)


def test_db2_filter_finds_the_needles():
    # The tiny needle workload: every planted needle token survives the db2
    # filter too (its block's approximation carries the needle).
    w = synth.WORKLOADS["c1"]
    u = synth.make_unit(w, 0, 1, planted=True, cfg="c1")
    mu0 = oracle.filter_wavelet(u.Q.numpy(), u.K.numpy(), w.levels, np.array(w.keep), oracle.DB2)
    assert np.isin(u.needles.numpy(), mu0).all()
