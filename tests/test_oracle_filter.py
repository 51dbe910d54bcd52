"""Pins for the oracle's skim/scan filtering (Eq. 7-11, Algorithm 1).

What fixes the answer independently of the oracle's code: closed forms of
the perception weights (two candidates -> logistic function), the planted
ladder (the generator plants a known answer), brute force over all k-subsets,
softmax invariances, the literal gathered-DWT reading of Eq. 11, and the
printed hyper-parameter ranges of Table 3.
"""
import itertools
import math
import os

import numpy as np
import pytest
import torch

from paper_2606_00724_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rng(seed):
    return np.random.default_rng(seed)


def test_skim_two_candidates_logistic(orc):
    # Eq. 7-8 with two candidate rows: softmax over two logits is the logistic
    # function of their difference, so W_0 = sum_i sigma((l_i0 - l_i1)) and
    # W_1 = q - W_0, with l = q.k / sqrt(d).
    d = 4
    Q = np.array([[2.0, 0, 0, 0], [0, 1.0, 0, 0], [0, 1.0, 0, 0], [0.5, -1.0, 3.0, 0]])
    rows = np.array([[1.0, -1.0, 0, 0], [0, 1.5, 0.5, 0]])
    W = orc.skim_weights(Q, rows)
    sig = lambda z: 1.0 / (1.0 + math.exp(-z))
    diffs = (Q @ rows[0] - Q @ rows[1]) / math.sqrt(d)
    w0 = sum(sig(z) for z in diffs)
    assert abs(W[0] - w0) <= 1e-14 and abs(W[1] - (len(Q) - w0)) <= 1e-14


def test_skim_rows_sum_to_q_and_scale(orc):
    # Each query row of Eq. 7 is a distribution over the candidates, so the
    # column sums of Eq. 8 add up to q; and the 1/sqrt(d) temperature is the
    # one of Eq. 7 (W for scaled keys equals W for scaled queries).
    r = rng(1)
    Q = r.standard_normal((5, 9))
    rows = r.standard_normal((13, 9))
    W = orc.skim_weights(Q, rows)
    assert abs(W.sum() - 5.0) <= 1e-12
    assert np.allclose(orc.skim_weights(2 * Q, rows), orc.skim_weights(Q, 2 * rows), atol=1e-14)
    # Single query: W is the softmax itself, compared with torch.
    w1 = orc.skim_weights(Q[:1], rows)
    ref = torch.softmax(torch.from_numpy(rows @ Q[0] / 3.0), dim=0).numpy()
    assert np.abs(w1 - ref).max() <= 1e-15


def _pyr64(orc, K, L):
    A, _ = orc.haar_analysis(K, L)
    return A


@pytest.mark.parametrize("seed", range(6))
def test_topk_brute_force(orc, seed):
    # n = 32, L = 2: at every scale the kept set must be the k-subset of the
    # candidates with the largest total W (ties -> lexicographically smallest
    # index set), found by enumerating all subsets.
    r = rng(seed)
    n, d, L, q = 32, 4, 2, 3
    K = r.standard_normal((n, d))
    Q = r.standard_normal((q, d))
    keep = np.array([6, 3, 4], dtype=np.int32)
    pyr = _pyr64(orc, K, L)
    mu0, sets = orc.filter(Q, pyr, K, n, L, keep, want_sets=True)
    cand = np.arange(n >> L)
    for b in range(L, 0, -1):
        rows = orc.level(pyr, n, b)[cand]
        W = orc.skim_weights(Q, rows)
        best = max(itertools.combinations(range(len(cand)), int(keep[b])),
                   key=lambda s: (round(sum(W[list(s)]), 12), [-i for i in s]))
        assert np.array_equal(sets[b], cand[list(best)])
        cand = np.stack([2 * sets[b], 2 * sets[b] + 1], 1).reshape(-1)
    assert np.array_equal(mu0, cand)


def test_level0_trim_brute_force(orc):
    r = rng(9)
    n, d, L, q = 16, 3, 1, 2
    K = r.standard_normal((n, d))
    Q = r.standard_normal((q, d))
    keep = np.array([5, 3], dtype=np.int32)  # 6 tokens after scale 1, trimmed to 5
    pyr = _pyr64(orc, K, L)
    mu0, sets = orc.filter(Q, pyr, K, n, L, keep, want_sets=True)
    toks = np.stack([2 * sets[1], 2 * sets[1] + 1], 1).reshape(-1)
    W = orc.skim_weights(Q, K[toks])
    drop = int(np.argmin(W))
    assert np.array_equal(mu0, np.delete(toks, drop))


def test_single_query_is_topk_by_logit(orc):
    # q = 1: W_j is a softmax, monotone in the logit, so each J_b is the top-k
    # of the raw logits q.A_b[j] (computed here with numpy, no softmax).
    r = rng(5)
    n, d, L = 256, 8, 3
    K = r.standard_normal((n, d))
    Q = r.standard_normal((1, d))
    keep = np.array([20, 10, 12, 14], dtype=np.int32)
    pyr = _pyr64(orc, K, L)
    _, sets = orc.filter(Q, pyr, K, n, L, keep, want_sets=True)
    cand = np.arange(n >> L)
    for b in range(L, 0, -1):
        logits = orc.level(pyr, n, b)[cand] @ Q[0]
        order = np.lexsort((cand, -logits))
        assert np.array_equal(sets[b], np.sort(cand[order[: keep[b]]]))
        cand = np.stack([2 * sets[b], 2 * sets[b] + 1], 1).reshape(-1)


@pytest.mark.parametrize("seed", range(3))
def test_invariances(orc, seed):
    r = rng(100 + seed)
    n, d, L, q = 512, 16, 3, 8
    K = r.standard_normal((n, d))
    Q = r.standard_normal((q, d))
    keep = np.array([41, 21, 30, 24], dtype=np.int32)
    base_mu, base_sets = orc.filter(Q, _pyr64(orc, K, L), K, n, L, keep, want_sets=True)
    # Shifting every key by one vector shifts each query row's logits by a
    # constant at every scale: the softmax of Eq. 7, hence every J_b, is unchanged.
    K2 = K + 0.75 * r.standard_normal(d)
    mu2, sets2 = orc.filter(Q, _pyr64(orc, K2, L), K2, n, L, keep, want_sets=True)
    assert all(np.array_equal(base_sets[b], sets2[b]) for b in base_sets)
    # Eq. 8 sums over the query rows: their order does not matter.
    perm = r.permutation(q)
    mu3 = orc.filter(Q[perm], _pyr64(orc, K, L), K, n, L, keep)
    assert np.array_equal(base_mu, mu3)


def test_keep_everything(orc):
    # k = n (every proportion m_b = 1) keeps every token.
    r = rng(2)
    n, d, L = 128, 4, 3
    K = r.standard_normal((n, d))
    Q = r.standard_normal((4, d))
    keep = orc.schedule_from_proportions(n, L, [0, 1.0, 1.0, 1.0])
    assert keep.tolist() == [n, n // 2, n // 4, n // 8]
    assert np.array_equal(orc.filter(Q, _pyr64(orc, K, L), K, n, L, keep), np.arange(n))


@pytest.mark.parametrize("seed,L,keep", [(0, 2, [10, 5, 6]), (1, 3, [7, 4, 5, 6]), (2, 4, [9, 5, 4, 3, 2]),
                                         (3, 1, [11, 6])])
def test_literal_eq11_matches_pyramid(orc, seed, L, keep):
    # Eq. 11 recomputes the DWT of the gathered tokens at every scale.  Because
    # the candidates are unions of aligned blocks and Haar has support 2, that
    # equals indexing the full pyramid; the literal Algorithm-1 oracle and the
    # pyramid oracle must select the same sets.
    r = rng(seed)
    n, d, q = 64, 5, 3
    K = r.standard_normal((n, d))
    Q = r.standard_normal((q, d))
    keep = np.array(keep, dtype=np.int32)
    mu_a, sets_a = orc.filter(Q, _pyr64(orc, K, L), K, n, L, keep, want_sets=True)
    mu_b, sets_b = orc.filter_literal(Q, K, L, keep, want_sets=True)
    assert np.array_equal(mu_a, mu_b)
    assert all(np.array_equal(sets_a[b], sets_b[b]) for b in sets_a)


@pytest.mark.parametrize("cfg", ["c1", "c2", "c3", "c4", "c5"])
def test_planted_ladder_is_recovered(orc, cfg):
    # The generator plants J_b by construction (a bonus along one direction on
    # the chosen blocks); the oracle, on the stored pyramid, must find exactly
    # those sets at every scale.
    w = synth.WORKLOADS[cfg]
    dt = synth.storage_dtype(w)
    heads = (0, 1, w.heads - 1) if w.n <= 8192 else (w.heads - 1,)
    for h in heads:
        u = synth.make_unit(w, w.batch - 1, h, planted=True, cfg=cfg)
        Q = u.Q.to(dt).float().numpy()
        K = u.K.to(dt).float().numpy()
        pyr = orc.haar_pyramid_spec32(K, w.levels, w.dtype == "bf16")
        mu0, sets = orc.filter(Q, pyr, K, w.n, w.levels, np.array(w.keep), want_sets=True)
        for b, tgt in u.targets.items():
            assert np.array_equal(sets[b], tgt.numpy()), (cfg, h, b)
        assert np.array_equal(mu0, u.targets[0].numpy())


def test_planted_ladder_breaks_when_bonus_is_off(orc, monkeypatch):
    # The planted answer is not a property of the random data: with no bonus
    # the oracle's choice differs from the planted sets.
    w = synth.WORKLOADS["c1"]
    monkeypatch.setattr(synth, "PLANT_GAP", 0.0)
    u = synth.make_unit(w, 0, 0, planted=True, cfg="c1")
    pyr = orc.haar_pyramid_spec32(u.K.numpy(), w.levels, False)
    _, sets = orc.filter(u.Q.numpy(), pyr, u.K.numpy(), w.n, w.levels, np.array(w.keep), want_sets=True)
    assert not np.array_equal(sets[w.levels], u.targets[w.levels].numpy())


def _table3():
    vals = {}
    for ln in open(os.path.join(GOLDEN, "table3_hyperparams.txt")):
        if ln.strip() and not ln.startswith("#"):
            k, v = ln.split()
            vals[k] = v
    return vals


@pytest.mark.parametrize("cfg", list(synth.WORKLOADS))
def test_default_schedule(orc, cfg):
    # The kept counts the workloads pass explicitly are the default schedule,
    # and its per-scale proportion lies in Table 3's range [0.3, 1].
    t3 = _table3()
    w = synth.WORKLOADS[cfg]
    keep = orc.default_schedule(w.n, w.levels, w.k)
    assert keep.tolist() == list(w.keep)
    m = (w.k / w.n) ** (1.0 / w.levels)
    assert float(t3["proportion_min"]) <= m <= float(t3["proportion_max"])
    cnt = w.n >> w.levels
    for b in range(w.levels, 1, -1):
        assert keep[b] == min(cnt, max(1, math.ceil(m * cnt - 1e-9)))
        cnt = 2 * keep[b]
    assert keep[1] == (w.k + 1) // 2 and keep[0] == w.k


def test_table3_default_scale_schedule(orc):
    # Table 3: scale B = 2 with proportions m_2, m_1 in [0.3, 1].
    t3 = _table3()
    B = int(t3["scale_B"])
    keep = orc.schedule_from_proportions(4096, B, [0.0, 0.3, 0.6])
    assert keep.tolist() == [2 * math.ceil(0.3 * 2 * math.ceil(0.6 * 1024)), math.ceil(0.3 * 2 * 615),
                             math.ceil(0.6 * 1024)]
    with pytest.raises(ValueError):
        orc.schedule_from_proportions(4096, B, [0.0, 0.0, 0.5])


@pytest.mark.parametrize("cfg", list(synth.WORKLOADS))
def test_level0_schedule(orc, cfg):
    # The token level as its own selection step: one proportion m over the
    # L pyramid scans and the token scan.  Each scale keeps between m and
    # m + 1/|C_b| of its candidates, the product of the kept fractions lands
    # on k/n, and m lies in the range the hot-path survey gives for these
    # shapes (about 0.50-0.57).
    w = synth.WORKLOADS[cfg]
    keep = orc.level0_schedule(w.n, w.levels, w.k)
    m = (w.k / w.n) ** (1.0 / (w.levels + 1))
    assert 0.49 <= m <= 0.58
    assert keep[0] == w.k
    cnt = w.n >> w.levels
    frac = 1.0
    for b in range(w.levels, 0, -1):
        assert 1 <= keep[b] <= cnt
        assert m - 1e-12 <= keep[b] / cnt <= m + 1.0 / cnt
        frac *= keep[b] / cnt
        cnt = 2 * int(keep[b])
    assert w.k <= cnt                       # the token scan keeps k of 2 keep[1]
    frac *= w.k / cnt
    assert abs(frac - w.k / w.n) / (w.k / w.n) < 0.05 * (w.levels + 1)
    with pytest.raises(ValueError):
        orc.level0_schedule(w.n, w.levels, w.n + 1)


@pytest.mark.parametrize("cfg", ["c1", "c2", "c3"])
def test_planted_ladder_level0_schedule(orc, cfg):
    # With the token level as its own selection step, the planted ladder
    # (built for that schedule, including the level-0 scan over raw keys)
    # is still what the oracle finds at every scale.
    import dataclasses
    w0 = synth.WORKLOADS[cfg]
    keep = tuple(int(x) for x in orc.level0_schedule(w0.n, w0.levels, w0.k))
    w = dataclasses.replace(w0, keep=keep, name=w0.name + "_level0")
    dt = synth.storage_dtype(w)
    u = synth.make_unit(w, 0, w.heads - 1, planted=True, cfg=cfg)
    Q = u.Q.to(dt).float().numpy()
    K = u.K.to(dt).float().numpy()
    pyr = orc.haar_pyramid_spec32(K, w.levels, w.dtype == "bf16")
    mu0, sets = orc.filter(Q, pyr, K, w.n, w.levels, np.array(w.keep), want_sets=True)
    for b, tgt in u.targets.items():
        assert np.array_equal(sets[b], tgt.numpy()), (cfg, b)
    assert np.array_equal(mu0, u.targets[0].numpy())
