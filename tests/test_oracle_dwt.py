"""Pins for the oracle's Haar DWT (Eq. 5, Section 2.2 recursion, Eq. 6).

Each test checks the oracle against something other than itself: the inverse
transform, energy conservation, closed forms for constant and ramp inputs, the
block-sum form of the orthonormal Haar approximation, a hand-derived worked
example, and torch's bf16 rounding for the storage step.
"""
import math
import os

import numpy as np
import pytest
import torch

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rng(seed):
    return np.random.default_rng(seed)


@pytest.mark.parametrize("n,d,L", [(8, 1, 3), (64, 5, 4), (1024, 16, 6), (96, 3, 5), (256, 7, 8)])
def test_perfect_reconstruction(orc, n, d, L):
    x = rng(n + d + L).standard_normal((n, d))
    A, D = orc.haar_analysis(x, L)
    xr = orc.haar_synthesis(A, D, n, L)
    assert np.abs(xr - x).max() <= 1e-12


@pytest.mark.parametrize("n,d,L", [(64, 4, 3), (512, 8, 5), (2048, 2, 11)])
def test_parseval(orc, n, d, L):
    # Orthonormal filter bank: sum x^2 = sum A_L^2 + sum_b sum D_b^2.
    x = rng(7 * n + L).standard_normal((n, d))
    A, D = orc.haar_analysis(x, L)
    energy = (orc.level(A, n, L) ** 2).sum() + sum((orc.level(D, n, b) ** 2).sum() for b in range(1, L + 1))
    assert abs(energy - (x ** 2).sum()) <= 1e-12 * (x ** 2).sum()


def test_constant_input_has_zero_details(orc):
    n, d, L = 256, 3, 6
    x = np.tile(np.array([1.5, -2.0, 0.25]), (n, 1))
    A, D = orc.haar_analysis(x, L)
    for b in range(1, L + 1):
        assert np.abs(orc.level(D, n, b)).max() <= 1e-12
        # A constant c maps to c 2^(b/2) at scale b.
        assert np.allclose(orc.level(A, n, b), x[: n >> b] * 2 ** (b / 2), rtol=0, atol=1e-12)


def test_ramp_closed_form(orc):
    # x[t] = s t.  Haar has one vanishing moment, so details of a ramp are a
    # constant -s 2^(3b/2 - 2) (not zero) and their first difference is zero;
    # A_b[j] = s 2^(b/2) (2^b j + (2^b - 1)/2).
    n, L, s = 512, 7, 0.37
    x = (s * np.arange(n, dtype=np.float64))[:, None]
    A, D = orc.haar_analysis(x, L)
    for b in range(1, L + 1):
        j = np.arange(n >> b)
        Ab = orc.level(A, n, b)[:, 0]
        Db = orc.level(D, n, b)[:, 0]
        assert np.allclose(Ab, s * 2 ** (b / 2) * (2 ** b * j + (2 ** b - 1) / 2), rtol=1e-13, atol=1e-10)
        assert np.allclose(Db, -s * 2 ** (1.5 * b - 2), rtol=1e-13, atol=1e-12)
        assert np.abs(np.diff(Db)).max() <= 1e-10


@pytest.mark.parametrize("L", [1, 2, 5])
def test_block_sum_form(orc, L):
    # Orthonormal Haar: A_b[j] = 2^(-b/2) * sum of the 2^b tokens of block j.
    n, d = 128, 6
    x = rng(L).standard_normal((n, d))
    A, _ = orc.haar_analysis(x, L)
    for b in range(1, L + 1):
        blocks = x.reshape(n >> b, 1 << b, d).sum(axis=1) * 2 ** (-b / 2)
        assert np.abs(orc.level(A, n, b) - blocks).max() <= 1e-12


def test_hand_worked_example(orc):
    s = math.sqrt(2.0)
    rows = [ln.split() for ln in open(os.path.join(GOLDEN, "haar_worked_example.txt")) if ln[0] not in "#\n"]
    x = np.array([float(v) for v in rows[0][1:]])[:, None]
    n, L = x.shape[0], 3
    A, D = orc.haar_analysis(x, L)
    for kind, b, j, expr in rows[1:]:
        want = eval(expr, {"s": s})
        got = (A if kind == "A" else D)[orc.pyramid_row_offset(n, int(b)) + int(j), 0]
        assert abs(got - want) <= 1e-14, (kind, b, j)


def test_bf16_rounding_matches_torch(orc):
    # orc_round_bf16 against torch's float32 -> bfloat16 conversion (round to
    # nearest even), including exact ties and values near overflow.
    r = rng(3)
    vals = np.concatenate([
        r.standard_normal(4000).astype(np.float32) * np.float32(1e3),
        r.standard_normal(1000).astype(np.float32) * np.float32(1e-30),
        np.array([0.0, -0.0, 1.0, 3.0e38, -3.39e38, 1e-40], dtype=np.float32),
    ])
    bits = r.integers(0, 2 ** 31, 2000, dtype=np.uint32)
    ties = ((bits & np.uint32(0x7e7f0000)) | np.uint32(0x8000)).view(np.float32)  # low half exactly 0x8000
    vals = np.concatenate([vals, ties])
    want = torch.from_numpy(vals).to(torch.bfloat16).to(torch.float32).numpy()
    got = np.array([orc.round_bf16(float(v)) for v in vals], dtype=np.float32)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("bf16", [False, True])
def test_spec32_pyramid_storage(orc, bf16):
    # The stored pyramid is the fp32 cascade (add, then multiply by
    # fl32(1/sqrt2)) of the stored keys, rounded once to the storage type.
    n, d, L = 256, 8, 5
    x = rng(11).standard_normal((n, d)).astype(np.float32)
    if bf16:
        x = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    A = orc.haar_pyramid_spec32(x, L, bf16)
    A64, _ = orc.haar_analysis(x.astype(np.float64), L)
    c32 = np.float32(1 / math.sqrt(2))
    prev = x.copy()
    for b in range(1, L + 1):
        # numpy float32 arithmetic is IEEE single: one rounding per op.
        cur = ((prev[0::2] + prev[1::2]).astype(np.float32) * c32).astype(np.float32)
        stored = torch.from_numpy(cur).to(torch.bfloat16).float().numpy() if bf16 else cur
        assert np.array_equal(orc.level(A, n, b), stored)
        # And close to the exact transform: at most ~1 ulp of the block's
        # magnitude per level on the fp32 cascade, plus the storage rounding.
        bound = (b * 2.0 ** -22) * np.abs(x).reshape(n >> b, 1 << b, d).sum(1) * 2 ** (-b / 2)
        if bf16:
            bound = bound + 2.0 ** -8 * np.abs(orc.level(A64, n, b))
        assert np.all(np.abs(orc.level(A, n, b) - orc.level(A64, n, b)) <= bound + 1e-30)
        prev = cur
