"""Exhaustive CPU checks of the integer identities the CUDA kernels rely on.

* The per-stage tensor-core kernels split a row of a grouped query block into
  (query head, row) with a reciprocal instead of a division:
  floor(i / qs) == trunc((i + 1/2) * fl32(1 / qs)) in fp32, for 0 <= i, qs <= 256.
* The fused kernel's producers copy rows r0 + 6 j of a tile (r0 < 6) into the
  128-byte swizzle, whose term ((c ^ r) & 7) then depends on j only through
  j % 4 (6 j mod 8 cycles through 0, 6, 4, 2), and the per-stage kernels'
  rows r0 + 16 i keep r % 8 fixed.
"""
import numpy as np


def test_reciprocal_head_split_is_exact():
    i = np.arange(0, 257, dtype=np.int64)
    for qs in range(1, 257):
        r = np.float32(1.0) / np.float32(qs)
        got = np.trunc((i.astype(np.float32) + np.float32(0.5)) * r).astype(np.int64)
        assert np.array_equal(got, i // qs), f"qs={qs}"


def test_producer_swizzle_term_period():
    for c in range(16):
        for r0 in range(6):
            for j in range(22):
                assert ((c ^ (r0 + 6 * j)) & 7) == ((c ^ (r0 + 6 * (j % 4))) & 7)
        for r0 in range(16):
            for i in range(8):
                assert ((c ^ (r0 + 16 * i)) & 7) == ((c ^ r0) & 7)
