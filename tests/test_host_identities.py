"""Exhaustive CPU checks of the integer identities the CUDA kernels rely on.

* The per-stage tensor-core kernels split a row of a grouped query block into
  (query head, row) with a reciprocal instead of a division:
  floor(i / qs) == trunc((i + 1/2) * fl32(1 / qs)) in fp32, for 0 <= i, qs <= 256.
* The fused kernel's producers copy rows r0 + 6 j of a tile (r0 < 6) into the
  128-byte swizzle, whose term ((c ^ r) & 7) then depends on j only through
  j % 4 (6 j mod 8 cycles through 0, 6, 4, 2), and the per-stage kernels'
  rows r0 + 16 i keep r % 8 fixed.
* The tensor-core attention kernels copy a 128-key tile with 256 threads:
  thread t takes 16-byte chunk t % 16 of rows t / 16 + 16 i (i < 8), the row
  addresses coming by shuffle from the half-warp lane i, which resolved that
  very row; every (row, chunk) of the tile is written once, at its place in
  the 128-byte-swizzled K-major layout.
* The query-rows attention kernel writes each thread's row of P (bf16) in
  16-byte chunks of 8 keys; the chunks tile its M tiles' P buffer exactly and
  sit where the MMA's K-major core-matrix descriptor (k-steps of 256 bytes,
  8-key stride 128, 8-row stride 2048) reads each element; both kernels'
  shared memory fits (one CTA of the rows kernel, two of the other, an SM).
"""
import numpy as np

HALF = 128 * 128          # one 64-column half of a 128-key tile, bytes
QGRP = (128 // 8) * 128   # bytes per 8-row group of a 128-element row block (query rows, P rows)
SMEM_BLOCK = 227 * 1024   # shared memory a CTA can take
SMEM_SM = 228 * 1024      # shared memory of an SM (1 KB of it reserved per CTA)


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


def test_attention_tile_copy_covers_each_chunk_once():
    seen = np.zeros(2 * HALF // 16, dtype=np.int64)
    for t in range(256):
        cc, r0, half = t & 15, t >> 4, t & 16
        xs = (cc >> 3) * HALF + r0 * 128 + (((cc ^ r0) & 7) << 4)
        for i in range(8):
            row = r0 + 16 * i
            # the lane the address comes from resolved this row
            src = (t & ~31) | half | i
            assert src >> 4 == r0 and (src >> 4) + 16 * ((src & 15) & 7) == row
            off = xs + 16 * 128 * i
            # 128-byte swizzle, K-major: half cc / 8, row, chunk (cc % 8) ^ (row % 8)
            assert off == (cc >> 3) * HALF + row * 128 + (((cc & 7) ^ (row & 7)) << 4)
            seen[off // 16] += 1
    assert np.all(seen == 1)


def test_rows_attention_p_layout_matches_descriptor():
    for nmt in (1, 2):
        seen = np.zeros(nmt * 16 * QGRP // 16, dtype=np.int64)
        for mt in range(nmt):
            for r in range(128):
                prow = (mt * 16 + (r >> 3)) * QGRP + (r & 7) * 16
                for c in range(16):  # keys 8c .. 8c + 7
                    off = prow + c * 128
                    seen[off // 16] += 1
                    for e in range(8):
                        k = 8 * c + e
                        # element (row r, key k) as the A operand reads it: k-step k // 16
                        # at 256 bytes, 8-key core matrices 128 apart, 8-row groups 2048 apart
                        want = mt * 16 * QGRP + (k // 16) * 256 + ((k % 16) // 8) * 128 + (r // 8) * QGRP + (r % 8) * 16 + (k % 8) * 2
                        assert off + 2 * e == want
        assert np.all(seen == 1)


def test_attention_shared_memory_fits():
    # query rows on the lanes: two K stages, one V tile, query rows and P of nmt M tiles, barriers
    for nmt in (1, 2):
        smem = 6 * HALF + 2 * nmt * 16 * QGRP + 32
        assert smem <= SMEM_BLOCK
    # keys on the lanes (32 query columns): two K stages, V, the query block, the reduction slots and
    # the per-query running max, sums and factors; two CTAs an SM
    smem = 6 * HALF + (32 // 8) * QGRP + 4 * (2 * 128 + 3 * 256) + 32
    assert 2 * (smem + 1024) <= SMEM_SM
