// Fused WaveFilter step (Algorithm 1 body): multi-scale skim/scan filtering
// (Eq. 7-11) and the final sparse attention, in one kernel.
//
// One thread-block cluster per (batch, head) unit; the cluster's CTAs split
// every scale's candidate list (and finally the sparse key list) into
// contiguous slices.  Per scale, each CTA:
//   1. gathers its candidate rows (pyramid level b, or raw keys for the
//      level-0 trim) with 16-byte cp.async copies straight into
//      128-byte-swizzled tiles of 128 rows; every thread pipelines its own
//      copies through a ring of stages and signals completion on the stage's
//      mbarrier (cp.async.mbarrier.arrive), and one thread issues
//      tcgen05.mma (bf16 in, fp32 out) for each tile that has landed,
//      writing S^T = rows . Q^T into TMEM (32 columns per tile);
//   2. reads the logits back from TMEM (tcgen05.ld) for the per-query max and
//      sum of exp over its slice and exchanges them through distributed
//      shared memory, giving every CTA the softmax normaliser of Eq. 7;
//   3. computes the ranking key log2 W_j (Eq. 8, as a log-sum-exp over the
//      query rows) of its candidates and writes them into every CTA's key
//      array (DSMEM all-gather);
//   4. runs the same deterministic Top-K (radix select on the key bits,
//      lowest index first on ties, Eq. 9) in every CTA, so each knows J_b and
//      hence the next scale's candidates {2j, 2j+1} (Eq. 10) without a
//      broadcast.
// The attention stage gathers the K rows of mu^0 and the generation rows the
// same way, forms S^T = K_s Q^T in TMEM, and then streams the V rows while
// four warps turn S into P = exp(S - m) (bf16) and the MMA thread
// accumulates O^T = V_s^T P^T (both operands MN-major); the cluster's partial
// (m, l, O) are combined in CTA 0.
//
// Every wait on asynchronous work (copies, MMA completion) is bounded
// (~1 s): on timeout the CTA records a status word, stops issuing MMAs, keeps
// joining every barrier and returns.
#include <math.h>
#include <string.h>

#include "wf_internal.cuh"
#include "wf_sm100.cuh"

namespace wf {
namespace {

using namespace sm100;

constexpr int NT = 256;                  // threads per CTA (8 warps)
constexpr int D = 128;                   // head_dim
constexpr int TM = 128;                  // rows per MMA tile (M)
constexpr int NQ = 32;                   // query rows per MMA (N), zero padded
constexpr int HALF_BYTES = TM * 128;     // one 64-column half of a tile, 128-byte rows
constexpr int TILE_BYTES = 2 * HALF_BYTES;
constexpr int QGRP = (D / 8) * 128;      // bytes per 8-row group of the query tile (core matrices)
constexpr int Q_BYTES = NQ * D * 2;
constexpr int P_BYTES = NQ * TM * 2;
constexpr long long kWaitLimit = 1ll << 31;
constexpr float kLog2e = 1.4426950408889634f;

constexpr uint32_t kIdescScore = idesc_bf16(TM, NQ, 0, 0);  // A = rows (K-major), B = Q (K-major)
constexpr uint32_t kIdescPV = idesc_bf16(D, NQ, 1, 1);      // A = V^T (MN-major), B = P^T (MN-major)

struct Misc {
  unsigned long long full[8], empty[8], done, pfull[2], pempty[2];
  float2 xstat[8][32];
  float red[8][32];
  float cvec[32];
  float mloc[32];
  float lacc[32];
  int wsum[8];
  uint32_t sel_bin, sel_need, sel_cnt;
  int abort;
  uint32_t tmem_base;
};

template <int STAGES>
struct Layout {
  static constexpr uint32_t off_stage = 0;
  static constexpr uint32_t off_q = STAGES * TILE_BYTES;
  static constexpr uint32_t off_p = off_q + Q_BYTES;
  static constexpr uint32_t off_hist = off_p + 2 * P_BYTES;
  static constexpr uint32_t off_misc = off_hist + 8 * 256 * 4;
  static constexpr uint32_t off_keys = (off_misc + sizeof(Misc) + 127) / 128 * 128;
};

struct FusedParams {
  const bf16* Q;
  int64_t qsb, qsh, qss;
  const bf16* K;
  const bf16* V;
  int64_t ksb, ksh, kss;
  const bf16* Kg;
  const bf16* Vg;
  int64_t gsb, gsh, gss;
  const bf16* coeffs;
  int64_t rows_total;
  bf16* O;
  int64_t osb, osh, oss;
  int32_t* idx;
  int32_t* level_sets;
  int64_t sets_stride;
  int* status;
  int q, n, ng, H, L, trim, cmax, kmax;
  uint32_t tmem_cols;
  int32_t keep[12];
  float scale_log2;  // log2(e) / sqrt(d)
};

__device__ __forceinline__ uint32_t okey(float f) {
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Reduce 32 values per lane across the warp's 32 lanes; afterwards lane i
// holds the reduction of column i (31 shuffles).
template <bool MAX>
__device__ __forceinline__ float transpose_reduce32(float (&v)[32], int lane) {
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int j = 0; j < off; ++j) {
      const float keep = up ? v[j + off] : v[j];
      const float send = up ? v[j] : v[j + off];
      const float recv = __shfl_xor_sync(0xffffffffu, send, off);
      v[j] = MAX ? fmaxf(keep, recv) : keep + recv;
    }
  }
  return v[0];
}

// Reduce 8 values per lane across the warp's 32 lanes; afterwards every lane
// L holds the reduction of column (L / 4) % 8 (9 shuffles).
template <bool MAX>
__device__ __forceinline__ float transpose_reduce8(float (&v)[8], int lane) {
#pragma unroll
  for (int off = 16, n = 4; off >= 4; off >>= 1, n >>= 1) {
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (j < n) {
        const float keep = up ? v[j + n] : v[j];
        const float send = up ? v[j] : v[j + n];
        const float recv = __shfl_xor_sync(0xffffffffu, send, off);
        v[j] = MAX ? fmaxf(keep, recv) : keep + recv;
      }
    }
  }
  float r = v[0];
#pragma unroll
  for (int off = 2; off >= 1; off >>= 1) {
    const float o = __shfl_xor_sync(0xffffffffu, r, off);
    r = MAX ? fmaxf(r, o) : r + o;
  }
  return r;
}

// Exclusive prefix sum over the CTA's 256 threads (thread order).
__device__ __forceinline__ int block_excl_scan(int v, Misc& ms) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) ms.wsum[warp] = incl;
  __syncthreads();
  int before = 0;
#pragma unroll
  for (int w = 0; w < 8; ++w) before += w < warp ? ms.wsum[w] : 0;
  __syncthreads();
  return before + incl - v;
}

// Candidate (or token) index of position j of the current candidate list.
__device__ __forceinline__ int cand_of(int j, bool top, const int32_t* Jprev) {
  return top ? j : 2 * Jprev[j >> 1] + (j & 1);
}

// Top-K of keys[0..m) (largest first, lower position wins ties); writes the
// kk chosen candidate indices in ascending position order to Jout.
// Each thread holds a run of R <= 32 keys in registers (slot x holds position
// j0 + (x + rot) % R; the rotation spreads a warp's reads over the banks).
// The boundary is found by range bucketing: the still-undecided keys are
// spread over 256 buckets linear in [min, max] of those keys (fp32
// arithmetic is monotone, so a key in a higher bucket is strictly larger),
// the bucket holding the boundary is located from the bucket counts, keys
// above it are taken and keys below it dropped, and the boundary bucket is
// bucketed again over its own range until it holds exactly the missing count
// or only equal keys, which are then taken lowest position first.  Buckets
// stay evenly filled, so the shared-memory histogram atomics rarely collide.
template <int R>
__device__ __forceinline__ void select_impl(const float* keys, int m, int kk, int32_t* Jout, bool top,
                                            const int32_t* Jprev, Misc& ms, uint32_t* hist) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int j0 = tid * R;
  const int rot = ((tid & 31) * R) >> 5;
  float kv[R];
  uint32_t act = 0, took = 0;  // bit x = slot x
#pragma unroll
  for (int x = 0; x < R; ++x) {
    const int j = j0 + ((x + rot) & (R - 1));
    kv[x] = j < m ? keys[j] : 0.f;
    act |= (uint32_t)(j < m) << x;
  }
  uint32_t need = (uint32_t)kk;
  uint32_t* wh = hist + warp * 256;
  for (int iter = 0; iter < 8; ++iter) {
    float lo = INFINITY, hi = -INFINITY;
#pragma unroll
    for (int x = 0; x < R; ++x) {
      const bool a = (act >> x) & 1u;
      lo = fminf(lo, a ? kv[x] : INFINITY);
      hi = fmaxf(hi, a ? kv[x] : -INFINITY);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (lane == 0) {
      ms.red[warp][0] = lo;
      ms.red[warp][1] = hi;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) wh[lane + 32 * i] = 0u;
    __syncthreads();
#pragma unroll
    for (int w = 0; w < 8; ++w) {
      lo = fminf(lo, ms.red[w][0]);
      hi = fmaxf(hi, ms.red[w][1]);
    }
    if (!(hi > lo)) break;  // every undecided key is equal (or none is left)
    const float scale = 256.f / (hi - lo);
    int bk[R];
#pragma unroll
    for (int x = 0; x < R; ++x) {
      bk[x] = min(255, (int)((kv[x] - lo) * scale));
      if ((act >> x) & 1u) atomicAdd(&wh[bk[x]], 1u);
    }
    __syncthreads();
    const int bin = 255 - tid;  // thread order = buckets from high to low
    uint32_t tot = 0;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += hist[w * 256 + bin];
    const uint32_t above = (uint32_t)block_excl_scan((int)tot, ms);
    if (above < need && above + tot >= need) {
      ms.sel_bin = (uint32_t)bin;
      ms.sel_need = need - above;
      ms.sel_cnt = tot;
    }
    __syncthreads();
    const int sb = (int)ms.sel_bin;
    const uint32_t cnt = ms.sel_cnt;
    need = ms.sel_need;
#pragma unroll
    for (int x = 0; x < R; ++x) {
      if ((act >> x) & 1u) {
        if (bk[x] > sb) took |= 1u << x;
        if (bk[x] != sb) act &= ~(1u << x);
      }
    }
    __syncthreads();  // ms.red / ms.sel are reused by the next round
    if (cnt == need) {
      took |= act;
      act = 0;
      break;
    }
  }
  // Position-order masks (bit i = position j0 + i).
  uint32_t gt = 0, eq = 0;
#pragma unroll
  for (int x = 0; x < R; ++x) {
    const int i = (x + rot) & (R - 1);
    gt |= ((took >> x) & 1u) << i;
    eq |= ((act >> x) & 1u) << i;
  }
  // The still-undecided (equal) keys: the first `need` by position are taken.
  const int eq_base = block_excl_scan(__popc(eq), ms);
  uint32_t take = gt;
  int remaining = (int)need - eq_base;
  for (uint32_t e = eq; e && remaining > 0; --remaining) {
    const uint32_t low = e & (~e + 1u);
    take |= low;
    e ^= low;
  }
  int pos = block_excl_scan(__popc(take), ms);
  while (take) {
    const int i = __ffs(take) - 1;
    take &= take - 1u;
    Jout[pos++] = cand_of(j0 + i, top, Jprev);
  }
  __syncthreads();
}

__device__ __forceinline__ void select_topk(const float* keys, int m, int kk, int32_t* Jout, bool top,
                                            const int32_t* Jprev, Misc& ms, uint32_t* hist) {
  if (m <= NT) select_impl<1>(keys, m, kk, Jout, top, Jprev, ms, hist);
  else if (m <= 2 * NT) select_impl<2>(keys, m, kk, Jout, top, Jprev, ms, hist);
  else if (m <= 4 * NT) select_impl<4>(keys, m, kk, Jout, top, Jprev, ms, hist);
  else if (m <= 8 * NT) select_impl<8>(keys, m, kk, Jout, top, Jprev, ms, hist);
  else if (m <= 16 * NT) select_impl<16>(keys, m, kk, Jout, top, Jprev, ms, hist);
  else select_impl<32>(keys, m, kk, Jout, top, Jprev, ms, hist);
}

// Per-CTA shared-memory addresses and constants.
struct Ctx {
  uint32_t tmem, sq_a, p_a, keys_a, done_a, stage_a, full_a, empty_a, pfull_a, pempty_a;
  uint32_t rank, cs;
  int stages, q;
  float sl2;
};

// Where the rows of a candidate or key list come from.
//  kind 0: position j -> row j (top scale);
//  kind 1: position j -> row 2 J[j/2] + j%2 (children of the kept coefficients);
//  kind 2: sparse key list, positions < kk -> token 2 J[j/2] + j%2 (or J[j]
//          when trimmed), then generation rows.
struct RowSrc {
  const bf16* base;
  int64_t stride;
  const bf16* gbase;
  int64_t gstride;
  const int32_t* J;
  int kind, trim, g0, mc, kk;
};

__device__ __forceinline__ const bf16* row_ptr(const RowSrc& s, int r) {
  const int valid = r < s.mc;
  const int pos = s.g0 + (valid ? r : 0);
  int row;
  if (s.kind == 0) {
    row = pos;
  } else if (s.kind == 1) {
    row = 2 * s.J[pos >> 1] + (pos & 1);
  } else {
    if (pos >= s.kk) return s.gbase + (int64_t)(pos - s.kk) * s.gstride;
    row = s.trim ? s.J[pos] : 2 * s.J[pos >> 1] + (pos & 1);
  }
  return s.base + (int64_t)row * s.stride;
}

__device__ __forceinline__ uint32_t stage_addr(const Ctx& c, int s) { return c.stage_a + s * TILE_BYTES; }

__device__ __forceinline__ bool aborted(const Misc& ms) { return *reinterpret_cast<const volatile int*>(&ms.abort); }

__device__ __forceinline__ void set_abort(Misc& ms, int* status) {
  ms.abort = 1;
  atomicExch(status, 1);
}

__device__ __forceinline__ void wait_or_abort(uint32_t bar, uint32_t parity, Misc& ms, int* status) {
  if (!aborted(ms) && !mbar_wait_bounded(bar, parity, kWaitLimit, &ms.abort)) set_abort(ms, status);
}

// This thread's share of one 128-row tile: chunk c = tid % 16 of rows
// tid/16 + 16 i, written in the 128-byte-swizzled K-major layout (row r,
// 16-byte chunk c at half c/8, byte r*128 + ((c%8) ^ (r%8))*16).
__device__ __forceinline__ void load_tile(uint32_t st, int t, const RowSrc& src) {
  const int tid = threadIdx.x;
  const int c = tid & 15, r0 = tid >> 4;
  const uint32_t cbase = st + ((c >> 3) << 14);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = r0 + 16 * i;
    cp_async16(cbase + r * 128 + (((c & 7) ^ (r & 7)) << 4), row_ptr(src, t * TM + r) + c * 8);
  }
}

// Stream ntl tiles of src through the stage ring (pipeline iterations
// it0..): all threads copy, thread 0 also issues the score MMAs
// S^T tile = rows . Q^T into TMEM columns 32 t, then commits `done`.
__device__ __forceinline__ void stream_scores(const Ctx& c, Misc& ms, int* status, int it0, int ntl, RowSrc src) {
  const int tid = threadIdx.x;
  const int S = c.stages;
  for (int t = 0; t < ntl + S - 1; ++t) {
    if (t < ntl) {
      const int it = it0 + t, s = it % S, n = it / S;
      if (n > 0) wait_or_abort(c.empty_a + 8 * s, (uint32_t)(n - 1) & 1u, ms, status);
      load_tile(stage_addr(c, s), t, src);
      cp_async_arrive_noinc(c.full_a + 8 * s);
    }
    const int tp = t - (S - 1);
    if (tid == 0 && tp >= 0) {
      const int it = it0 + tp, s = it % S, n = it / S;
      wait_or_abort(c.full_a + 8 * s, (uint32_t)n & 1u, ms, status);
      fence_proxy_async();
      if (!aborted(ms)) {
        tc_fence_after();
        const uint32_t st = stage_addr(c, s);
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_bf16(c.tmem + 32 * tp, smem_desc_sw128(st + h * HALF_BYTES + kk * 32, 16, 1024),
                     smem_desc(c.sq_a + (4 * h + kk) * 256, 128, QGRP), kIdescScore, (h | kk) != 0);
      }
      mma_commit(c.empty_a + 8 * s);
    }
  }
  if (tid == 0) mma_commit(c.done_a);
}

// Thread 0 waits (bounded) for phase `parity` of mbarrier `bar`; uniform.
__device__ __forceinline__ void wait_all(uint32_t bar, uint32_t parity, Misc& ms, int* status) {
  if (threadIdx.x == 0) wait_or_abort(bar, parity, ms, status);
  __syncthreads();
  tc_fence_after();
}

// Per-query max (x sl2, log2 units) of the valid rows of TMEM tiles
// 0..ntl-1 -> ms.mloc.
__device__ __forceinline__ void pass_max(const Ctx& c, Misc& ms, int ntl, int mc) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, qd = warp & 3, half = warp >> 2;
  const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
  float mx[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) mx[i] = -INFINITY;
  for (int t = half; t < ntl; t += 2) {
    uint32_t ra[32];
    tmem_ld32_issue(c.tmem + lane_base + 32 * t, ra);
    tmem_wait_ld();
    if (t * TM + qd * 32 + lane < mc) {
#pragma unroll
      for (int i = 0; i < 32; ++i) mx[i] = fmaxf(mx[i], __uint_as_float(ra[i]));
    }
  }
  ms.red[warp][lane] = transpose_reduce32<true>(mx, lane);
  __syncthreads();
  if (tid < 32) {
    float m = -INFINITY;
#pragma unroll
    for (int w = 0; w < 8; ++w) m = fmaxf(m, ms.red[w][tid]);
    ms.mloc[tid] = m * c.sl2;
  }
  __syncthreads();
}

// Per-query sum of 2^(l - mloc) over the valid rows; (mloc, sum) of this CTA
// are written into slot `rank` of every cluster CTA's xstat.
__device__ __forceinline__ void pass_sum(const Ctx& c, Misc& ms, int ntl, int mc) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, qd = warp & 3, half = warp >> 2;
  const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
  float ml[32], acc[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    ml[i] = ms.mloc[i];
    acc[i] = 0.f;
  }
  for (int t = half; t < ntl; t += 2) {
    uint32_t ra[32];
    tmem_ld32_issue(c.tmem + lane_base + 32 * t, ra);
    tmem_wait_ld();
    if (t * TM + qd * 32 + lane < mc) {
#pragma unroll
      for (int i = 0; i < 32; ++i) acc[i] += ex2(fmaf(__uint_as_float(ra[i]), c.sl2, -ml[i]));
    }
  }
  ms.red[warp][lane] = transpose_reduce32<false>(acc, lane);
  __syncthreads();
  if (tid < 32) {
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) sum += ms.red[w][tid];
    const uint32_t local = smem_u32(&ms.xstat[c.rank][tid]);
    for (uint32_t r = 0; r < c.cs; ++r) st_cluster_v2f32(map_rank(local, r), ms.mloc[tid], sum);
  }
}

// Ranking key log2 W_j of each valid row (Eq. 8 as a log-sum-exp over the
// query rows, against the normaliser c_i in ms.cvec), written to position
// g0 + j of every cluster CTA's key array.
__device__ __forceinline__ void pass_keys(const Ctx& c, Misc& ms, int ntl, int mc, int g0) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, qd = warp & 3, half = warp >> 2;
  const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
  float cv[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) cv[i] = ms.cvec[i];
  const int q = c.q;
  for (int t = half; t < ntl; t += 2) {
    uint32_t ra[32];
    tmem_ld32_issue(c.tmem + lane_base + 32 * t, ra);
    tmem_wait_ld();
    const int j = t * TM + qd * 32 + lane;
    float v[32];
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      v[i] = fmaf(__uint_as_float(ra[i]), c.sl2, -cv[i]);
      if (i < q) mx = fmaxf(mx, v[i]);
    }
    float z = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (i < q) z += ex2(v[i] - mx);
    const float key = mx + lg2(z);
    if (j < mc) {
      const uint32_t local = c.keys_a + 4u * (uint32_t)(g0 + j);
      for (uint32_t r = 0; r < c.cs; ++r) st_cluster_f32(map_rank(local, r), key);
    }
  }
}

// Attention phase 2: every thread streams the V rows; warps 4-7 write
// P = 2^(s - m) (bf16, P^T MN-major) and accumulate its row sums into
// ms.lacc; thread 0 accumulates O^T += V_s^T P^T in TMEM column ocol.
__device__ __forceinline__ void attn_pv(const Ctx& c, Misc& ms, int* status, int it_v, int ntl, RowSrc src,
                                     uint32_t ocol, uint8_t* pbase) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, qd = warp & 3;
  const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
  const int S = c.stages;
  float ml[32], lsum[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    ml[i] = ms.mloc[i];
    lsum[i] = 0.f;
  }
  for (int t = 0; t < ntl + S - 1; ++t) {
    if (t < ntl) {
      const int itv = it_v + t, s = itv % S, n = itv / S;
      if (n > 0) wait_or_abort(c.empty_a + 8 * s, (uint32_t)(n - 1) & 1u, ms, status);
      load_tile(stage_addr(c, s), t, src);
      cp_async_arrive_noinc(c.full_a + 8 * s);
    }
    const int tp = t - (S - 1);
    if (tp < 0) continue;
    const int pb = tp & 1, pn = tp >> 1;
    if (warp >= 4) {
      if (tp >= 2) {
        if (lane == 0) wait_or_abort(c.pempty_a + 8 * pb, (uint32_t)(pn - 1) & 1u, ms, status);
        __syncwarp();
      }
      uint32_t ra[32];
      tmem_ld32_issue(c.tmem + lane_base + 32 * tp, ra);
      tmem_wait_ld();
      const int r = qd * 32 + lane;
      const bool ok = tp * TM + r < src.mc;
      uint32_t w[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        const float p0 = ok ? ex2(fmaf(__uint_as_float(ra[i]), c.sl2, -ml[i])) : 0.f;
        const float p1 = ok ? ex2(fmaf(__uint_as_float(ra[i + 1]), c.sl2, -ml[i + 1])) : 0.f;
        const __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
        lsum[i] += __low2float(h2);
        lsum[i + 1] += __high2float(h2);
        w[i / 2] = *reinterpret_cast<const uint32_t*>(&h2);
      }
      // P^T, MN-major core matrices: key group r / 8, query chunk c.
      uint8_t* dst = pbase + pb * P_BYTES + (r >> 3) * 512 + (r & 7) * 16;
#pragma unroll
      for (int ch = 0; ch < 4; ++ch)
        *reinterpret_cast<uint4*>(dst + ch * 128) =
            make_uint4(w[4 * ch], w[4 * ch + 1], w[4 * ch + 2], w[4 * ch + 3]);
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive(c.pfull_a + 8 * pb);
    }
    if (tid == 0) {
      const int itv = it_v + tp, s = itv % S, n = itv / S;
      wait_or_abort(c.full_a + 8 * s, (uint32_t)n & 1u, ms, status);
      wait_or_abort(c.pfull_a + 8 * pb, (uint32_t)pn & 1u, ms, status);
      fence_proxy_async();
      if (!aborted(ms)) {
        tc_fence_after();
        const uint32_t st = stage_addr(c, s);
#pragma unroll
        for (int kq = 0; kq < TM / 16; ++kq)
          mma_bf16(c.tmem + ocol, smem_desc_sw128(st + kq * 2048, HALF_BYTES, 1024),
                   smem_desc(c.p_a + pb * P_BYTES + kq * 1024, 512, 128), kIdescPV, (tp > 0 || kq > 0) ? 1u : 0u);
      }
      mma_commit(c.empty_a + 8 * s);
      mma_commit(c.pempty_a + 8 * pb);
    }
  }
  if (tid == 0) mma_commit(c.done_a);
  if (warp >= 4) ms.red[warp][lane] = transpose_reduce32<false>(lsum, lane);
  __syncthreads();
  if (tid < 32) {
    float sum = 0.f;
#pragma unroll
    for (int w = 4; w < 8; ++w) sum += ms.red[w][tid];
    ms.lacc[tid] = sum;
  }
}

// Partial O^T of this CTA -> CTA 0, which combines the cluster's partials and
// writes O (bf16).
__device__ __forceinline__ void attn_combine(const Ctx& c, Misc& ms, const FusedParams& p, int64_t bb, int64_t hh,
                                          uint32_t ocol, const float* part_base) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, qd = warp & 3;
  const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
  uint32_t orow[32];
  if (warp >= 4) {
    tmem_ld32_issue(c.tmem + lane_base + ocol, orow);
    tmem_wait_ld();
  }
  tc_fence_before();
  cluster_sync();
  const uint32_t recv = c.stage_a;
  if (warp >= 4) {
    const int d = qd * 32 + lane;
    const uint32_t dst = map_rank(recv + 4u * (uint32_t)((c.rank * D + d) * NQ), 0);
#pragma unroll
    for (int i = 0; i < 32; i += 4)
      st_cluster_v4f32(dst + 4u * i, __uint_as_float(orow[i]), __uint_as_float(orow[i + 1]),
                       __uint_as_float(orow[i + 2]), __uint_as_float(orow[i + 3]));
  }
  if (tid < 32) {
    const uint32_t ml_a = recv + 4u * (uint32_t)(c.cs * NQ * D) + 8u * (c.rank * NQ + tid);
    st_cluster_v2f32(map_rank(ml_a, 0), ms.mloc[tid], ms.lacc[tid]);
  }
  cluster_sync();
  if (c.rank == 0) {
    const float2* mlp = reinterpret_cast<const float2*>(part_base + c.cs * NQ * D);
    bf16* ob = p.O + bb * p.osb + hh * p.osh;
    for (int e = tid; e < NQ * D; e += NT) {
      const int qi = e % NQ, d = e / NQ;
      if (qi >= c.q) continue;
      float M = -INFINITY;
      for (uint32_t r = 0; r < c.cs; ++r)
        if (mlp[r * NQ + qi].y > 0.f) M = fmaxf(M, mlp[r * NQ + qi].x);
      float num = 0.f, den = 0.f;
      for (uint32_t r = 0; r < c.cs; ++r) {
        const float2 x = mlp[r * NQ + qi];
        if (!(x.y > 0.f)) continue;  // a CTA with no keys sent no partial output
        const float f = ex2(x.x - M);
        num = fmaf(part_base[(r * D + d) * NQ + qi], f, num);
        den = fmaf(x.y, f, den);
      }
      ob[(int64_t)qi * p.oss + d] = __float2bfloat16_rn(num / den);
    }
  }
}

template <int STAGES>
__global__ void __launch_bounds__(NT, 1) wf_fused_kernel(const __grid_constant__ FusedParams p) {
  using LY = Layout<STAGES>;
  extern __shared__ __align__(1024) uint8_t smem[];
  Misc& ms = *reinterpret_cast<Misc*>(smem + LY::off_misc);
  uint32_t* hist = reinterpret_cast<uint32_t*>(smem + LY::off_hist);
  float* keys = reinterpret_cast<float*>(smem + LY::off_keys);
  int32_t* const J0 = reinterpret_cast<int32_t*>(smem + LY::off_keys + 4 * p.cmax);
  int32_t* const J1 = J0 + p.kmax;

  Ctx c;
  c.sq_a = smem_u32(smem + LY::off_q);
  c.p_a = smem_u32(smem + LY::off_p);
  c.keys_a = smem_u32(keys);
  c.done_a = smem_u32(&ms.done);
  c.stage_a = smem_u32(smem + LY::off_stage);
  c.full_a = smem_u32(&ms.full[0]);
  c.empty_a = smem_u32(&ms.empty[0]);
  c.pfull_a = smem_u32(&ms.pfull[0]);
  c.pempty_a = smem_u32(&ms.pempty[0]);
  c.rank = cluster_rank();
  c.cs = cluster_size();
  c.stages = STAGES;
  c.q = p.q;
  c.sl2 = p.scale_log2;
  const int u = (int)cluster_id_x();
  const int64_t bb = u / p.H, hh = u % p.H;
  const int tid = threadIdx.x, warp = tid >> 5;

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(c.full_a + 8 * s, NT);
      mbar_init(c.empty_a + 8 * s, 1);
    }
    mbar_init(c.done_a, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(c.pfull_a + 8 * i, 4);
      mbar_init(c.pempty_a + 8 * i, 1);
    }
    ms.abort = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(&ms.tmem_base), p.tmem_cols);
    tmem_relinquish();
  }
  // Query block -> shared memory, K-major core matrices, rows >= q zero.
  {
    const bf16* qb = p.Q + bb * p.qsb + hh * p.qsh;
    uint8_t* sq = smem + LY::off_q;
    for (int e = tid; e < NQ * (D / 8); e += NT) {
      const int rr = e & 7, ch = (e >> 3) & (D / 8 - 1), g = e >> 7;
      const int i = g * 8 + rr;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (i < p.q) v = __ldg(reinterpret_cast<const uint4*>(qb + (int64_t)i * p.qss + ch * 8));
      *reinterpret_cast<uint4*>(sq + g * QGRP + ch * 128 + rr * 16) = v;
    }
  }
  fence_proxy_async();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  c.tmem = ms.tmem_base;
  cluster_sync();

  const int L = p.L;
  int m_total = p.n >> L;
  bool top = true;
  bool jsel = false;  // false: the current level writes J0
  const int32_t* Jprev = J1;
  int64_t sets_off = 0;
  int it = 0;             // pipeline iteration counter (uniform)
  uint32_t done_cnt = 0;  // completions of `done` so far (uniform)
  const int lev_end = p.trim ? 0 : 1;
  const int64_t krow_off = bb * p.ksb + hh * p.ksh;

  for (int lev = L; lev >= lev_end; --lev) {
    // This CTA's slice of the candidate positions (pairs kept together).
    const int pairs = (m_total + 1) >> 1;
    const int g0 = min(m_total, 2 * (int)((int64_t)c.rank * pairs / c.cs));
    const int g1 = min(m_total, 2 * (int)((int64_t)(c.rank + 1) * pairs / c.cs));
    const int mc = g1 - g0;
    const int ntl = (mc + TM - 1) / TM;
    RowSrc src;
    src.base = lev >= 1 ? p.coeffs + ((int64_t)u * p.rows_total + ((int64_t)p.n - ((int64_t)p.n >> (lev - 1)))) * D
                        : p.K + krow_off;
    src.stride = lev >= 1 ? D : p.kss;
    src.gbase = nullptr;
    src.gstride = 0;
    src.J = Jprev;
    src.kind = top ? 0 : 1;
    src.trim = 0;
    src.g0 = g0;
    src.mc = mc;
    src.kk = 0;
    stream_scores(c, ms, p.status, it, ntl, src);
    wait_all(c.done_a, done_cnt & 1u, ms, p.status);
    ++done_cnt;
    it += ntl;

    pass_max(c, ms, ntl, mc);
    pass_sum(c, ms, ntl, mc);
    cluster_sync();
    // Softmax normaliser per query: c = M + log2 S over the whole candidate set.
    if (tid < 32) {
      float M = -INFINITY;
      for (uint32_t r = 0; r < c.cs; ++r)
        if (ms.xstat[r][tid].y > 0.f) M = fmaxf(M, ms.xstat[r][tid].x);
      float S = 0.f;
      for (uint32_t r = 0; r < c.cs; ++r) {
        const float2 x = ms.xstat[r][tid];
        if (x.y > 0.f) S += x.y * ex2(x.x - M);
      }
      ms.cvec[tid] = M + lg2(S);
    }
    __syncthreads();
    pass_keys(c, ms, ntl, mc, g0);
    tc_fence_before();
    cluster_sync();
    tc_fence_after();

    // Eq. 9: Top-K (same result in every CTA of the cluster).
    const int kb = p.keep[lev];
    int32_t* Jcur = jsel ? J1 : J0;
    select_topk(keys, m_total, kb, Jcur, top, Jprev, ms, hist);
    if (lev >= 1) {
      if (c.rank == 0 && p.level_sets) {
        int32_t* out = p.level_sets + (int64_t)u * p.sets_stride + sets_off;
        for (int i = tid; i < kb; i += NT) out[i] = Jcur[i];
      }
      sets_off += kb;
    }
    Jprev = Jcur;
    jsel = !jsel;
    m_total = 2 * kb;  // Eq. 10: children of the kept coefficients
    top = false;
  }

  // mu^0 and the sparse key list [K[mu^0]; Kg].
  const int kk = p.keep[0];
  const int32_t* Jfin = Jprev;
  const bool trim = p.trim != 0;
  if (c.rank == 0) {
    int32_t* out = p.idx + (int64_t)u * kk;
    int32_t* ls = p.level_sets ? p.level_sets + (int64_t)u * p.sets_stride + sets_off : nullptr;
    for (int t = tid; t < kk; t += NT) {
      const int tok = trim ? Jfin[t] : 2 * Jfin[t >> 1] + (t & 1);
      out[t] = tok;
      if (ls) ls[t] = tok;
    }
  }
  const int total = kk + p.ng;
  const int a0 = (int)((int64_t)c.rank * total / c.cs);
  const int a1 = (int)((int64_t)(c.rank + 1) * total / c.cs);
  const int mc = a1 - a0;
  const int ntl = (mc + TM - 1) / TM;
  const uint32_t ocol = p.tmem_cols - 32;
  RowSrc src;
  src.base = p.K + krow_off;
  src.stride = p.kss;
  src.gbase = p.Kg + (bb * p.gsb + hh * p.gsh);
  src.gstride = p.gss;
  src.J = Jfin;
  src.kind = 2;
  src.trim = trim ? 1 : 0;
  src.g0 = a0;
  src.mc = mc;
  src.kk = kk;

  // Attention phase 1: S^T = K_s Q^T and the per-query max (log2 units).
  stream_scores(c, ms, p.status, it, ntl, src);
  wait_all(c.done_a, done_cnt & 1u, ms, p.status);
  ++done_cnt;
  pass_max(c, ms, ntl, mc);

  // Attention phase 2: O^T = V_s^T P^T.
  src.base = p.V + krow_off;
  src.gbase = p.Vg + (bb * p.gsb + hh * p.gsh);
  attn_pv(c, ms, p.status, it + ntl, ntl, src, ocol, smem + LY::off_p);
  wait_all(c.done_a, done_cnt & 1u, ms, p.status);
  ++done_cnt;
  attn_combine(c, ms, p, bb, hh, ocol, reinterpret_cast<const float*>(smem + LY::off_stage));
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(c.tmem, p.tmem_cols);
}

}  // namespace

// ---------------------------------------------------------------------------
// Host side.
// ---------------------------------------------------------------------------
FusedPlan plan_fused(const wf_tensor& q, const wf_tensor& kv, int levels, const int32_t* keep, int n_g,
                     const wf_tensor* g, int num_sms) {
  (void)g;
  FusedPlan fp{};
  fp.ok = false;
  if (kv.dtype != WF_BF16 || kv.head_dim != D || q.seq > NQ || levels > 10) return fp;
  const int U = kv.batch * kv.heads;
  const int n = kv.seq;
  const bool trim = keep[0] < 2 * keep[1];
  int cmax = n >> levels, kmax = 0;
  for (int l = 0; l <= levels; ++l) kmax = kmax > keep[l] ? kmax : keep[l];
  for (int l = 1; l <= levels; ++l) cmax = cmax > 2 * keep[l] ? cmax : 2 * keep[l];
  if (cmax > 8192 || kmax > 8192) return fp;
  const int total = keep[0] + n_g;
  auto tiles_ok = [&](int cs, int* cols) {
    auto slice_tiles = [&](int m) { return (2 * (((m + 1) / 2 + cs - 1) / cs) + TM - 1) / TM; };
    int tmax = slice_tiles(n >> levels);
    for (int l = levels; l >= 1; --l) {
      const int t = slice_tiles(2 * keep[l]);
      tmax = tmax > t ? tmax : t;
    }
    const int ta = ((total + cs - 1) / cs + TM - 1) / TM + 1;
    tmax = tmax > ta ? tmax : ta;
    int c = 32;
    while (c < 32 * tmax) c *= 2;
    *cols = c;
    return 32 * tmax <= 512;
  };
  int cs = 1, cols = 0;
  while (cs < 4 && (!tiles_ok(cs, &cols) || U * cs * 2 <= num_sms)) cs *= 2;
  if (!tiles_ok(cs, &cols)) return fp;
  const size_t kMaxSmem = 227 * 1024;
  const size_t tail = 4 * (size_t)cmax + 8 * (size_t)kmax;
  int stages = 4;
  if (Layout<4>::off_keys + tail > kMaxSmem) stages = 3;
  const size_t smem = (stages == 4 ? Layout<4>::off_keys : Layout<3>::off_keys) + tail;
  if (smem > kMaxSmem) return fp;
  // CTA 0 receives every partial output in its stage area.
  if ((size_t)cs * (NQ * D * 4 + NQ * 8) > (size_t)stages * TILE_BYTES) return fp;
  fp.ok = true;
  fp.cs = cs;
  fp.stages = stages;
  fp.smem = smem;
  fp.tmem_cols = cols;
  fp.cmax = cmax;
  fp.kmax = kmax;
  fp.trim = trim;
  fp.U = U;
  return fp;
}

cudaError_t launch_fused(const FusedPlan& fp, const void* Q, const wf_tensor& qd, const void* K, const void* V,
                         const wf_tensor& kv, const void* Kg, const void* Vg, const wf_tensor* g,
                         const void* coeffs, int levels, const int32_t* keep, int32_t* idx, int32_t* level_sets,
                         void* O, const wf_tensor& od, int* status, cudaStream_t s) {
  FusedParams p;
  memset(&p, 0, sizeof(p));
  p.Q = static_cast<const bf16*>(Q);
  p.qsb = qd.stride_b; p.qsh = qd.stride_h; p.qss = qd.stride_s;
  p.K = static_cast<const bf16*>(K);
  p.V = static_cast<const bf16*>(V);
  p.ksb = kv.stride_b; p.ksh = kv.stride_h; p.kss = kv.stride_s;
  p.Kg = static_cast<const bf16*>(Kg);
  p.Vg = static_cast<const bf16*>(Vg);
  if (g) { p.gsb = g->stride_b; p.gsh = g->stride_h; p.gss = g->stride_s; }
  p.coeffs = static_cast<const bf16*>(coeffs);
  p.rows_total = (int64_t)kv.seq - ((int64_t)kv.seq >> levels);
  p.O = static_cast<bf16*>(O);
  p.osb = od.stride_b; p.osh = od.stride_h; p.oss = od.stride_s;
  p.idx = idx;
  p.level_sets = level_sets;
  int64_t stride = 0;
  for (int l = 0; l <= levels; ++l) stride += keep[l];
  p.sets_stride = stride;
  p.status = status;
  p.q = qd.seq; p.n = kv.seq; p.ng = g ? g->seq : 0; p.H = kv.heads; p.L = levels; p.trim = fp.trim ? 1 : 0;
  p.cmax = fp.cmax; p.kmax = fp.kmax;
  p.tmem_cols = (uint32_t)fp.tmem_cols;
  for (int l = 0; l <= levels; ++l) p.keep[l] = keep[l];
  p.scale_log2 = kLog2e / sqrtf((float)D);

  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(fp.U * fp.cs), 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = fp.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = fp.cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e;
  if (fp.stages == 4) {
    e = cudaFuncSetAttribute(wf_fused_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)cfg.dynamicSmemBytes);
    if (e != cudaSuccess) return e;
    e = cudaLaunchKernelEx(&cfg, wf_fused_kernel<4>, p);
  } else {
    e = cudaFuncSetAttribute(wf_fused_kernel<3>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)cfg.dynamicSmemBytes);
    if (e != cudaSuccess) return e;
    e = cudaLaunchKernelEx(&cfg, wf_fused_kernel<3>, p);
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace wf
