// Tensor-core skim for the per-stage filter (bf16 keys, head_dim 128): the
// scores of one scale (Eq. 7 logits) as tcgen05 MMAs of 128 gathered
// candidate rows against the unit's whole query block (up to 256 rows: the
// grouped heads of a key head), in two passes over the same tiles.
//   stats: per (tile, query row) the max and the sum of 2^(s - max) of the
//          tile's logits (log2 units) -> part[unit][tile][row];
//   keys:  the query rows' normalisers c_i = M_i + log2 S_i (folded from all
//          tiles' partials by a small kernel in between), then each
//          candidate's ranking key log2 W_j = log2 sum_i 2^(s_ij - c_i)
//          (Eq. 8 as a log-sum-exp) -> W[unit][j].
// The keys pass recomputes the MMA instead of storing the logits: a tile's
// rows are read twice (the second time mostly from L2) and no logit matrix
// goes through memory.
//
// One CTA of two warpgroups per (tile, unit).  All threads gather the tile
// (16-byte cp.async into the 128-byte-swizzled K-major layout) and the query
// block (cp.async into K-major core matrices, zero rows up to a multiple of
// 32); one thread issues the eight MMAs (K = 128) into TMEM and commits them
// to an mbarrier.  Each warpgroup covers the 128 TMEM lanes (a warp per lane
// quarter, a thread per candidate) and reads back every other 32-column
// chunk of the query columns.  The wait on the MMAs is bounded (~1 s): on a
// timeout the CTA sets the status word, waits once more with the same
// bound, frees its TMEM and leaves.
#include <math.h>

#include "wf_internal.cuh"
#include "wf_sm100.cuh"

namespace wf {
namespace {

using namespace sm100;

constexpr int D = 128;
constexpr int TM = 128;                // candidate rows per tile (MMA M)
constexpr int NTH = 256;               // threads per CTA: two warpgroups
constexpr int NWG = NTH / 128;         // warpgroups; each covers all 128 TMEM lanes
constexpr int HALF = TM * 128;         // one 64-column half of the tile
constexpr int QGRP = (D / 8) * 128;    // bytes per 8-row group of the query block
constexpr long long kWait = 1ll << 31;

// floor(i / qs) for 0 <= i, qs <= 256 from the reciprocal: (i + 1/2) / qs
// lies at least 1/(2 qs) from an integer, far beyond the rounding of the
// product, so truncation is exact.
__device__ __forceinline__ int head_of(int i, float rqs) { return __float2int_rz(((float)i + 0.5f) * rqs); }

struct TcArgs {
  const bf16* Q;
  int64_t qsb, qsh, qss;
  int q, G, qs, H;              // query rows per unit (G heads of qs rows), key heads
  float rqs;                    // 1 / qs (head of a query row without a division)
  RowSrc src;                   // candidate rows (row index = cand[j] or j)
  const int32_t* cand;
  int64_t cand_stride;
  int m;                        // candidates of the scale
  int nq;                       // query columns of the MMA (q rounded up to 32)
  uint32_t tcols;               // TMEM columns allocated
  float2* part;                 // [unit][tile][q]
  int64_t part_unit;
  float* W;                     // [unit][w_unit]
  int64_t w_unit;
  float* cvec;                  // [unit][q] normalisers c_i (folded between the passes)
  int* status;
  float sl2;                    // log2(e) / sqrt(d)
};

// c_i = M_i + log2 S_i of every query row from all tiles' partials.
__global__ void __launch_bounds__(256) norm_kernel(const float2* __restrict__ part, int64_t part_unit, int ntiles,
                                                   int q, float* __restrict__ cvec) {
  const int u = blockIdx.y;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= q) return;
  const float2* pu = part + (int64_t)u * part_unit + i;
  float M = -INFINITY;
  for (int tt = 0; tt < ntiles; ++tt) M = fmaxf(M, pu[(int64_t)tt * q].x);
  float S = 0.f;
  for (int tt = 0; tt < ntiles; ++tt) {
    const float2 p = pu[(int64_t)tt * q];
    S += p.y * ex2(p.x - M);
  }
  cvec[(int64_t)u * q + i] = M + lg2(S);
}

// Barrier of one warpgroup (named barriers 1, 2).
__device__ __forceinline__ void wg_sync(int wg) { asm volatile("bar.sync %0, 128;" ::"r"(1 + wg) : "memory"); }

// Lane l of the warp ends with the reduction of column l over the warp's 32
// lanes (31 shuffles).
template <bool MAX>
__device__ __forceinline__ float xpose_reduce32(float (&v)[32], int lane) {
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

template <int MODE>
__global__ void __launch_bounds__(NTH) tc_score_kernel(const __grid_constant__ TcArgs a) {
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* tile = smem;                        // 2 x HALF, 1024-aligned
  uint8_t* sq = smem + 2 * HALF;               // nq / 8 groups of QGRP
  // [NWG][4 lane quarters][4 chunks][32] (max, sum) of each warp's rows per column (MODE 0)
  float* red = reinterpret_cast<float*>(sq + (a.nq / 8) * QGRP);
  float* col = red + NWG * 4 * 4 * 32 * 2;     // [256]: the c_i (MODE 1)
  float2* xch = reinterpret_cast<float2*>(col + 256);  // [128]: the second warpgroup's (max, sum) per row
  unsigned long long* bar = reinterpret_cast<unsigned long long*>(xch + 128);
  uint32_t* tbase = reinterpret_cast<uint32_t*>(bar + 1);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int wg = tid >> 7, wt = tid & 127, quarter = warp & 3;
  const int t = blockIdx.x, u = blockIdx.y;
  const int64_t bb = u / a.H, hh = u % a.H;

  if (warp == 0) {
    tmem_alloc(smem_u32(tbase), a.tcols);
    tmem_relinquish();
  }
  if (tid == 0) {
    mbar_init(smem_u32(bar), 1);
    fence_mbar_init();
  }
  // The tile: chunk c = tid % 16 of rows r0 + 16 i (r0 = tid / 16),
  // 128-byte swizzle.  The 16 lanes of a half-warp copy the same 8 rows: lane
  // c loads the index of row r0 + 16 (c % 8) and the half-warp shares them
  // by shuffles; the swizzle term of a thread's rows is constant.
  {
    constexpr int RPT = TM / (NTH / 16);  // rows a thread copies
    static_assert(RPT == 8 && (NTH / 16) % 8 == 0, "rows of a thread share r % 8");
    const int c = tid & 15, r0 = tid >> 4, half = tid & 16;
    const char* rb = reinterpret_cast<const char*>(static_cast<const bf16*>(a.src.base) + bb * a.src.sb +
                                                   hh * a.src.sh + a.src.off) + c * 16;
    const int32_t* cd = a.cand ? a.cand + (int64_t)u * a.cand_stride : nullptr;
    const int jl = min(t * TM + r0 + (NTH / 16) * (c & (RPT - 1)), a.m - 1);  // rows past the list repeat its last row
    const uint32_t rowl = cd ? (uint32_t)cd[jl] : (uint32_t)jl;
    const uint32_t sb = (uint32_t)a.src.ss * 2u;
    const uint32_t dbase = smem_u32(tile) + ((c >> 3) * HALF) + (uint32_t)r0 * 128u + (uint32_t)(((c ^ r0) & 7) << 4);
#pragma unroll
    for (int i = 0; i < RPT; ++i) {
      const uint32_t row = __shfl_sync(0xffffffffu, rowl, half | i);
      cp_async16(dbase + (uint32_t)(NTH / 16) * 128u * i, rb + (size_t)row * sb);
    }
  }
  // The query block, K-major core matrices; rows q .. nq - 1 zero.
  for (int e = tid; e < a.nq * (D / 8); e += NTH) {
    const int rr = e & 7, ch = (e >> 3) & (D / 8 - 1), g = e >> 7;
    const int i = g * 8 + rr;
    const uint32_t dst = smem_u32(sq + g * QGRP + ch * 128 + rr * 16);
    if (i < a.q) {
      const int hi = head_of(i, a.rqs);
      const bf16* qp = a.Q + bb * a.qsb + (hh * a.G + hi) * a.qsh + (int64_t)(i - hi * a.qs) * a.qss;
      cp_async16(dst, qp + ch * 8);
    } else {
      sts_v4(dst, make_uint4(0, 0, 0, 0));
    }
  }
  cp_async_wait_all();
  fence_proxy_async();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tbase;
  const uint32_t idesc = idesc_bf16(TM, a.nq, 0, 0);
  if (tid == 0) {
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        mma_bf16(tmem, smem_desc_sw128(smem_u32(tile) + h * HALF + kk * 32, 16, 1024),
                 smem_desc(smem_u32(sq) + (4 * h + kk) * 256, 128, QGRP), idesc, (h | kk) != 0);
    mma_commit(smem_u32(bar));
  }
  __syncwarp();
  bool ok = mbar_wait_bounded(smem_u32(bar), 0u, kWait);
  if (!ok) {
    atomicExch(a.status, 1);
    (void)mbar_wait_bounded(smem_u32(bar), 0u, kWait);
  }
  ok = __syncthreads_and(ok);
  tc_fence_after();

  // Thread wt of either warpgroup owns candidate j (TMEM lane wt); the two
  // warpgroups take alternate 32-column chunks.
  const int j = t * TM + wt;
  const bool valid = j < a.m;
  const uint32_t lane_base = tmem + ((uint32_t)(quarter * 32) << 16);
  const int nch = a.nq / 32;
  if (ok && MODE == 0) {
    // Each warp takes its own column maxima (the warp-wide max instruction)
    // and sums its rows against them, with no barrier per chunk; the four
    // lane quarters' (max, sum) of a column then merge into the tile's.
    float2* pt = a.part + (int64_t)u * a.part_unit + (int64_t)t * a.q;
    float2* sl = reinterpret_cast<float2*>(red);
    int k = 0;
#pragma unroll 1
    for (int ch = wg; ch < nch; ch += NWG, ++k) {
      float v[32], w[32];
      tmem_ld32(lane_base + 32 * ch, v);
      float mcol = -INFINITY;  // lane i: this warp's max of column i (x sl2)
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float mi = warp_max_f32(valid ? v[i] : -INFINITY) * a.sl2;
        mcol = lane == i ? mi : mcol;
        w[i] = valid ? ex2(fmaf(v[i], a.sl2, -mi)) : 0.f;
      }
      const float sum = xpose_reduce32<false>(w, lane);
      sl[((wg * 4 + quarter) * 4 + k) * 32 + lane] = make_float2(mcol, sum);
    }
    wg_sync(wg);
    k = 0;
#pragma unroll 1
    for (int ch = wg; ch < nch; ch += NWG, ++k) {
      if (wt < 32 && ch * 32 + wt < a.q) {
        float2 r[4];
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) r[q4] = sl[((wg * 4 + q4) * 4 + k) * 32 + wt];
        float M = -INFINITY;
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4)
          if (r[q4].y > 0.f) M = fmaxf(M, r[q4].x);
        float S = 0.f;
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4)
          if (r[q4].y > 0.f) S = fmaf(r[q4].y, ex2(r[q4].x - M), S);
        pt[ch * 32 + wt] = make_float2(M, S);
      }
    }
  }
  if (ok && MODE == 1) {
    // The normalisers (columns past q never count).
    for (int i = tid; i < a.nq; i += NTH) col[i] = i < a.q ? a.cvec[(int64_t)u * a.q + i] : INFINITY;
    __syncthreads();
    // Every exponent l sl2 - c_i is at most 0 (c_i is the log of a sum that
    // contains this candidate's own term), so the sum is taken unshifted; the
    // padded columns have c_i = +inf and add 0.  A warp with a valid row whose
    // sum is tiny (below 2^-96, where flushed terms could matter) takes that
    // row again shifted by its largest exponent (TMEM loads are warp-wide, so
    // the whole warp runs the pass).
    float mx = 0.f, z = 0.f;
#pragma unroll 1
    for (int ch = wg; ch < nch; ch += NWG) {
      float v[32];
      tmem_ld32(lane_base + 32 * ch, v);
#pragma unroll
      for (int i = 0; i < 32; ++i) z += ex2(fmaf(v[i], a.sl2, -col[ch * 32 + i]));
    }
    const bool tiny = valid && z < 0x1p-96f;
    if (__any_sync(0xffffffffu, tiny)) {
      float m2 = -INFINITY;
#pragma unroll 1
      for (int ch = wg; ch < nch; ch += NWG) {
        float v[32];
        tmem_ld32(lane_base + 32 * ch, v);
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (ch * 32 + i < a.q) m2 = fmaxf(m2, fmaf(v[i], a.sl2, -col[ch * 32 + i]));
      }
      float z2 = 0.f;
#pragma unroll 1
      for (int ch = wg; ch < nch; ch += NWG) {
        float v[32];
        tmem_ld32(lane_base + 32 * ch, v);
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (ch * 32 + i < a.q) z2 += ex2(fmaf(v[i], a.sl2, -col[ch * 32 + i]) - m2);
      }
      if (tiny) {
        mx = m2;
        z = z2;
      }
    }
    // Fold the second warpgroup's (max, sum) of the row into the first's.
    if (wg == 1) xch[wt] = make_float2(mx, z);
    __syncthreads();
    if (wg == 0) {
      const float2 o = xch[wt];
      const float M = fmaxf(mx, o.x);
      const float Z = (z > 0.f ? z * ex2(mx - M) : 0.f) + (o.y > 0.f ? o.y * ex2(o.x - M) : 0.f);
      if (valid) a.W[(int64_t)u * a.w_unit + j] = M + lg2(Z);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, a.tcols);
  }
}

}  // namespace

bool tc_skim_supported(const FilterPlan& p) { return p.dtype == WF_BF16 && p.d == D && p.q <= 256; }

cudaError_t launch_tc_skim(const FilterPlan& p, const void* Q, const wf_tensor& qd, RowSrc src, const int32_t* cand,
                           int m, float2* part, float* W, float* cvec, int* status, cudaStream_t s) {
  TcArgs a;
  a.Q = static_cast<const bf16*>(Q);
  a.qsb = qd.stride_b; a.qsh = qd.stride_h; a.qss = qd.stride_s;
  a.q = p.q; a.G = p.G; a.qs = p.qs; a.H = p.H;
  a.rqs = 1.0f / (float)a.qs;
  a.src = src;
  a.cand = cand;
  a.cand_stride = p.cmax;
  a.m = m;
  a.nq = (p.q + 31) / 32 * 32;
  uint32_t cols = 32;
  while ((int)cols < a.nq) cols *= 2;
  a.tcols = cols;
  a.part = part;
  a.part_unit = (int64_t)p.tiles_max * p.q;
  a.W = W;
  a.w_unit = p.cmax;
  a.cvec = cvec;
  a.status = status;
  a.sl2 = 1.4426950408889634f / sqrtf((float)D);
  // Shared memory: the tile, the query block, the reductions, the barrier.
  // At most 512 / cols CTAs may share an SM (TMEM); the request is padded so
  // that shared memory enforces it.
  size_t smem = 2 * HALF + (size_t)(a.nq / 8) * QGRP + sizeof(float) * (NWG * 4 * 4 * 32 * 2 + 256) +
                sizeof(float2) * 128 + 16;
  const size_t per_sm = 228 * 1024;
  const size_t cap = 512 / cols;  // CTAs per SM the TMEM allows
  const size_t floor_smem = per_sm / (cap + 1) + 1;
  if (cap < (size_t)(2048 / NTH) && smem < floor_smem) smem = floor_smem;
  const dim3 grid((unsigned)((m + TM - 1) / TM), (unsigned)p.U);
  cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(tc_score_kernel<0>), smem);
  if (e == cudaSuccess)
    e = raise_smem_limit(reinterpret_cast<const void*>(tc_score_kernel<1>), smem);
  if (e != cudaSuccess) return e;
  tc_score_kernel<0><<<grid, NTH, smem, s>>>(a);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  norm_kernel<<<dim3((unsigned)((p.q + 255) / 256), (unsigned)p.U), 256, 0, s>>>(part, a.part_unit,
                                                                                (m + TM - 1) / TM, p.q, cvec);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  tc_score_kernel<1><<<grid, NTH, smem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace wf

// ---------------------------------------------------------------------------
// Tensor-core sparse attention (Algorithm 1, final step) for the per-stage
// path: one CTA per (key unit, split of 128 sparse keys).  The split's K and
// V rows ([K[idx]; Kg] and [V[idx]; Vg]) are gathered into two
// 128-byte-swizzled tiles, S^T = K Q^T goes to TMEM (keys on the lanes, the
// unit's query rows on the columns), every thread turns its key's row into
// P = 2^(s - m) with m the split's per-query max (bf16, stored as P^T in
// MN-major core matrices over the dead K tile), and O^T = V^T P^T goes to
// TMEM.  A key unit's query rows are cut into column blocks of at most 128
// (grid z), so S^T and O^T fit 256 TMEM columns and two CTAs share an SM.
// The partial (O, m, l) of every query row lands in the flash-decoding
// layout of the fp32 kernels, per query head, so the same combine kernel
// finishes it.
// ---------------------------------------------------------------------------
namespace wf {
namespace {

using namespace sm100;

struct TcAttnArgs {
  const bf16* Q;
  int64_t qsb, qsh, qss;
  const bf16* K;
  const bf16* V;
  int64_t ksb, ksh, kss;
  const bf16* Kg;
  const bf16* Vg;
  int64_t gsb, gsh, gss;
  const int32_t* idx;
  int n, k, ng, q, G, qs, H;  // q = G qs query rows per key unit; H key heads
  float rqs;                  // 1 / qs
  int cb;                     // query columns per CTA block (blockIdx.z = block)
  int nq;                     // MMA columns of a block (its query rows rounded up to 32)
  uint32_t tcols;
  int nsplit;
  int tps;                    // key tiles of 128 a split (a CTA), taken one after the other
  float* Opart;               // [query unit][nsplit][qstride][D]
  float2* ML;                 // [query unit][nsplit][qstride]
  int qstride;
  int* status;
  float sl2;
  long long wait_limit;  // bound of the waits that can give up (cycles)
  int stall;             // test-only: the wait on the score MMAs uses a barrier nothing completes
};

__global__ void __launch_bounds__(NTH) tc_attn_kernel(const __grid_constant__ TcAttnArgs a) {
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* kt = smem;                          // K tile, 2 x HALF
  uint8_t* vt = smem + 2 * HALF;               // V tile, 2 x HALF
  uint8_t* sq = smem + 4 * HALF;               // query block, nq / 8 groups of QGRP
  // P^T (16 key groups of nq * 16 bytes, nq <= 128) takes the K tile's place:
  // the K rows are dead once the S^T products have completed.
  uint8_t* pb = kt;
  float* red = reinterpret_cast<float*>(sq + (a.nq / 8) * QGRP);  // [NWG][4][32]
  float* cm = red + NWG * 4 * 32;              // [256] running max per query (log2 units)
  float* cl = cm + 256;                        // [256] running row sums of P
  float* ca = cl + 256;                        // [256] this tile's factor 2^(m_old - m_new)
  unsigned long long* bar = reinterpret_cast<unsigned long long*>(ca + 256);  // [3]: S done, PV done, stall
  uint32_t* tbase = reinterpret_cast<uint32_t*>(bar + 3);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int wg = tid >> 7, wt = tid & 127, quarter = warp & 3;
  const int sp = blockIdx.x, u = blockIdx.y;
  const int64_t bb = u / a.H, hh = u % a.H;
  const int total = a.k + a.ng;
  const int c0 = blockIdx.z * a.cb;           // first query row of this column block
  const int qb = min(a.cb, a.q - c0);         // its query rows

  if (warp == 0) {
    tmem_alloc(smem_u32(tbase), a.tcols);
    tmem_relinquish();
  }
  if (tid == 0) {
    mbar_init(smem_u32(&bar[0]), 1);
    mbar_init(smem_u32(&bar[1]), 1);
    mbar_init(smem_u32(&bar[2]), 1);
    fence_mbar_init();
  }
  for (int e = tid; e < 256; e += NTH) {
    cm[e] = -INFINITY;
    cl[e] = 0.f;
  }
  for (int e = tid; e < a.nq * (D / 8); e += NTH) {
    const int rr = e & 7, ch = (e >> 3) & (D / 8 - 1), g = e >> 7;
    const int i = g * 8 + rr;
    const uint32_t dst = smem_u32(sq + g * QGRP + ch * 128 + rr * 16);
    if (i < qb) {
      const int qi = c0 + i;
      const int hi = head_of(qi, a.rqs);
      const bf16* qp = a.Q + bb * a.qsb + (hh * a.G + hi) * a.qsh + (int64_t)(qi - hi * a.qs) * a.qss;
      cp_async16(dst, qp + ch * 8);
    } else {
      sts_v4(dst, make_uint4(0, 0, 0, 0));
    }
  }
  const uint32_t qoff = (uint32_t)(quarter * 32) << 16;
  const int nch = a.nq / 32;
  float* rw = red + wg * 4 * 32;
  uint32_t tmem = 0, ocol = 0;
  bool ok = true;
  // The split's tiles of 128 sparse keys, one after the other: S^T, P with a
  // running per-query max (a raised max rescales the partial O^T and the row
  // sums by 2^(m_old - m_new)), O^T += V^T P^T.
#pragma unroll 1
  for (int j = 0; j < a.tps && ok; ++j) {
    const int t0 = (sp * a.tps + j) * TM;
    if (t0 >= total) break;  // the last split may hold fewer tiles
    // K and V rows of the tile: chunk c = tid % 16 of rows r0 + 16 i
    // (r0 = tid / 16).  Lane c resolves the K and V rows of row r0 + 16 (c % 8)
    // (a sparse key or a generation row) and the half-warp shares the two row
    // addresses by shuffles; the swizzle term of a thread's rows is constant.
    {
      constexpr int RPT = TM / (NTH / 16);
      static_assert(RPT == 8 && (NTH / 16) % 8 == 0, "rows of a thread share r % 8");
      const int c = tid & 15, r0 = tid >> 4, half = tid & 16;
      const int32_t* ui = a.idx + (int64_t)u * a.k;
      const uint32_t xs = (uint32_t)r0 * 128u + (uint32_t)(((c ^ r0) & 7) << 4);
      const uint32_t koff = smem_u32(kt) + ((c >> 3) * HALF) + xs, voff = smem_u32(vt) + ((c >> 3) * HALF) + xs;
      const int tl = min(t0 + r0 + (NTH / 16) * (c & (RPT - 1)), total - 1);  // keys past the list repeat its last key (P = 0 there)
      const bf16 *kl, *vl;
      if (tl < a.k) {
        int row = ui[tl];
        row = row < 0 ? 0 : (row >= a.n ? a.n - 1 : row);
        const int64_t o = bb * a.ksb + hh * a.ksh + (int64_t)row * a.kss;
        kl = a.K + o;
        vl = a.V + o;
      } else {
        const int64_t o = bb * a.gsb + hh * a.gsh + (int64_t)(tl - a.k) * a.gss;
        kl = a.Kg + o;
        vl = a.Vg + o;
      }
      const unsigned long long ka = reinterpret_cast<unsigned long long>(kl),
                               va = reinterpret_cast<unsigned long long>(vl);
#pragma unroll
      for (int i = 0; i < RPT; ++i) {
        const unsigned long long kp = __shfl_sync(0xffffffffu, ka, half | i), vp = __shfl_sync(0xffffffffu, va, half | i);
        const uint32_t so = (uint32_t)(NTH / 16) * 128u * i;
        cp_async16(koff + so, reinterpret_cast<const bf16*>(kp) + c * 8);
        cp_async16(voff + so, reinterpret_cast<const bf16*>(vp) + c * 8);
      }
    }
    cp_async_wait_all();
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    tmem = *tbase;
    ocol = tmem + (uint32_t)a.nq;  // O^T columns after S^T
    const uint32_t ph = (uint32_t)j & 1u;
    if (tid == 0) {
      const uint32_t idesc = idesc_bf16(TM, a.nq, 0, 0);
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_bf16(tmem, smem_desc_sw128(smem_u32(kt) + h * HALF + kk * 32, 16, 1024),
                   smem_desc(smem_u32(sq) + (4 * h + kk) * 256, 128, QGRP), idesc, (h | kk) != 0);
      mma_commit(smem_u32(&bar[0]));
    }
    __syncwarp();
    bool sok = mbar_wait_bounded(smem_u32(&bar[(a.stall && j == 0) ? 2 : 0]), ph, a.wait_limit);
    if (!sok) {
      // Drain the score MMAs (default bound) before the TMEM is freed.
      atomicExch(a.status, 1);
      (void)mbar_wait_bounded(smem_u32(&bar[0]), ph, kWait);
    }
    ok = __syncthreads_and(sok);
    tc_fence_after();
    if (!ok) break;

    // Thread wt of either warpgroup owns key t0 + wt (TMEM lane wt); the two
    // warpgroups take alternate 32-column chunks.
    const bool valid = t0 + wt < total;
    uint8_t* prow = pb + (wt >> 3) * (a.nq * 16) + (wt & 7) * 16;
    bool raised = false;
#pragma unroll 1
    for (int ch = wg; ch < nch; ch += NWG) {
      float v[32], w[32];
      tmem_ld32(tmem + qoff + 32 * ch, v);
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        v[i] = valid ? v[i] * a.sl2 : -INFINITY;
        w[i] = v[i];
      }
      rw[quarter * 32 + lane] = xpose_reduce32<true>(w, lane);
      wg_sync(wg);
      if (wt < 32) {
        const float mo = cm[ch * 32 + wt];
        const float mn = fmaxf(mo, fmaxf(fmaxf(rw[wt], rw[32 + wt]), fmaxf(rw[64 + wt], rw[96 + wt])));
        ca[ch * 32 + wt] = mo == mn ? 1.f : ex2(mo - mn);  // mo = -inf: nothing accumulated yet
        cm[ch * 32 + wt] = mn;
      }
      wg_sync(wg);
      raised |= j > 0;
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        const float p0 = valid ? ex2(v[i] - cm[ch * 32 + i]) : 0.f;
        const float p1 = valid ? ex2(v[i + 1] - cm[ch * 32 + i + 1]) : 0.f;
        const __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
        w[i] = __low2float(h2);
        w[i + 1] = __high2float(h2);
        pk[i / 2] = *reinterpret_cast<const uint32_t*>(&h2);
      }
#pragma unroll
      for (int c4 = 0; c4 < 4; ++c4)
        *reinterpret_cast<uint4*>(prow + (ch * 4 + c4) * 128) =
            make_uint4(pk[4 * c4], pk[4 * c4 + 1], pk[4 * c4 + 2], pk[4 * c4 + 3]);
      rw[quarter * 32 + lane] = xpose_reduce32<false>(w, lane);
      wg_sync(wg);
      if (wt < 32) cl[ch * 32 + wt] = cl[ch * 32 + wt] * ca[ch * 32 + wt] + ((rw[wt] + rw[32 + wt]) + (rw[64 + wt] + rw[96 + wt]));
      wg_sync(wg);
      if (raised) {
        // The partial O^T of the tiles before (every PV product of them is
        // done) takes the columns' factors.
        float o[32];
        tmem_ld32(ocol + qoff + 32 * ch, o);
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] *= ca[ch * 32 + i];
        tmem_st32(ocol + qoff + 32 * ch, reinterpret_cast<const uint32_t*>(o));
        tmem_wait_st();
      }
    }
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0) {
      const uint32_t idesc = idesc_bf16(D, a.nq, 1, 1);
#pragma unroll
      for (int kq = 0; kq < TM / 16; ++kq)
        mma_bf16(ocol, smem_desc_sw128(smem_u32(vt) + kq * 2048, HALF, 1024),
                 smem_desc(smem_u32(pb) + kq * 2 * (a.nq * 16), a.nq * 16, 128), idesc, (j > 0 || kq > 0) ? 1u : 0u);
      mma_commit(smem_u32(&bar[1]));
    }
    __syncwarp();
    bool pok = mbar_wait_bounded(smem_u32(&bar[1]), ph, a.wait_limit);
    if (!pok) {
      atomicExch(a.status, 1);
      (void)mbar_wait_bounded(smem_u32(&bar[1]), ph, kWait);
    }
    ok = __syncthreads_and(pok);
    tc_fence_after();
  }
  if (ok) {  // every split holds at least one tile, so the loop ran
    // Thread wt holds head-dim row wt of O^T: its warpgroup's query chunks.
    const float ln2 = 0.69314718055994531f;
#pragma unroll 1
    for (int ch = wg; ch < nch; ch += NWG) {
      float o[32];
      tmem_ld32(ocol + qoff + 32 * ch, o);
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int cl_ = ch * 32 + i;  // column within the block
        if (cl_ < qb) {
          const int colq = c0 + cl_;
          const int hq = head_of(colq, a.rqs);
          const int64_t uq = bb * (a.H * a.G) + hh * a.G + hq;
          const int iq = colq - hq * a.qs;
          a.Opart[(((int64_t)uq * a.nsplit + sp) * a.qstride + iq) * D + wt] = o[i];
        }
      }
    }
    for (int cl_ = tid; cl_ < qb; cl_ += NTH) {
      const int colq = c0 + cl_;
      const int hq = head_of(colq, a.rqs);
      const int64_t uq = bb * (a.H * a.G) + hh * a.G + hq;
      a.ML[((int64_t)uq * a.nsplit + sp) * a.qstride + colq - hq * a.qs] = make_float2(cm[cl_] * ln2, cl[cl_]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(*tbase, a.tcols);
  }
}

}  // namespace

bool tc_attn_supported(const AttnPlan& p, int kv_group_rows) {
  return p.dtype == WF_BF16 && p.d == D && kv_group_rows <= 256;
}

cudaError_t launch_tc_attn(const AttnPlan& p, const void* Q, const wf_tensor& qd, const void* K, const void* V,
                           const wf_tensor& kv, const int32_t* idx, const void* Kg, const void* Vg,
                           const wf_tensor* g, float scale, int* status, void* ws, int* nsplit_out,
                           cudaStream_t s) {
  TcAttnArgs a;
  a.Q = static_cast<const bf16*>(Q);
  a.qsb = qd.stride_b; a.qsh = qd.stride_h; a.qss = qd.stride_s;
  a.K = static_cast<const bf16*>(K);
  a.V = static_cast<const bf16*>(V);
  a.ksb = kv.stride_b; a.ksh = kv.stride_h; a.kss = kv.stride_s;
  a.Kg = static_cast<const bf16*>(Kg);
  a.Vg = static_cast<const bf16*>(Vg);
  a.gsb = g ? g->stride_b : 0; a.gsh = g ? g->stride_h : 0; a.gss = g ? g->stride_s : 0;
  a.idx = idx;
  a.n = kv.seq; a.k = p.k; a.ng = p.ng;
  a.G = p.G; a.qs = p.q; a.q = p.G * p.q; a.H = kv.heads;
  a.rqs = 1.0f / (float)a.qs;
  // Column blocks of at most 128 query rows: S^T and O^T then take at most
  // 256 TMEM columns, so two CTAs share an SM.
  const int nblk = (a.q + 127) / 128;
  a.cb = (((a.q + nblk - 1) / nblk) + 31) / 32 * 32;
  a.nq = a.cb;
  uint32_t cols = 32;
  while ((int)cols < 2 * a.nq) cols *= 2;
  a.tcols = cols;
  // Splits of several key tiles when the grid would otherwise exceed about
  // two CTAs an SM (a CTA keeps a running max across its tiles): fewer
  // partials to write and fold.
  const int tiles = (p.k + p.ng + TM - 1) / TM;
  int sms = sm_count();
  if (sms <= 0) sms = 148;
  const int64_t ctas_per_split = (int64_t)kv.batch * kv.heads * nblk;
  a.tps = 1;
  while (a.tps < tiles && ctas_per_split * ((tiles + a.tps - 1) / a.tps) > 2 * sms) ++a.tps;
  a.nsplit = (tiles + a.tps - 1) / a.tps;
  a.Opart = reinterpret_cast<float*>(static_cast<char*>(ws) + p.off_o);
  a.ML = reinterpret_cast<float2*>(static_cast<char*>(ws) + p.off_ml);
  a.qstride = p.qstride;
  a.status = status;
  a.sl2 = 1.4426950408889634f * scale;
  const WaitControls wc = wait_controls();
  a.wait_limit = wc.limit;
  a.stall = wc.stall;
  size_t smem = 4 * HALF + (size_t)(a.nq / 8) * QGRP + sizeof(float) * (NWG * 4 * 32 + 768) + 32;
  const size_t per_sm = 228 * 1024;
  const size_t cap = 512 / cols;
  const size_t floor_smem = per_sm / (cap + 1) + 1;
  if (cap < (size_t)(2048 / NTH) && smem < floor_smem) smem = floor_smem;
  cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(tc_attn_kernel), smem);
  if (e != cudaSuccess) return e;
  tc_attn_kernel<<<dim3((unsigned)a.nsplit, (unsigned)(kv.batch * kv.heads), (unsigned)nblk), NTH, smem, s>>>(a);
  *nsplit_out = a.nsplit;
  return cudaGetLastError();
}

}  // namespace wf
