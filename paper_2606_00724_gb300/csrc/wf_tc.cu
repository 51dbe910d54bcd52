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

#include <algorithm>

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
// path: one CTA per (key unit, query-column block, split of consecutive
// 128-key tiles).  A tile's K and V rows ([K[idx]; Kg] and [V[idx]; Vg]) are
// gathered into 128-byte-swizzled tiles, S^T = K Q^T goes to TMEM (keys on
// the lanes, the unit's query rows on the columns), every thread turns its
// key's row into P = 2^(s - m) with m the running per-query max (bf16,
// stored as P^T in MN-major core matrices), and O^T += V^T P^T accumulates in
// TMEM; a raised max rescales the partial O^T and the row sums.
// The copies run one tile ahead: the next tile's K rows are issued as soon as
// the current tile's S^T has been issued (two K stages), its V rows as soon as
// the current PV product has completed, so the gathers overlap the softmax.
// This kernel takes key units of at most 32 query rows (one chunk of 32 TMEM
// columns, two CTAs an SM); wider units (grouped heads) go to the kernel with
// the query rows on the TMEM lanes further below.  The partial (O, m, l) of
// every query row lands in the flash-decoding layout of the fp32 kernels, per
// query head, so the same combine kernel finishes it.
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
  int cb;                     // query rows of a CTA's column block (all of the unit's: the grid has one block)
  int nq;                     // query rows padded: to 32 (keys-on-lanes kernel) or to M tiles of 128 (rows kernel)
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

// Shared-memory bytes of a CTA: two K stages, the V tile, the query block,
// the reduction slots, the per-query running max, row sums and factors,
// barriers.
__host__ __device__ constexpr size_t tc_attn_smem(int nq) {
  return 6 * (size_t)HALF + (size_t)(nq / 8) * QGRP + sizeof(float) * (NWG * 128 + 3 * 256) + 32;
}

__global__ void __launch_bounds__(NTH, 2) tc_attn_kernel(const __grid_constant__ TcAttnArgs a) {
  constexpr int NTA = NTH, NW = NWG, CW = 1;  // CW: query chunks of 32 a warpgroup takes (nq = 32)
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* kst = smem;                         // K stages, 2 x (2 x HALF)
  uint8_t* vt = smem + 4 * HALF;               // V tile, 2 x HALF
  uint8_t* sq = smem + 6 * HALF;               // query block, nq / 8 groups of QGRP
  // P^T (16 key groups of nq * 16 bytes) takes the current K stage's place:
  // the K rows are dead once the S^T products have completed.
  float* red = reinterpret_cast<float*>(sq + (a.nq / 8) * QGRP);  // [NW][CW][4][32]
  float* cm = red + NW * CW * 128;             // [256] running max per query (log2 units)
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
  const int tile0 = sp * a.tps;               // the split's first tile
  const int nt = min(a.tps, (total + TM - 1) / TM - tile0);  // its tiles (at least one)

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
  for (int e = tid; e < 256; e += NTA) {
    cm[e] = -INFINITY;
    cl[e] = 0.f;
  }
  for (int e = tid; e < a.nq * (D / 8); e += NTA) {
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

  // Row copies of a tile: chunk c = tid % 16 of rows r0 + (NTA / 16) i
  // (r0 = tid / 16).  Lane c resolves the K and V rows of row
  // r0 + (NTA / 16) (c % RPT) (a sparse key or a generation row) and the
  // half-warp shares the row addresses by shuffles; the swizzle term of a
  // thread's rows is constant.
  constexpr int RPT = TM / (NTA / 16);
  static_assert(RPT * (NTA / 16) == TM && (NTA / 16) % 8 == 0, "rows of a thread share r % 8");
  const int cc = tid & 15, r0 = tid >> 4, half = tid & 16;
  const uint32_t xs = ((cc >> 3) * HALF) + (uint32_t)r0 * 128u + (uint32_t)(((cc ^ r0) & 7) << 4);
  const int32_t* ui = a.idx + (int64_t)u * a.k;
  auto row_addrs = [&](int t0, unsigned long long& ka, unsigned long long& va) {
    const int tl = min(t0 + r0 + (NTA / 16) * (cc & (RPT - 1)), total - 1);  // keys past the list repeat its last key (P = 0 there)
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
    ka = reinterpret_cast<unsigned long long>(kl);
    va = reinterpret_cast<unsigned long long>(vl);
  };
  auto issue_rows = [&](uint32_t base, unsigned long long pa) {
#pragma unroll
    for (int i = 0; i < RPT; ++i) {
      const unsigned long long p = __shfl_sync(0xffffffffu, pa, half | i);
      cp_async16(base + xs + (uint32_t)(NTA / 16) * 128u * i, reinterpret_cast<const bf16*>(p) + cc * 8);
    }
  };
  // Copy groups, oldest first: [Q, K_0] [V_0], then per tile j: [K_{j+1}]
  // after the S^T issue, [V_{j+1}] after the PV product (empty groups past
  // the split's last tile), so "all but the newest group" is always the
  // group a step needs.
  unsigned long long kan, van;
  row_addrs(tile0 * TM, kan, van);
  issue_rows(smem_u32(kst), kan);
  cp_async_commit();
  issue_rows(smem_u32(vt), van);
  cp_async_commit();

  const uint32_t qoff = (uint32_t)(quarter * 32) << 16;
  const int nch = a.nq / 32;
  const int ncw = (nch - wg + NW - 1) / NW;  // this warpgroup's chunks: wg, wg + NW, ...
  float* rw = red + wg * CW * 128;
  uint32_t tmem = 0, ocol = 0;
  bool ok = true;
#pragma unroll 1
  for (int j = 0; j < nt; ++j) {
    const int t0 = (tile0 + j) * TM;
    uint8_t* kt = kst + (j & 1) * 2 * HALF;
    uint8_t* pb = kt;
    cp_async_wait<1>();  // K_j (and the query block)
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
    // The next tile's K rows into the other stage (its last reader, the S^T
    // products of tile j - 1 and, when P^T lives there, the PV product of
    // tile j - 1, has completed).
    if (j + 1 < nt) {
      row_addrs(t0 + TM, kan, van);
      issue_rows(smem_u32(kst + ((j + 1) & 1) * 2 * HALF), kan);
    }
    cp_async_commit();
    bool sok = mbar_wait_bounded(smem_u32(&bar[(a.stall && j == 0) ? 2 : 0]), ph, a.wait_limit);
    if (!sok) {
      // Drain the score MMAs (default bound) before the TMEM is freed.
      atomicExch(a.status, 1);
      (void)mbar_wait_bounded(smem_u32(&bar[0]), ph, kWait);
    }
    ok = __syncthreads_and(sok);
    tc_fence_after();
    if (!ok) break;

    // Thread wt of every warpgroup owns key t0 + wt (TMEM lane wt); the
    // warpgroups take the 32-column chunks in turn.  (1) Each warp's max per
    // column of every chunk; (2) the column's new running max and factor;
    // (3) P, its bf16 copy into P^T, each warp's row sums per column and the
    // partial O^T rescaled where a max rose; (4) the running row sums.
    const bool valid = t0 + wt < total;
#pragma unroll 1
    for (int cw = 0; cw < ncw; ++cw) {
      float v[32];
      tmem_ld32(tmem + qoff + 32 * (wg + NW * cw), v);
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = valid ? v[i] : -INFINITY;
      rw[(cw * 4 + quarter) * 32 + lane] = xpose_reduce32<true>(v, lane);
    }
    wg_sync(wg);
    const int ucw = wt >> 5, ucol = (wg + NW * ucw) * 32 + lane;  // the column this thread updates
    if (ucw < ncw) {
      const float* r = rw + ucw * 128 + lane;
      const float mo = cm[ucol];
      const float mn = fmaxf(mo, fmaxf(fmaxf(r[0], r[32]), fmaxf(r[64], r[96])) * a.sl2);
      ca[ucol] = mo == mn ? 1.f : ex2(mo - mn);  // mo = -inf: nothing accumulated yet
      cm[ucol] = mn;
    }
    wg_sync(wg);
    uint8_t* prow = pb + (wt >> 3) * (a.nq * 16) + (wt & 7) * 16;
#pragma unroll 1
    for (int cw = 0; cw < ncw; ++cw) {
      const int ch = wg + NW * cw;
      float v[32];
      uint32_t pk[16];
      tmem_ld32(tmem + qoff + 32 * ch, v);
      const uint32_t cma = smem_u32(cm + ch * 32), caa = smem_u32(ca + ch * 32);
      bool rescale = false;
#pragma unroll
      for (int k4 = 0; k4 < 8; ++k4) {
        const uint4 mc = lds_v4(cma + 16u * k4);
        const float m4[4] = {__uint_as_float(mc.x), __uint_as_float(mc.y), __uint_as_float(mc.z), __uint_as_float(mc.w)};
#pragma unroll
        for (int e = 0; e < 4; e += 2) {
          const int i = 4 * k4 + e;
          const float p0 = valid ? ex2(fmaf(v[i], a.sl2, -m4[e])) : 0.f;
          const float p1 = valid ? ex2(fmaf(v[i + 1], a.sl2, -m4[e + 1])) : 0.f;
          const __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
          v[i] = __low2float(h2);
          v[i + 1] = __high2float(h2);
          pk[i / 2] = *reinterpret_cast<const uint32_t*>(&h2);
        }
        if (j > 0) {
          const uint4 f = lds_v4(caa + 16u * k4);
          rescale |= (__uint_as_float(f.x) != 1.f) | (__uint_as_float(f.y) != 1.f) |
                     (__uint_as_float(f.z) != 1.f) | (__uint_as_float(f.w) != 1.f);
        }
      }
#pragma unroll
      for (int c4 = 0; c4 < 4; ++c4)
        *reinterpret_cast<uint4*>(prow + (ch * 4 + c4) * 128) =
            make_uint4(pk[4 * c4], pk[4 * c4 + 1], pk[4 * c4 + 2], pk[4 * c4 + 3]);
      rw[(cw * 4 + quarter) * 32 + lane] = xpose_reduce32<false>(v, lane);
      if (rescale) {
        // The partial O^T of the tiles before (every PV product of them is
        // done) takes the columns' factors (the same for every thread of the
        // warpgroup, so the branch is uniform).
        float o[32];
        tmem_ld32(ocol + qoff + 32 * ch, o);
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] *= ca[ch * 32 + i];
        tmem_st32(ocol + qoff + 32 * ch, reinterpret_cast<const uint32_t*>(o));
        tmem_wait_st();
      }
    }
    wg_sync(wg);
    if (ucw < ncw) {
      const float* r = rw + ucw * 128 + lane;
      cl[ucol] = cl[ucol] * ca[ucol] + ((r[0] + r[32]) + (r[64] + r[96]));
    }
    cp_async_wait<1>();  // V_j
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
    // The next tile's V rows (the V tile's reader, this PV product, is done;
    // after a failed wait nothing more is issued).
    if (ok && j + 1 < nt) issue_rows(smem_u32(vt), van);
    cp_async_commit();
    if (!ok) break;
  }
  cp_async_wait_all();  // no copy outlives the CTA
  if (ok) {
    // Thread wt holds head-dim row wt of O^T: its warpgroup's query chunks.
    const float ln2 = 0.69314718055994531f;
#pragma unroll 1
    for (int ch = wg; ch < nch; ch += NW) {
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
    for (int cl_ = tid; cl_ < qb; cl_ += NTA) {
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

// The same attention with the query rows on the TMEM lanes, for key units of
// more than 32 query rows (grouped heads): S = Q K^T per M tile of 128 query
// rows (N = the tile's 128 keys), one thread per query row, so the row max and
// the row sum are a thread's own serial reductions with no cross-lane
// exchange.  The thread writes its row of P (bf16) into shared memory in the
// K-major core-matrix layout of an A operand, and O = P V (N = head_dim, V the
// MN-major B operand) accumulates in TMEM.  The stabiliser is raised lazily:
// a row keeps its max until a tile's max exceeds it by more than kLazy (log2
// units), so P stays below 2^kLazy and the partial O and row sum are rescaled
// only then (the warp together).  Copies run one tile ahead as in the kernel
// above.  Up to two M tiles (256 query rows); warpgroup mt computes M tile mt.
constexpr float kLazy = 8.f;

__host__ __device__ constexpr size_t tc_attn_rows_smem(int nmt) {
  return 6 * (size_t)HALF + 2 * (size_t)nmt * 16 * QGRP + 32;  // K stages, V, Q blocks, P blocks
}

__global__ void __launch_bounds__(NTH, 1) tc_attn_rows_kernel(const __grid_constant__ TcAttnArgs a) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const int nmt = a.nq / 128;                  // M tiles of 128 query rows (1 or 2)
  uint8_t* kst = smem;                         // K stages, 2 x (2 x HALF)
  uint8_t* vt = smem + 4 * HALF;               // V tile, 2 x HALF
  uint8_t* sq = smem + 6 * HALF;               // query rows: 16 groups of QGRP an M tile
  uint8_t* pq = sq + nmt * 16 * QGRP;          // P: 16 groups of 8 rows x 128 keys (2048 bytes) an M tile
  unsigned long long* bar = reinterpret_cast<unsigned long long*>(pq + nmt * 16 * QGRP);  // S done, PV done, stall
  uint32_t* tbase = reinterpret_cast<uint32_t*>(bar + 3);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int mt = tid >> 7, r = tid & 127, quarter = warp & 3;
  const int sp = blockIdx.x, u = blockIdx.y;
  const int64_t bb = u / a.H, hh = u % a.H;
  const int total = a.k + a.ng;
  const int qb = a.q;                          // one column block: every query row of the key unit
  const int tile0 = sp * a.tps;
  const int nt = min(a.tps, (total + TM - 1) / TM - tile0);

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
  for (int e = tid; e < nmt * 128 * (D / 8); e += NTH) {
    const int rr = e & 7, ch = (e >> 3) & (D / 8 - 1), g = e >> 7;
    const int i = g * 8 + rr;
    const uint32_t dst = smem_u32(sq + g * QGRP + ch * 128 + rr * 16);
    if (i < qb) {
      const int hi = head_of(i, a.rqs);
      const bf16* qp = a.Q + bb * a.qsb + (hh * a.G + hi) * a.qsh + (int64_t)(i - hi * a.qs) * a.qss;
      cp_async16(dst, qp + ch * 8);
    } else {
      sts_v4(dst, make_uint4(0, 0, 0, 0));
    }
  }
  // Row copies as in the kernel above (256 threads: 8 rows a thread).
  constexpr int RPT = TM / (NTH / 16);
  static_assert(RPT == 8 && (NTH / 16) % 8 == 0, "rows of a thread share r % 8");
  const int cc = tid & 15, r0 = tid >> 4, half = tid & 16;
  const uint32_t xs = ((cc >> 3) * HALF) + (uint32_t)r0 * 128u + (uint32_t)(((cc ^ r0) & 7) << 4);
  const int32_t* ui = a.idx + (int64_t)u * a.k;
  auto row_addrs = [&](int t0, unsigned long long& ka, unsigned long long& va) {
    const int tl = min(t0 + r0 + (NTH / 16) * (cc & (RPT - 1)), total - 1);
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
    ka = reinterpret_cast<unsigned long long>(kl);
    va = reinterpret_cast<unsigned long long>(vl);
  };
  auto issue_rows = [&](uint32_t base, unsigned long long pa) {
#pragma unroll
    for (int i = 0; i < RPT; ++i) {
      const unsigned long long p = __shfl_sync(0xffffffffu, pa, half | i);
      cp_async16(base + xs + (uint32_t)(NTH / 16) * 128u * i, reinterpret_cast<const bf16*>(p) + cc * 8);
    }
  };
  unsigned long long kan, van;
  row_addrs(tile0 * TM, kan, van);
  issue_rows(smem_u32(kst), kan);
  cp_async_commit();
  issue_rows(smem_u32(vt), van);
  cp_async_commit();

  const uint32_t lq = (uint32_t)(quarter * 32) << 16;  // this warp's TMEM lane quarter
  const bool active = mt < nmt;                        // a warpgroup past the M tiles only copies
  uint32_t tmem = 0;
  float mrun = -INFINITY, lrun = 0.f;  // the row's stabiliser (log2 units) and sum of P
  // This thread's row of P: group r / 8 of its M tile, row r % 8 of the core matrices.
  const uint32_t prow = smem_u32(pq) + (uint32_t)(mt * 16 + (r >> 3)) * QGRP + (uint32_t)(r & 7) * 16u;
  bool ok = true;
#pragma unroll 1
  for (int j = 0; j < nt; ++j) {
    const int t0 = (tile0 + j) * TM;
    uint8_t* kt = kst + (j & 1) * 2 * HALF;
    cp_async_wait<1>();  // K_j (and the query rows)
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    tmem = *tbase;
    const uint32_t ph = (uint32_t)j & 1u;
    if (tid == 0) {
      const uint32_t idesc = idesc_bf16(128, TM, 0, 0);
#pragma unroll 1
      for (int m = 0; m < nmt; ++m)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_bf16(tmem + (uint32_t)(m * TM), smem_desc(smem_u32(sq) + m * 16 * QGRP + (4 * h + kk) * 256, 128, QGRP),
                     smem_desc_sw128(smem_u32(kt) + h * HALF + kk * 32, 16, 1024), idesc, (h | kk) != 0);
      mma_commit(smem_u32(&bar[0]));
    }
    __syncwarp();
    if (j + 1 < nt) {
      row_addrs(t0 + TM, kan, van);
      issue_rows(smem_u32(kst + ((j + 1) & 1) * 2 * HALF), kan);
    }
    cp_async_commit();
    bool sok = mbar_wait_bounded(smem_u32(&bar[(a.stall && j == 0) ? 2 : 0]), ph, a.wait_limit);
    if (!sok) {
      atomicExch(a.status, 1);
      (void)mbar_wait_bounded(smem_u32(&bar[0]), ph, kWait);
    }
    ok = __syncthreads_and(sok);
    tc_fence_after();
    if (!ok) break;

    if (active) {
      // The row's 128 logits (keys past the list: -inf, P = 0).
      uint32_t sv[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32_issue(tmem + (uint32_t)(mt * TM + 32 * c) + lq, sv + 32 * c);
      tmem_wait_ld();
      const int nvalid = total - t0;
      if (nvalid < TM) {
#pragma unroll
        for (int k = 0; k < TM; ++k) sv[k] = k < nvalid ? sv[k] : __float_as_uint(-INFINITY);
      }
      float mx = -INFINITY;
#pragma unroll
      for (int k = 0; k < TM; k += 2) mx = fmax3(mx, __uint_as_float(sv[k]), __uint_as_float(sv[k + 1]));
      const float mnew = mx * a.sl2;
      float alpha = 1.f;
      if (mnew > mrun + kLazy) {
        alpha = ex2(mrun - mnew);  // 0 on the first tile (mrun = -inf)
        mrun = mnew;
      }
      const float nm = -mrun;
      float sum[4] = {0.f, 0.f, 0.f, 0.f};  // of the bf16 values the PV product uses
#pragma unroll
      for (int c = 0; c < TM / 8; ++c) {
        uint32_t pk[4];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
          const float p0 = ex2(fmaf(__uint_as_float(sv[8 * c + e]), a.sl2, nm));
          const float p1 = ex2(fmaf(__uint_as_float(sv[8 * c + e + 1]), a.sl2, nm));
          const __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
          sum[e / 2] += __low2float(h2) + __high2float(h2);
          pk[e / 2] = *reinterpret_cast<const uint32_t*>(&h2);
        }
        sts_v4(prow + (uint32_t)c * 128u, make_uint4(pk[0], pk[1], pk[2], pk[3]));
      }
      lrun = lrun * alpha + ((sum[0] + sum[1]) + (sum[2] + sum[3]));
      if (j > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
        // The partial O of the tiles before (their PV products are done)
        // takes the row's factor.
        const uint32_t orow = tmem + (uint32_t)(nmt * TM + mt * D) + lq;
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(orow + 32 * c, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(orow + 32 * c, reinterpret_cast<const uint32_t*>(o));
        }
        tmem_wait_st();
      }
    }
    cp_async_wait<1>();  // V_j
    fence_proxy_async();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0) {
      const uint32_t idesc = idesc_bf16(128, D, 0, 1);
#pragma unroll 1
      for (int m = 0; m < nmt; ++m)
#pragma unroll
        for (int kq = 0; kq < TM / 16; ++kq)
          mma_bf16(tmem + (uint32_t)(nmt * TM + m * D), smem_desc(smem_u32(pq) + m * 16 * QGRP + kq * 256, 128, QGRP),
                   smem_desc_sw128(smem_u32(vt) + kq * 2048, HALF, 1024), idesc, (j > 0 || kq > 0) ? 1u : 0u);
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
    if (ok && j + 1 < nt) issue_rows(smem_u32(vt), van);
    cp_async_commit();
    if (!ok) break;
  }
  cp_async_wait_all();
  const int row = mt * 128 + r;  // query row of the key unit
  if (ok && active) {
    const uint32_t orow = tmem + (uint32_t)(nmt * TM + mt * D) + lq;
    const bool own = row < qb;
    const int hq = head_of(own ? row : 0, a.rqs);
    const int64_t uq = bb * (a.H * a.G) + hh * a.G + hq;
    const int iq = row - hq * a.qs;
    float* op = a.Opart + (((int64_t)uq * a.nsplit + sp) * a.qstride + iq) * D;
#pragma unroll 1
    for (int c = 0; c < D / 32; ++c) {
      float o[32];
      tmem_ld32(orow + 32 * c, o);
      if (own) {
#pragma unroll
        for (int i = 0; i < 32; i += 4)
          *reinterpret_cast<float4*>(op + 32 * c + i) = make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]);
      }
    }
    if (own) a.ML[((int64_t)uq * a.nsplit + sp) * a.qstride + iq] = make_float2(mrun * 0.69314718055994531f, lrun);
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
  a.cb = a.q;  // one column block: every query row of the key unit
  a.Opart = reinterpret_cast<float*>(static_cast<char*>(ws) + p.off_o);
  a.ML = reinterpret_cast<float2*>(static_cast<char*>(ws) + p.off_ml);
  a.qstride = p.qstride;
  a.status = status;
  a.sl2 = 1.4426950408889634f * scale;
  const WaitControls wc = wait_controls();
  a.wait_limit = wc.limit;
  a.stall = wc.stall;
  const int tiles = (p.k + p.ng + TM - 1) / TM;
  int sms = sm_count();
  if (sms <= 0) sms = 148;
  const int64_t units = (int64_t)kv.batch * kv.heads;
  // Splits of several key tiles (taken in a pipeline with a running max) so
  // that the grid fits one wave of `occ` CTAs an SM: fewer partials to write
  // and fold.
  auto split = [&](int occ) {
    a.tps = 1;
    while (a.tps < tiles && units * ((tiles + a.tps - 1) / a.tps) > (int64_t)occ * sms) ++a.tps;
    a.nsplit = (tiles + a.tps - 1) / a.tps;
  };
  const dim3 block(NTH);
  cudaError_t e;
  if (a.q > 32) {
    // Query rows on the TMEM lanes: one or two M tiles of 128 rows; S and O
    // take 256 TMEM columns an M tile, shared memory holds one CTA an SM.
    const int nmt = (a.q + 127) / 128;
    a.nq = 128 * nmt;
    a.tcols = 256u * (uint32_t)nmt;
    const size_t smem = tc_attn_rows_smem(nmt);
    split(1);
    if ((e = raise_smem_limit(reinterpret_cast<const void*>(tc_attn_rows_kernel), smem)) != cudaSuccess) return e;
    tc_attn_rows_kernel<<<dim3((unsigned)a.nsplit, (unsigned)units, 1), block, smem, s>>>(a);
  } else {
    // Keys on the TMEM lanes, one chunk of 32 query columns: S^T and O^T take
    // 64 TMEM columns; shared memory and registers hold two CTAs an SM.
    a.nq = 32;
    a.tcols = 64;
    const size_t smem = tc_attn_smem(a.nq);
    split(2);
    if ((e = raise_smem_limit(reinterpret_cast<const void*>(tc_attn_kernel), smem)) != cudaSuccess) return e;
    tc_attn_kernel<<<dim3((unsigned)a.nsplit, (unsigned)units, 1), block, smem, s>>>(a);
  }
  *nsplit_out = a.nsplit;
  return cudaGetLastError();
}

}  // namespace wf
