// Fused WaveFilter step (Algorithm 1 body): multi-scale skim/scan filtering
// (Eq. 7-11) and the final sparse attention, in one kernel.
//
// One thread-block cluster per (batch, head) unit; the cluster's CTAs split
// every scale's candidate list (and finally the sparse key list) into
// contiguous slices.  Per scale, each CTA:
//   1. gathers its candidate rows (pyramid level b, or raw keys for the
//      level-0 trim) with 16-byte cp.async into shared memory laid out as
//      8-row x 16-byte core matrices, and multiplies each 128-row tile by the
//      query block on the tensor cores: tcgen05.mma (bf16 in, fp32 out)
//      writes S^T = rows . Q^T into TMEM, 32 columns per tile;
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
// The attention stage gathers K/V rows of mu^0 and the generation rows, forms
// S^T = K_s Q^T in TMEM, P = exp(S - m) in bf16, and O^T = V_s^T P^T with a
// second tcgen05.mma (both operands MN-major), then the cluster's partial
// (m, l, O) are combined in CTA 0.
//
// The only waits on asynchronous work are on MMA completion mbarriers; each
// is bounded (~1 s): on timeout the CTA records a status word, skips further
// MMAs, keeps joining every cluster barrier and returns.
#include <math.h>

#include "wf_internal.cuh"
#include "wf_sm100.cuh"

namespace wf {
namespace {

using namespace sm100;

constexpr int NT = 256;                 // threads per CTA (8 warps)
constexpr int D = 128;                  // head_dim
constexpr int NCH = D / 8;              // 16-byte chunks per row
constexpr int TM = 128;                 // rows per MMA tile (M)
constexpr int NQ = 32;                  // query rows per MMA (N), zero padded
constexpr int GRP = NCH * 128;          // bytes per 8-row group of a K-major tile
constexpr int TILE_BYTES = TM * D * 2;  // 32 KB
constexpr int Q_BYTES = NQ * D * 2;     // 8 KB
constexpr int P_BYTES = NQ * TM * 2;    // 8 KB
constexpr long long kWaitLimit = 1ll << 31;
constexpr float kLog2e = 1.4426950408889634f;

constexpr uint32_t kIdescScore = idesc_bf16(TM, NQ, 0, 0);  // A = rows (K-major), B = Q (K-major)
constexpr uint32_t kIdescPV = idesc_bf16(D, NQ, 1, 1);      // A = V^T (MN-major), B = P^T (MN-major)

struct Misc {
  float2 xstat[8][32];
  float red[8][32];
  float cvec[32];
  float mloc[32];
  float lacc[32];
  int wsum[8];
  uint32_t sel_bin, sel_need, sel_cnt;
  int abort;
  uint32_t tmem_base;
  uint32_t pad;
  unsigned long long mbar[8];
};

template <int STAGES>
struct Layout {
  static constexpr uint32_t off_q = 0;
  static constexpr uint32_t off_stage = Q_BYTES;
  static constexpr uint32_t off_p = off_stage + STAGES * TILE_BYTES;
  static constexpr uint32_t off_hist = off_p + 2 * P_BYTES;
  static constexpr uint32_t off_misc = off_hist + 8 * 256 * 4;
  static constexpr uint32_t off_keys = (off_misc + sizeof(Misc) + 127) / 128 * 128;
};

__device__ __forceinline__ uint32_t okey(float f) {
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Reduce 32 values per lane across the warp's 32 lanes; afterwards lane i
// holds the reduction of column i (31 shuffles).
template <bool MAX>
__device__ __forceinline__ float transpose_reduce32(float* v, int lane) {
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

// 16 values per lane summed across all 32 lanes; lane i < 16 gets column i.
__device__ __forceinline__ float transpose_sum16(float* v, int lane) {
#pragma unroll
  for (int j = 0; j < 16; ++j) v[j] += __shfl_xor_sync(0xffffffffu, v[j], 16);
#pragma unroll
  for (int off = 8; off >= 1; off >>= 1) {
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int j = 0; j < off; ++j) {
      const float keep = up ? v[j + off] : v[j];
      const float send = up ? v[j] : v[j + off];
      v[j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
    }
  }
  return v[0];
}

// Exclusive prefix sum over the CTA's 256 threads (thread order).
__device__ __forceinline__ int block_excl_scan(int v, Misc& ms, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) ms.wsum[warp] = incl;
  __syncthreads();
  int before = 0, tot = 0;
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    const int s = ms.wsum[w];
    before += w < warp ? s : 0;
    tot += s;
  }
  __syncthreads();
  if (total) *total = tot;
  return before + incl - v;
}

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
  int q, n, ng, H, L, trim;
  int cmax, kmax;
  uint32_t tmem_cols;
  int32_t keep[12];
  float scale_log2;  // log2(e) / sqrt(d)
};

// Candidate (or token) index of position j in the current candidate list.
__device__ __forceinline__ int cand_of(int j, bool top, const int32_t* Jprev) {
  return top ? j : 2 * Jprev[j >> 1] + (j & 1);
}

// Gather 128 rows (positions g0 + t*128 + r of the candidate list) into a
// K-major core-matrix tile; rows past `mc` are zero.
__device__ __forceinline__ void load_cand_tile(uint32_t dst, const bf16* base, int64_t rstride, int g0, int t,
                                               int mc, bool top, const int32_t* Jprev) {
  const int tid = threadIdx.x;
#pragma unroll
  for (int i = 0; i < (TM * NCH) / NT; ++i) {
    const int e = tid + NT * i;
    const int rr = e & 7, c = (e >> 3) & (NCH - 1), g = e >> 7;
    const int r = t * TM + g * 8 + rr;
    const uint32_t d = dst + g * GRP + c * 128 + rr * 16;
    if (r < mc) {
      const int64_t row = cand_of(g0 + r, top, Jprev);
      cp_async16(d, base + row * rstride + c * 8);
    } else {
      st_shared_zero16(d);
    }
  }
}

// Gather 128 rows of the sparse key list [K[mu0]; Kg] (or of V) starting at
// position a0 + t*128.
__device__ __forceinline__ void load_kv_tile(uint32_t dst, const bf16* X, const bf16* Xg, const FusedParams& p,
                                             int64_t bb, int64_t hh, int a0, int t, int mc, int kk,
                                             const int32_t* Jfin) {
  const int tid = threadIdx.x;
#pragma unroll
  for (int i = 0; i < (TM * NCH) / NT; ++i) {
    const int e = tid + NT * i;
    const int rr = e & 7, c = (e >> 3) & (NCH - 1), g = e >> 7;
    const int r = t * TM + g * 8 + rr;
    const uint32_t d = dst + g * GRP + c * 128 + rr * 16;
    if (r < mc) {
      const int pos = a0 + r;
      const bf16* src;
      if (pos < kk) {
        const int tok = p.trim ? Jfin[pos] : 2 * Jfin[pos >> 1] + (pos & 1);
        src = X + bb * p.ksb + hh * p.ksh + (int64_t)tok * p.kss;
      } else {
        src = Xg + bb * p.gsb + hh * p.gsh + (int64_t)(pos - kk) * p.gss;
      }
      cp_async16(d, src + c * 8);
    } else {
      st_shared_zero16(d);
    }
  }
}

// Top-K of keys[0..m) (largest first, lower position wins ties); writes the
// kk chosen candidate indices in ascending position order to Jout.
__device__ void select_topk(const float* keys, int m, int kk, int32_t* Jout, bool top, const int32_t* Jprev,
                            Misc& ms, uint32_t* hist) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t prefix = 0, mask = 0, need = (uint32_t)kk;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = tid; i < 8 * 256; i += NT) hist[i] = 0;
    __syncthreads();
    for (int base = 0; base < m; base += NT) {
      const int j = base + tid;
      const uint32_t key = j < m ? okey(keys[j]) : 0u;
      const bool match = j < m && (key & mask) == prefix;
      const uint32_t bin = (key >> shift) & 255u;
      const unsigned act = __ballot_sync(0xffffffffu, match);
      if (match) {
        const unsigned peers = __match_any_sync(act, bin);
        if (lane == __ffs(peers) - 1) atomicAdd(&hist[warp * 256 + bin], (uint32_t)__popc(peers));
      }
    }
    __syncthreads();
    const int bin = 255 - tid;  // thread order = bins from high to low
    uint32_t tot = 0;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += hist[w * 256 + bin];
    const uint32_t above = (uint32_t)block_excl_scan((int)tot, ms, nullptr);
    if (above < need && above + tot >= need) {
      ms.sel_bin = (uint32_t)bin;
      ms.sel_need = need - above;
      ms.sel_cnt = tot;
    }
    __syncthreads();
    prefix |= ms.sel_bin << shift;
    mask |= 255u << shift;
    need = ms.sel_need;
    const bool done = ms.sel_cnt == need;
    __syncthreads();
    if (done) break;
  }
  // Order-preserving compaction over contiguous runs of positions.
  const int R = (m + NT - 1) / NT;
  const int j0 = min(m, tid * R), j1 = min(m, j0 + R);
  int eq_cnt = 0;
  for (int j = j0; j < j1; ++j) eq_cnt += (okey(keys[j]) & mask) == prefix;
  const int eq_base = block_excl_scan(eq_cnt, ms, nullptr);
  int eqs = eq_base, take_cnt = 0;
  for (int j = j0; j < j1; ++j) {
    const uint32_t km = okey(keys[j]) & mask;
    const bool eq = km == prefix;
    take_cnt += km > prefix || (eq && (uint32_t)eqs < need);
    eqs += eq;
  }
  int pos = block_excl_scan(take_cnt, ms, nullptr);
  eqs = eq_base;
  for (int j = j0; j < j1; ++j) {
    const uint32_t km = okey(keys[j]) & mask;
    const bool eq = km == prefix;
    if (km > prefix || (eq && (uint32_t)eqs < need)) Jout[pos++] = cand_of(j, top, Jprev);
    eqs += eq;
  }
  __syncthreads();
}

template <int STAGES>
struct Pipe {
  uint32_t stage_a;
  uint32_t mbar_a;
  uint32_t parity_bits;  // bit s = (commits on stage s) & 1

  __device__ uint32_t stage(int s) const { return stage_a + s * TILE_BYTES; }
  __device__ uint32_t mbar(int s) const { return mbar_a + 8 * s; }
  __device__ void committed(int s) { parity_bits ^= 1u << s; }
  // Wait (thread 0, bounded) for the last commit on stage s; uniform result.
  __device__ void wait_stage(int s, Misc& ms, int* status) {
    if (threadIdx.x == 0 && !ms.abort) {
      if (!mbar_wait_bounded(mbar(s), ((parity_bits >> s) & 1u) ^ 1u, kWaitLimit)) {
        ms.abort = 1;
        atomicExch(status, 1);
      }
    }
    __syncthreads();
  }
};

// Score the candidate slice [g0, g0 + mc) of the current scale: S^T tiles in
// TMEM columns 32 t.  Returns the number of tiles.
template <int STAGES>
__device__ int score_slice(Pipe<STAGES>& pipe, Misc& ms, int* status, uint32_t sq_a, uint32_t tmem,
                           const bf16* base, int64_t rstride, int g0, int mc, bool top, const int32_t* Jprev) {
  const int tid = threadIdx.x;
  const int ntl = (mc + TM - 1) / TM;
#pragma unroll
  for (int s = 0; s < STAGES; ++s) {
    if (s < ntl) load_cand_tile(pipe.stage(s), base, rstride, g0, s, mc, top, Jprev);
    cp_async_commit();
  }
  for (int t = 0; t < ntl; ++t) {
    const int s = t % STAGES;
    cp_async_wait<STAGES - 1>();
    fence_proxy_async();
    __syncthreads();
    const bool ab = ms.abort;
    if (tid == 0 && !ab) {
      tc_fence_after();
      const uint32_t a0 = pipe.stage(s);
#pragma unroll
      for (int ks = 0; ks < D / 16; ++ks)
        mma_bf16(tmem + 32 * t, smem_desc(a0 + ks * 256, 128, GRP), smem_desc(sq_a + ks * 256, 128, GRP),
                 kIdescScore, ks > 0);
      mma_commit(pipe.mbar(s));
    }
    if (!ab) pipe.committed(s);
    if (t + STAGES < ntl) {
      pipe.wait_stage(s, ms, status);
      load_cand_tile(pipe.stage(s), base, rstride, g0, t + STAGES, mc, top, Jprev);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();
  if (ntl > 0 && !ms.abort) pipe.wait_stage((ntl - 1) % STAGES, ms, status);
  __syncthreads();
  tc_fence_after();
  return ntl;
}

template <int STAGES>
__global__ void __launch_bounds__(NT, 1) wf_fused_kernel(const __grid_constant__ FusedParams p) {
  using LY = Layout<STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
  Misc& ms = *reinterpret_cast<Misc*>(smem + LY::off_misc);
  uint32_t* hist = reinterpret_cast<uint32_t*>(smem + LY::off_hist);
  float* keys = reinterpret_cast<float*>(smem + LY::off_keys);
  int32_t* Jbuf[2] = {reinterpret_cast<int32_t*>(smem + LY::off_keys + 4 * p.cmax),
                      reinterpret_cast<int32_t*>(smem + LY::off_keys + 4 * p.cmax + 4 * p.kmax)};
  const uint32_t sq_a = smem_u32(smem + LY::off_q);
  const uint32_t p_a = smem_u32(smem + LY::off_p);
  const uint32_t keys_a = smem_u32(keys);

  const uint32_t rank = cluster_rank(), CS = cluster_size();
  const int u = (int)cluster_id_x();
  const int64_t bb = u / p.H, hh = u % p.H;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int qd = warp & 3, half = warp >> 2;
  const uint32_t lane_base = (uint32_t)(qd * 32) << 16;

  Pipe<STAGES> pipe{smem_u32(smem + LY::off_stage), smem_u32(&ms.mbar[0]), 0u};

  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(pipe.mbar(s), 1);
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
    for (int e = tid; e < NQ * NCH; e += NT) {
      const int rr = e & 7, c = (e >> 3) & (NCH - 1), g = e >> 7;
      const int i = g * 8 + rr;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (i < p.q) v = __ldg(reinterpret_cast<const uint4*>(qb + (int64_t)i * p.qss + c * 8));
      *reinterpret_cast<uint4*>(sq + g * GRP + c * 128 + rr * 16) = v;
    }
  }
  fence_proxy_async();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ms.tmem_base;
  cluster_sync();

  const float sl2 = p.scale_log2;
  const int L = p.L;
  int m_total = p.n >> L;
  bool top = true;
  int jb = 0;  // Jbuf index of the current level's output
  const int32_t* Jprev = Jbuf[1];
  int64_t sets_off = 0;
  const int lev_end = p.trim ? 0 : 1;

  for (int lev = L; lev >= lev_end; --lev) {
    // This CTA's slice of the candidate positions.
    int g0, g1;
    if (top) {
      g0 = (int)((int64_t)rank * m_total / CS);
      g1 = (int)((int64_t)(rank + 1) * m_total / CS);
    } else {
      const int pairs = m_total / 2;
      g0 = 2 * (int)((int64_t)rank * pairs / CS);
      g1 = 2 * (int)((int64_t)(rank + 1) * pairs / CS);
    }
    const int mc = g1 - g0;
    const bf16* base;
    int64_t rstride;
    if (lev >= 1) {
      base = p.coeffs + (int64_t)u * p.rows_total * D + ((int64_t)p.n - ((int64_t)p.n >> (lev - 1))) * D;
      rstride = D;
    } else {
      base = p.K + bb * p.ksb + hh * p.ksh;
      rstride = p.kss;
    }
    const int ntl = score_slice<STAGES>(pipe, ms, p.status, sq_a, tmem, base, rstride, g0, mc, top, Jprev);

    // Pass A: per-query max over this CTA's candidates.
    float acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = -INFINITY;
    for (int t = half; t < ntl; t += 2) {
      float v[32];
      tmem_ld32(tmem + lane_base + 32 * t, v);
      if (t * TM + qd * 32 + lane < mc) {
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[i] = fmaxf(acc[i], v[i]);
      }
    }
    ms.red[warp][lane] = transpose_reduce32<true>(acc, lane);
    __syncthreads();
    if (tid < 32) {
      float m = -INFINITY;
#pragma unroll
      for (int w = 0; w < 8; ++w) m = fmaxf(m, ms.red[w][tid]);
      ms.mloc[tid] = m * sl2;  // log2 units
    }
    __syncthreads();
    // Pass B: per-query sum of 2^(l - m) over this CTA's candidates.
    {
      float ml[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) { ml[i] = ms.mloc[i]; acc[i] = 0.f; }
      for (int t = half; t < ntl; t += 2) {
        float v[32];
        tmem_ld32(tmem + lane_base + 32 * t, v);
        if (t * TM + qd * 32 + lane < mc) {
#pragma unroll
          for (int i = 0; i < 32; ++i) acc[i] += exp2f(fmaf(v[i], sl2, -ml[i]));
        }
      }
    }
    ms.red[warp][lane] = transpose_reduce32<false>(acc, lane);
    __syncthreads();
    if (tid < 32) {
      float s = 0.f;
#pragma unroll
      for (int w = 0; w < 8; ++w) s += ms.red[w][tid];
      const float m = ms.mloc[tid];
      const uint32_t local = smem_u32(&ms.xstat[rank][tid]);
      for (uint32_t r = 0; r < CS; ++r) st_cluster_v2f32(map_rank(local, r), m, s);
    }
    cluster_sync();
    // Softmax normaliser per query: c = M + log2 S over the whole candidate set.
    if (tid < 32) {
      float M = -INFINITY;
      for (uint32_t r = 0; r < CS; ++r) M = fmaxf(M, ms.xstat[r][tid].x);
      float S = 0.f;
      for (uint32_t r = 0; r < CS; ++r) {
        const float2 x = ms.xstat[r][tid];
        if (x.y > 0.f) S += x.y * exp2f(x.x - M);
      }
      ms.cvec[tid] = M + log2f(S);
    }
    __syncthreads();
    // Pass C: ranking key log2 W_j, all-gathered into every CTA's key array.
    {
      float cv[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) cv[i] = ms.cvec[i];
      for (int t = half; t < ntl; t += 2) {
        float v[32];
        tmem_ld32(tmem + lane_base + 32 * t, v);
        const int j = t * TM + qd * 32 + lane;
        float mx = -INFINITY;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          v[i] = fmaf(v[i], sl2, -cv[i]);
          if (i < p.q) mx = fmaxf(mx, v[i]);
        }
        float z = 0.f;
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (i < p.q) z += exp2f(v[i] - mx);
        const float key = mx + log2f(z);
        if (j < mc) {
          const uint32_t local = keys_a + 4u * (uint32_t)(g0 + j);
          for (uint32_t r = 0; r < CS; ++r) st_cluster_f32(map_rank(local, r), key);
        }
      }
    }
    tc_fence_before();
    cluster_sync();
    tc_fence_after();

    // Eq. 9: Top-K (same result in every CTA of the cluster).
    const int kb = p.keep[lev];
    int32_t* Jcur = Jbuf[jb];
    select_topk(keys, m_total, kb, Jcur, top, Jprev, ms, hist);
    if (lev >= 1) {
      if (rank == 0 && p.level_sets) {
        int32_t* out = p.level_sets + (int64_t)u * p.sets_stride + sets_off;
        for (int i = tid; i < kb; i += NT) out[i] = Jcur[i];
      }
      sets_off += kb;
    }
    Jprev = Jcur;
    jb ^= 1;
    m_total = 2 * kb;  // Eq. 10: children of the kept coefficients
    top = false;
  }

  // mu^0 and the sparse key list [K[mu^0]; Kg].
  const int kk = p.keep[0];
  const int32_t* Jfin = Jprev;
  if (rank == 0) {
    int32_t* out = p.idx + (int64_t)u * kk;
    int32_t* ls = p.level_sets ? p.level_sets + (int64_t)u * p.sets_stride + sets_off : nullptr;
    for (int t = tid; t < kk; t += NT) {
      const int tok = p.trim ? Jfin[t] : 2 * Jfin[t >> 1] + (t & 1);
      out[t] = tok;
      if (ls) ls[t] = tok;
    }
  }
  const int total = kk + p.ng;
  const int a0 = (int)((int64_t)rank * total / CS);
  const int a1 = (int)((int64_t)(rank + 1) * total / CS);
  const int mc = a1 - a0;
  const int ntl = (mc + TM - 1) / TM;
  const uint32_t ocol = p.tmem_cols - 32;

  // Attention phase 1: S^T = K_s Q^T.
  {
#pragma unroll
    for (int s = 0; s < STAGES; ++s) {
      if (s < ntl) load_kv_tile(pipe.stage(s), p.K, p.Kg, p, bb, hh, a0, s, mc, kk, Jfin);
      cp_async_commit();
    }
    for (int t = 0; t < ntl; ++t) {
      const int s = t % STAGES;
      cp_async_wait<STAGES - 1>();
      fence_proxy_async();
      __syncthreads();
      const bool ab = ms.abort;
      if (tid == 0 && !ab) {
        tc_fence_after();
        const uint32_t a = pipe.stage(s);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks)
          mma_bf16(tmem + 32 * t, smem_desc(a + ks * 256, 128, GRP), smem_desc(sq_a + ks * 256, 128, GRP),
                   kIdescScore, ks > 0);
        mma_commit(pipe.mbar(s));
      }
      if (!ab) pipe.committed(s);
      if (t + STAGES < ntl) {
        pipe.wait_stage(s, ms, p.status);
        load_kv_tile(pipe.stage(s), p.K, p.Kg, p, bb, hh, a0, t + STAGES, mc, kk, Jfin);
      }
      cp_async_commit();
    }
    cp_async_wait<0>();
    if (ntl > 0 && !ms.abort) pipe.wait_stage((ntl - 1) % STAGES, ms, p.status);
    __syncthreads();
    tc_fence_after();
  }
  // Per-query max over this CTA's keys (log2 units).
  {
    float acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = -INFINITY;
    for (int t = half; t < ntl; t += 2) {
      float v[32];
      tmem_ld32(tmem + lane_base + 32 * t, v);
      if (t * TM + qd * 32 + lane < mc) {
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[i] = fmaxf(acc[i], v[i]);
      }
    }
    ms.red[warp][lane] = transpose_reduce32<true>(acc, lane);
    __syncthreads();
    if (tid < 32) {
      float m = -INFINITY;
#pragma unroll
      for (int w = 0; w < 8; ++w) m = fmaxf(m, ms.red[w][tid]);
      ms.mloc[tid] = m * sl2;
    }
    __syncthreads();
  }
  // Attention phase 2: P = 2^(s - m) (bf16), O^T += V_s^T P^T.
  float lsum[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) lsum[i] = 0.f;
  {
    float ml[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) ml[i] = ms.mloc[16 * half + i];
#pragma unroll
    for (int s = 0; s < STAGES; ++s) {
      if (s < ntl) load_kv_tile(pipe.stage(s), p.V, p.Vg, p, bb, hh, a0, s, mc, kk, Jfin);
      cp_async_commit();
    }
    uint8_t* pbuf = smem + LY::off_p;
    for (int t = 0; t < ntl; ++t) {
      const int s = t % STAGES;
      const int pb = t & 1;
      // P^T tile, MN-major: key-group g = r / 8, query chunk c = i / 8.
      {
        float v[16];
        tmem_ld16(tmem + lane_base + 32 * t + 16 * half, v);
        const int r = qd * 32 + lane;
        const bool valid = t * TM + r < mc;
        uint32_t w[8];
#pragma unroll
        for (int i = 0; i < 16; i += 2) {
          const float p0 = valid ? exp2f(fmaf(v[i], sl2, -ml[i])) : 0.f;
          const float p1 = valid ? exp2f(fmaf(v[i + 1], sl2, -ml[i + 1])) : 0.f;
          const __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
          lsum[i] += __low2float(h2);
          lsum[i + 1] += __high2float(h2);
          w[i / 2] = *reinterpret_cast<const uint32_t*>(&h2);
        }
        uint8_t* dst = pbuf + pb * P_BYTES + (r >> 3) * 512 + (2 * half) * 128 + (r & 7) * 16;
        *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
        *reinterpret_cast<uint4*>(dst + 128) = make_uint4(w[4], w[5], w[6], w[7]);
      }
      cp_async_wait<STAGES - 1>();
      fence_proxy_async();
      tc_fence_before();
      __syncthreads();
      const bool ab = ms.abort;
      if (tid == 0 && !ab) {
        tc_fence_after();
        const uint32_t a = pipe.stage(s);
        const uint32_t b = p_a + pb * P_BYTES;
#pragma unroll
        for (int ks = 0; ks < TM / 16; ++ks)
          mma_bf16(tmem + ocol, smem_desc(a + ks * 2 * GRP, GRP, 128), smem_desc(b + ks * 1024, 512, 128),
                   kIdescPV, (t > 0 || ks > 0) ? 1u : 0u);
        mma_commit(pipe.mbar(s));
      }
      if (!ab) pipe.committed(s);
      // The MMA reads this V stage and P buffer: wait before either is reused.
      pipe.wait_stage(s, ms, p.status);
      tc_fence_after();
      if (t + STAGES < ntl) load_kv_tile(pipe.stage(s), p.V, p.Vg, p, bb, hh, a0, t + STAGES, mc, kk, Jfin);
      cp_async_commit();
    }
    cp_async_wait<0>();
  }
  // Row sums l over this CTA's keys.
  {
    const float r = transpose_sum16(lsum, lane);
    if (lane < 16) ms.red[warp][lane] = r;
    __syncthreads();
    if (tid < 32) {
      const int hf = tid >> 4, i = tid & 15;
      float s = 0.f;
#pragma unroll
      for (int w = 0; w < 4; ++w) s += ms.red[4 * hf + w][i];
      ms.lacc[tid] = s;
    }
    __syncthreads();
  }
  // Partial O^T -> CTA 0 of the cluster (into its stage area, now idle).
  float o[16];
  tmem_ld16(tmem + lane_base + ocol + 16 * half, o);
  tc_fence_before();
  cluster_sync();
  {
    const uint32_t recv = pipe.stage(0);
    const int d = qd * 32 + lane;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int qi = 16 * half + i;
      st_cluster_f32(map_rank(recv + 4u * (uint32_t)((rank * NQ + qi) * D + d), 0), o[i]);
    }
    if (tid < 32) {
      const uint32_t ml_a = recv + 4u * (uint32_t)(CS * NQ * D) + 8u * (rank * NQ + tid);
      st_cluster_v2f32(map_rank(ml_a, 0), ms.mloc[tid], ms.lacc[tid]);
    }
  }
  cluster_sync();
  if (rank == 0) {
    const float* part = reinterpret_cast<const float*>(smem + LY::off_stage);
    const float2* mlp = reinterpret_cast<const float2*>(part + CS * NQ * D);
    bf16* ob = p.O + bb * p.osb + hh * p.osh;
    for (int e = tid; e < p.q * D; e += NT) {
      const int qi = e / D, d = e % D;
      float M = -INFINITY;
      for (uint32_t r = 0; r < CS; ++r)
        if (mlp[r * NQ + qi].y > 0.f) M = fmaxf(M, mlp[r * NQ + qi].x);
      float num = 0.f, den = 0.f;
      for (uint32_t r = 0; r < CS; ++r) {
        const float2 x = mlp[r * NQ + qi];
        if (!(x.y > 0.f)) continue;  // a CTA with no keys sent no partial output
        const float f = exp2f(x.x - M);
        num = fmaf(part[(r * NQ + qi) * D + d], f, num);
        den = fmaf(x.y, f, den);
      }
      ob[(int64_t)qi * p.oss + d] = __float2bfloat16_rn(num / den);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, p.tmem_cols);
}

}  // namespace

// ---------------------------------------------------------------------------
// Host side.
// ---------------------------------------------------------------------------
FusedPlan plan_fused(const wf_tensor& q, const wf_tensor& kv, int levels, const int32_t* keep, int n_g,
                     int num_sms) {
  FusedPlan fp{};
  fp.ok = false;
  if (kv.dtype != WF_BF16 || kv.head_dim != D || q.seq > NQ || levels > 10) return fp;
  const int U = kv.batch * kv.heads;
  const int n = kv.seq;
  const bool trim = keep[0] < 2 * keep[1];
  int cmax = n >> levels, kmax = 0;
  for (int l = 0; l <= levels; ++l) kmax = kmax > keep[l] ? kmax : keep[l];
  for (int l = 1; l <= levels; ++l) cmax = cmax > 2 * keep[l] ? cmax : 2 * keep[l];
  const int total = keep[0] + n_g;
  auto tiles_ok = [&](int cs, int* cols) {
    int tmax = (((n >> levels) + cs - 1) / cs + TM - 1) / TM;
    for (int l = levels; l >= 1; --l) {
      const int t = (2 * ((keep[l] + cs - 1) / cs) + TM - 1) / TM;
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
  const size_t kMaxSmem = 227 * 1024 - 128;  // 128 bytes of alignment slack
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
  FusedParams p{};
  p.Q = static_cast<const bf16*>(Q);
  p.qsb = qd.stride_b; p.qsh = qd.stride_h; p.qss = qd.stride_s;
  p.K = static_cast<const bf16*>(K);
  p.V = static_cast<const bf16*>(V);
  p.ksb = kv.stride_b; p.ksh = kv.stride_h; p.kss = kv.stride_s;
  p.Kg = static_cast<const bf16*>(Kg);
  p.Vg = static_cast<const bf16*>(Vg);
  p.gsb = g ? g->stride_b : 0; p.gsh = g ? g->stride_h : 0; p.gss = g ? g->stride_s : 0;
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
  cfg.dynamicSmemBytes = fp.smem + 128;
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
    e = cudaFuncSetAttribute(wf_fused_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cfg.dynamicSmemBytes);
    if (e != cudaSuccess) return e;
    e = cudaLaunchKernelEx(&cfg, wf_fused_kernel<4>, p);
  } else {
    e = cudaFuncSetAttribute(wf_fused_kernel<3>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cfg.dynamicSmemBytes);
    if (e != cudaSuccess) return e;
    e = cudaLaunchKernelEx(&cfg, wf_fused_kernel<3>, p);
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace wf
