// Skim and scan (Eq. 7-11): per scale, three kernels over all (batch, head)
// units at once.
//   score   : logits s_ij = Q_i . A_l[c_j] / sqrt(d) for a tile of 32
//             candidates (gathered by index), plus the tile's per-query
//             softmax partials (max, sum of exp).
//   weights : the global per-query max / normaliser from the tile partials,
//             then the ranking key log W_j, W_j = sum_i exp(s_ij - M_i) / S_i,
//             for 256 candidates.
//   select  : one CTA per unit; radix select of the keep[l]-th largest key
//             (four 8-bit passes over the fp32 bit patterns), then an
//             order-preserving compaction: every key above the threshold plus
//             the lowest-index ties, emitted in candidate (= index) order and
//             expanded to the children {2c, 2c+1} of Eq. 10.
// fp32 arithmetic throughout, exact fp32 exp (expf).
#include <math.h>

#include "wf_internal.cuh"

namespace wf {
namespace {

constexpr int TILE = kScoreTile;
constexpr int QMAX = kMaxQ;

// Query row i of unit (b, h): row i % qs of query head h G + i / qs.
template <typename T>
__device__ __forceinline__ const T* query_row(const T* Q, int64_t qsb, int64_t qsh, int64_t qss, int64_t bb,
                                              int64_t hh, int G, int qs, int i) {
  return Q + bb * qsb + (hh * G + i / qs) * qsh + (int64_t)(i % qs) * qss;
}

// Grid (candidate tiles, units, query chunks of QM rows).
template <typename T, int D, int QM>
__global__ void __launch_bounds__(256) score_kernel(const T* __restrict__ Q, int64_t qsb, int64_t qsh, int64_t qss,
                                                    int q, int G, int qs, int H, RowSrc src,
                                                    const int32_t* __restrict__ cand,
                                                    int64_t cand_stride, int m, float scale,
                                                    float* __restrict__ logits, int64_t lg_unit, int64_t lg_row,
                                                    float2* __restrict__ part, int64_t part_unit) {
  constexpr int VEC = Vec<T>::N;
  constexpr int RS = D + 4;  // padded row stride of the candidate tile (keeps 16-byte alignment)
  extern __shared__ __align__(16) float smem[];
  float* Qs = smem;              // [QM][D]
  float* Rs = smem + QM * D;     // [TILE][RS]
  const int u = blockIdx.y;
  const int j0 = blockIdx.x * TILE;
  const int i0 = blockIdx.z * QM;  // first query row of this chunk
  const int64_t bb = u / H, hh = u % H;
  const int tid = threadIdx.x;

  for (int e = tid; e < QM * (D / VEC); e += blockDim.x) {
    const int i = e / (D / VEC), c = (e % (D / VEC)) * VEC;
    float v[VEC];
    if (i0 + i < q) ld_vec(query_row(Q, qsb, qsh, qss, bb, hh, G, qs, i0 + i) + c, v);
    else
#pragma unroll
      for (int x = 0; x < VEC; ++x) v[x] = 0.f;
#pragma unroll
    for (int x = 0; x < VEC; ++x) Qs[i * D + c + x] = v[x];
  }
  const T* rbase = static_cast<const T*>(src.base) + bb * src.sb + hh * src.sh + src.off;
  for (int e = tid; e < TILE * (D / VEC); e += blockDim.x) {
    const int j = e / (D / VEC), c = (e % (D / VEC)) * VEC;
    const int jj = j0 + j;
    float v[VEC];
    if (jj < m) {
      const int64_t r = cand ? (int64_t)cand[(int64_t)u * cand_stride + jj] : (int64_t)jj;
      ld_vec(rbase + r * src.ss + c, v);
    } else {
#pragma unroll
      for (int x = 0; x < VEC; ++x) v[x] = 0.f;
    }
#pragma unroll
    for (int x = 0; x < VEC; ++x) Rs[j * RS + c + x] = v[x];
  }
  __syncthreads();

  const int lane = tid & 31, warp = tid >> 5;  // lane = candidate, warp = query phase
  float acc[QM / 8];
#pragma unroll
  for (int r = 0; r < QM / 8; ++r) acc[r] = 0.f;
#pragma unroll 4
  for (int c = 0; c < D; c += 4) {
    const float4 rv = *reinterpret_cast<const float4*>(&Rs[lane * RS + c]);
#pragma unroll
    for (int r = 0; r < QM / 8; ++r) {
      const float4 qv = *reinterpret_cast<const float4*>(&Qs[(warp + 8 * r) * D + c]);
      acc[r] = fmaf(qv.x, rv.x, acc[r]);
      acc[r] = fmaf(qv.y, rv.y, acc[r]);
      acc[r] = fmaf(qv.z, rv.z, acc[r]);
      acc[r] = fmaf(qv.w, rv.w, acc[r]);
    }
  }
  const int jj = j0 + lane;
  const bool valid = jj < m;
  float* lg = logits + (int64_t)u * lg_unit;
  float2* pt = part + (int64_t)u * part_unit + (int64_t)blockIdx.x * q;
#pragma unroll
  for (int r = 0; r < QM / 8; ++r) {
    const int i = i0 + warp + 8 * r;
    if (i >= q) break;
    const float s = acc[r] * scale;
    if (valid) lg[(int64_t)i * lg_row + jj] = s;
    float mx = valid ? s : -INFINITY;
#pragma unroll
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float e = valid ? expf(s - mx) : 0.f;
#pragma unroll
    for (int o = 16; o; o >>= 1) e += __shfl_xor_sync(0xffffffffu, e, o);
    if (lane == 0) pt[i] = make_float2(mx, e);
  }
}

__global__ void __launch_bounds__(256) weights_kernel(const float* __restrict__ logits, int64_t lg_unit,
                                                      int64_t lg_row, const float2* __restrict__ part,
                                                      int64_t part_unit, int ntiles, int q, int m,
                                                      float* __restrict__ W, int64_t w_unit) {
  // Per query row i: M_i = max_j s_ij and log S_i = log sum_j exp(s_ij - M_i),
  // combined from the tile partials.  Then the ranking key of candidate j is
  // log W_j = log sum_i exp(s_ij - M_i - log S_i), evaluated as a
  // log-sum-exp over the query rows: the same order as W_j, without the
  // underflow that would turn very small weights into ties.
  __shared__ float Ms[kMaxQR];
  const int u = blockIdx.y;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float2* pt = part + (int64_t)u * part_unit;
  for (int i = warp; i < q; i += 8) {
    float mx = -INFINITY;
    for (int t = lane; t < ntiles; t += 32) mx = fmaxf(mx, pt[(int64_t)t * q + i].x);
#pragma unroll
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float z = 0.f;
    for (int t = lane; t < ntiles; t += 32) {
      const float2 p = pt[(int64_t)t * q + i];
      z += p.y * expf(p.x - mx);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if (lane == 0) Ms[i] = mx + logf(z);
  }
  __syncthreads();
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= m) return;
  const float* lg = logits + (int64_t)u * lg_unit + j;
  float mx = -INFINITY;
#pragma unroll 8
  for (int i = 0; i < q; ++i) mx = fmaxf(mx, lg[(int64_t)i * lg_row] - Ms[i]);
  float z = 0.f;
#pragma unroll 8
  for (int i = 0; i < q; ++i) z += expf((lg[(int64_t)i * lg_row] - Ms[i]) - mx);
  W[(int64_t)u * w_unit + j] = mx + logf(z);
}

__device__ __forceinline__ uint32_t order_key(float f) {
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Exclusive block scan of a 0/1 flag over 1024 threads; returns the prefix
// and writes the block total.
__device__ __forceinline__ int block_scan_flag(bool flag, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned bal = __ballot_sync(0xffffffffu, flag);
  const int in_warp = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) warp_tot[warp] = __popc(bal);
  __syncthreads();
  if (warp == 0) {
    const int v = warp_tot[lane];
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    warp_tot[lane] = incl - v;
    if (lane == 31) *total = incl;
  }
  __syncthreads();
  const int r = warp_tot[warp] + in_warp;
  __syncthreads();
  return r;
}

// R > 0: the unit's keys stay in registers, R a thread (m <= 1024 R), read
// once for the four passes and the output; R == 0: read again every pass.
template <int R>
__global__ void __launch_bounds__(1024) select_kernel(const float* __restrict__ W, int64_t w_unit,
                                                      const int32_t* __restrict__ cand, int64_t cand_stride,
                                                      int m, int kk, int expand, int32_t* __restrict__ out,
                                                      int64_t out_stride, int32_t* __restrict__ sets,
                                                      int64_t sets_stride, int64_t sets_off) {
  __shared__ uint32_t hist[256];
  __shared__ uint32_t s_prefix, s_need;
  __shared__ int warp_tot[32];
  __shared__ int s_total;
  const int u = blockIdx.x;
  const int tid = threadIdx.x;
  const float* w = W + (int64_t)u * w_unit;
  uint32_t prefix = 0, mask = 0;
  uint32_t need = (uint32_t)kk;
  const int lane = tid & 31;
  const int nch = R > 0 ? R : (m + 1023) / 1024;  // 1024-key chunks
  uint32_t kr[R > 0 ? R : 1];
#pragma unroll
  for (int r = 0; r < (R > 0 ? R : 1); ++r) {
    const int j = r * 1024 + tid;
    kr[r] = (R > 0 && j < m) ? order_key(w[j]) : 0u;
  }
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    if (tid < 256) hist[tid] = 0;
    __syncthreads();
    // Keys crowd into few bins (sign and exponent bits first): the lanes of a
    // warp that share a bin add their count with one atomic.
#pragma unroll
    for (int r = 0; r < (R > 0 ? R : 64); ++r) {
      if (R == 0 && r >= nch) break;
      const int j = r * 1024 + tid;
      const uint32_t key = R > 0 ? kr[r] : (j < m ? order_key(w[j]) : 0u);
      const bool in = j < m && (key & mask) == prefix;
      const unsigned act = __ballot_sync(0xffffffffu, in);
      if (in) {
        const uint32_t bin = (key >> shift) & 255u;
        const unsigned peers = __match_any_sync(act, bin);
        if (lane == __ffs(peers) - 1) atomicAdd(&hist[bin], (uint32_t)__popc(peers));
      }
    }
    __syncthreads();
    if (tid < 32) {
      // Warp 0: bins high to low, eight per lane; the lane whose run reaches
      // `need` picks the bin.
      uint32_t c[8], run = 0;
#pragma unroll
      for (int b = 0; b < 8; ++b) {
        c[b] = hist[255 - (lane * 8 + b)];
        run += c[b];
      }
      uint32_t incl = run;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      uint32_t cum = incl - run;  // keys in higher bins than this lane's
      const bool mine = cum < need && incl >= need;
      if (mine) {
        int sel = 0;
#pragma unroll 1
        for (int b = 0; b < 8; ++b) {
          if (cum + c[b] >= need) { sel = 255 - (lane * 8 + b); break; }
          cum += c[b];
        }
        s_need = need - cum;
        s_prefix = prefix | ((uint32_t)sel << shift);
      }
    }
    __syncthreads();
    prefix = s_prefix;
    need = s_need;
    mask |= 255u << shift;
    __syncthreads();
  }
  // prefix = key of the kk-th largest W; take every larger key and the
  // `need` lowest-index keys equal to it.
  const int32_t* cd = cand ? cand + (int64_t)u * cand_stride : nullptr;
  int32_t* o = out + (int64_t)u * out_stride;
  int32_t* st = sets ? sets + (int64_t)u * sets_stride + sets_off : nullptr;
  int running = 0, eq_seen = 0;
#pragma unroll
  for (int r = 0; r < (R > 0 ? R : 64); ++r) {
    if (R == 0 && r >= nch) break;
    const int j = r * 1024 + tid;
    const uint32_t key = R > 0 ? kr[r] : (j < m ? order_key(w[j]) : 0u);
    const bool gt = j < m && key > prefix;
    const bool eq = j < m && key == prefix;
    const int eq_rank = block_scan_flag(eq, warp_tot, &s_total);
    const int eq_tot = s_total;
    const bool take = gt || (eq && (uint32_t)(eq_seen + eq_rank) < need);
    const int pos = block_scan_flag(take, warp_tot, &s_total);
    const int tot = s_total;
    if (take) {
      const int32_t c = cd ? cd[j] : j;
      const int p = running + pos;
      if (st) st[p] = c;
      if (expand) { o[2 * p] = 2 * c; o[2 * p + 1] = 2 * c + 1; }
      else o[p] = c;
    }
    running += tot;
    eq_seen += eq_tot;
    __syncthreads();
  }
}

// The Top-K launch: keys in registers up to 8192 candidates.
static void launch_select(int U, const float* W, int64_t w_unit, const int32_t* cand, int64_t cand_stride, int m,
                          int kk, int expand, int32_t* out, int64_t out_stride, int32_t* sets, int64_t sets_stride,
                          int64_t sets_off, cudaStream_t s) {
  const int nch = (m + 1023) / 1024;
#define WF_SELECT(R) select_kernel<R><<<U, 1024, 0, s>>>(W, w_unit, cand, cand_stride, m, kk, expand, out, out_stride, \
                                                         sets, sets_stride, sets_off)
  if (nch <= 1) WF_SELECT(1);
  else if (nch <= 2) WF_SELECT(2);
  else if (nch <= 4) WF_SELECT(4);
  else if (nch <= 8) WF_SELECT(8);
  else WF_SELECT(0);
#undef WF_SELECT
}

template <typename T, int D, int QM>
cudaError_t run_score_q(const FilterPlan& p, const void* Q, const wf_tensor& qd, RowSrc src, const int32_t* cand,
                        int m, float* logits, float2* part, cudaStream_t s) {
  const size_t smem = sizeof(float) * (size_t)(QM * D + TILE * (D + 4));
  cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(score_kernel<T, D, QM>), smem);
  if (e != cudaSuccess) return e;
  dim3 grid((m + TILE - 1) / TILE, p.U, (p.q + QM - 1) / QM);
  score_kernel<T, D, QM><<<grid, 256, smem, s>>>(static_cast<const T*>(Q), qd.stride_b, qd.stride_h, qd.stride_s, p.q,
                                             p.G, p.qs, p.H, src, cand, p.cmax, m, 1.0f / sqrtf((float)D), logits,
                                             (int64_t)p.q * p.cmax, p.cmax, part, (int64_t)p.tiles_max * p.q);
  return cudaGetLastError();
}

// Query blocks of up to 32 rows take the 32-row tile; larger ones 64-row chunks.
template <typename T, int D>
cudaError_t run_score(const FilterPlan& p, const void* Q, const wf_tensor& qd, RowSrc src, const int32_t* cand,
                      int m, float* logits, float2* part, cudaStream_t s) {
  return p.q <= 32 ? run_score_q<T, D, 32>(p, Q, qd, src, cand, m, logits, part, s)
                   : run_score_q<T, D, QMAX>(p, Q, qd, src, cand, m, logits, part, s);
}

cudaError_t score(const FilterPlan& p, const void* Q, const wf_tensor& qd, RowSrc src, const int32_t* cand, int m,
                  float* logits, float2* part, cudaStream_t s) {
  if (p.dtype == WF_BF16) {
    return p.d == 64 ? run_score<bf16, 64>(p, Q, qd, src, cand, m, logits, part, s)
                     : run_score<bf16, 128>(p, Q, qd, src, cand, m, logits, part, s);
  }
  return p.d == 64 ? run_score<float, 64>(p, Q, qd, src, cand, m, logits, part, s)
                   : run_score<float, 128>(p, Q, qd, src, cand, m, logits, part, s);
}

}  // namespace

FilterPlan plan_filter(const wf_tensor& q, const wf_tensor& kv, int levels, const int32_t* keep) {
  FilterPlan p{};
  p.U = kv.batch * kv.heads;
  p.H = kv.heads;
  p.G = q.heads / kv.heads;
  p.qs = q.seq;
  p.q = p.G * q.seq;
  p.d = kv.head_dim;
  p.n = kv.seq;
  p.L = levels;
  p.dtype = kv.dtype;
  for (int l = 0; l <= levels; ++l) p.keep[l] = keep[l];
  int cmax = kv.seq >> levels;
  for (int l = 1; l <= levels; ++l) cmax = cmax > 2 * keep[l] ? cmax : 2 * keep[l];
  p.cmax = cmax;
  p.tiles_max = (cmax + TILE - 1) / TILE;
  p.trim = keep[0] < 2 * keep[1];
  const size_t U = (size_t)p.U;
  size_t off = 256;  // status block
  p.off_cand_a = off; off = align_up(off + U * cmax * sizeof(int32_t), 256);
  p.off_cand_b = off; off = align_up(off + U * cmax * sizeof(int32_t), 256);
  p.off_w = off;      off = align_up(off + U * cmax * sizeof(float), 256);
  p.off_logits = off; off = align_up(off + U * (size_t)p.q * cmax * sizeof(float), 256);
  p.off_part = off;   off = align_up(off + U * (size_t)p.tiles_max * p.q * sizeof(float2), 256);
  p.total = off;
  return p;
}

namespace {
// Eq. 7-8 for one scale: the ranking key of each of the m candidates into W
// (tensor cores where they apply, else the fp32 score and weights kernels).
cudaError_t skim(const FilterPlan& p, const void* Q, const wf_tensor& qd, RowSrc src, const int32_t* cand, int m,
                 float* logits, float2* part, float* W, int* status, cudaStream_t s) {
  // The fp32 logits buffer is not used by the tensor-core skim: its first
  // U q floats hold the normalisers between the two passes.
  if (tc_skim_supported(p)) return launch_tc_skim(p, Q, qd, src, cand, m, part, W, logits, status, s);
  cudaError_t e;
  if ((e = score(p, Q, qd, src, cand, m, logits, part, s)) != cudaSuccess) return e;
  const int ntiles = (m + TILE - 1) / TILE;
  weights_kernel<<<dim3((m + 255) / 256, p.U), 256, 0, s>>>(logits, (int64_t)p.q * p.cmax, p.cmax, part,
                                                            (int64_t)p.tiles_max * p.q, ntiles, p.q, m, W, p.cmax);
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_filter(const FilterPlan& p, const void* Q, const wf_tensor& qd, const void* coeffs,
                          const void* K, const wf_tensor& kv, int32_t* idx, int32_t* level_sets, void* ws,
                          int* status, cudaStream_t s) {
  char* base = static_cast<char*>(ws);
  int32_t* cand_cur = reinterpret_cast<int32_t*>(base + p.off_cand_a);
  int32_t* cand_nxt = reinterpret_cast<int32_t*>(base + p.off_cand_b);
  float* W = reinterpret_cast<float*>(base + p.off_w);
  float* logits = reinterpret_cast<float*>(base + p.off_logits);
  float2* part = reinterpret_cast<float2*>(base + p.off_part);
  const int64_t esz = p.dtype == WF_BF16 ? 2 : 4;
  (void)esz;
  const int64_t rows_total = (int64_t)p.n - ((int64_t)p.n >> p.L);
  int64_t sets_stride = 0;
  for (int l = 0; l <= p.L; ++l) sets_stride += p.keep[l];
  int64_t sets_off = 0;
  bool first = true;
  int m = p.n >> p.L;
  cudaError_t e;
  for (int l = p.L; l >= 1; --l) {
    RowSrc src;
    src.base = coeffs;
    src.sh = rows_total * p.d;
    src.sb = src.sh * p.H;
    src.ss = p.d;
    src.off = ((int64_t)p.n - ((int64_t)p.n >> (l - 1))) * p.d;
    const int32_t* cand = first ? nullptr : cand_cur;
    if ((e = skim(p, Q, qd, src, cand, m, logits, part, W, status, s)) != cudaSuccess) return e;
    const bool last = (l == 1) && !p.trim;
    int32_t* out = last ? idx : cand_nxt;
    const int64_t out_stride = last ? p.keep[0] : p.cmax;
    launch_select(p.U, W, p.cmax, cand, p.cmax, m, p.keep[l], 1, out, out_stride, level_sets,
                                       sets_stride, sets_off, s);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    sets_off += p.keep[l];
    m = 2 * p.keep[l];
    int32_t* t = cand_cur; cand_cur = cand_nxt; cand_nxt = t;
    first = false;
  }
  if (p.trim) {
    RowSrc src;
    src.base = K;
    src.sb = kv.stride_b;
    src.sh = kv.stride_h;
    src.ss = kv.stride_s;
    src.off = 0;
    if ((e = skim(p, Q, qd, src, cand_cur, m, logits, part, W, status, s)) != cudaSuccess) return e;
    launch_select(p.U, W, p.cmax, cand_cur, p.cmax, m, p.keep[0], 0, idx, p.keep[0], nullptr, 0, 0, s);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (level_sets) {
    // mu^0 follows J_1 in the level-set record.
    e = cudaMemcpy2DAsync(level_sets + sets_off, sizeof(int32_t) * sets_stride, idx, sizeof(int32_t) * p.keep[0],
                          sizeof(int32_t) * p.keep[0], p.U, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

size_t wavelet_filter_bytes(const FilterPlan& p) {
  const size_t esz = p.dtype == WF_BF16 ? 2 : 4;
  return align_up(p.total, 256) + (size_t)p.U * p.cmax * p.d * esz;
}

cudaError_t launch_filter_wavelet(const FilterPlan& p, const void* Q, const wf_tensor& qd, const void* top,
                                  const void* K, const wf_tensor& kv, int wavelet, int32_t* idx, int32_t* level_sets,
                                  void* ws, int* status, cudaStream_t s) {
  // The same scan as launch_filter, except that the rows of scale l < L are
  // the approximation rows of the transform of the candidates' gathered
  // blocks (computed here, in candidate order) instead of pyramid rows.
  char* base = static_cast<char*>(ws);
  int32_t* cand_cur = reinterpret_cast<int32_t*>(base + p.off_cand_a);
  int32_t* cand_nxt = reinterpret_cast<int32_t*>(base + p.off_cand_b);
  float* W = reinterpret_cast<float*>(base + p.off_w);
  float* logits = reinterpret_cast<float*>(base + p.off_logits);
  float2* part = reinterpret_cast<float2*>(base + p.off_part);
  void* arows = base + align_up(p.total, 256);
  int64_t sets_stride = 0;
  for (int l = 0; l <= p.L; ++l) sets_stride += p.keep[l];
  int64_t sets_off = 0;
  int m = p.n >> p.L;
  cudaError_t e;
  for (int l = p.L; l >= 1; --l) {
    RowSrc src;
    src.off = 0;
    src.ss = p.d;
    if (l == p.L) {
      src.base = top;  // the whole prompt's level-L rows (Eq. 6), [units][m][d]
      src.sh = (int64_t)m * p.d;
    } else {
      if ((e = launch_wavelet_approx(K, kv, cand_cur, p.cmax, m, l, wavelet, arows, (int64_t)p.cmax * p.d, s)) !=
          cudaSuccess)
        return e;
      src.base = arows;
      src.sh = (int64_t)p.cmax * p.d;
    }
    src.sb = src.sh * p.H;
    if ((e = skim(p, Q, qd, src, nullptr, m, logits, part, W, status, s)) != cudaSuccess) return e;
    const bool last = (l == 1) && !p.trim;
    int32_t* out = last ? idx : cand_nxt;
    const int64_t out_stride = last ? p.keep[0] : p.cmax;
    const int32_t* cand = l == p.L ? nullptr : cand_cur;  // position -> block index at scale l
    launch_select(p.U, W, p.cmax, cand, p.cmax, m, p.keep[l], 1, out, out_stride, level_sets,
                                       sets_stride, sets_off, s);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    sets_off += p.keep[l];
    m = 2 * p.keep[l];
    int32_t* t = cand_cur; cand_cur = cand_nxt; cand_nxt = t;
  }
  if (p.trim) {
    RowSrc src;
    src.base = K;
    src.sb = kv.stride_b;
    src.sh = kv.stride_h;
    src.ss = kv.stride_s;
    src.off = 0;
    if ((e = skim(p, Q, qd, src, cand_cur, m, logits, part, W, status, s)) != cudaSuccess) return e;
    launch_select(p.U, W, p.cmax, cand_cur, p.cmax, m, p.keep[0], 0, idx, p.keep[0], nullptr, 0, 0, s);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (level_sets) {
    e = cudaMemcpy2DAsync(level_sets + sets_off, sizeof(int32_t) * sets_stride, idx, sizeof(int32_t) * p.keep[0],
                          sizeof(int32_t) * p.keep[0], p.U, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace wf
