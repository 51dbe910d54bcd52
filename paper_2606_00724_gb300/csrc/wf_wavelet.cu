// Approximation rows of the periodized DWT of a gathered key sub-sequence
// (Eq. 6 for the whole prompt, Eq. 11 for the blocks of the candidates kept
// one scale up), for the Haar and db2 filter banks.
//
// The sequence of a unit is the keys of blocks [2^b c, 2^b (c + 1)) for the
// unit's candidates c, in candidate order, taken as periodic.  One level of
// analysis is a[j] = sum_k h[k] x[(2j + k) mod len]; b levels give one
// approximation row per candidate.
//
// One CTA computes TO consecutive level-b rows for DS head-dim channels: it
// gathers the TO 2^b input rows plus the (taps - 2)(2^b - 1) rows the filter
// reaches past them (wrapping around the gathered sequence) into shared
// memory with 16-byte cp.async copies, and runs the b levels of the cascade
// there in fp32 (two buffers alternating; a thread slides its filter window
// over a run of outputs for a channel pair).  Arithmetic, the storage rule:
// Haar: fl32(x0 + x1) * fl32(1 / sqrt 2), as the stored pyramid; db2:
// fl32(fl32(h[0]) x0), then fused multiply-adds with fl32(h[1..3]) in order.
// A channel pair goes through the packed fp32 instructions, which round each
// lane as the scalar ones do.  Only the last level is rounded to the key
// dtype.
#include <math.h>

#include "wf_internal.cuh"
#include "wf_sm100.cuh"

namespace wf {
namespace {

using namespace sm100;

constexpr int NTH = 256;      // threads per CTA
constexpr int IN_ROWS = 128;  // gathered rows per CTA before the filter's reach

// Output rows per CTA at scale `level`.
__host__ __device__ inline int outputs_per_cta(int level) { return (IN_ROWS >> level) > 0 ? (IN_ROWS >> level) : 1; }

// Rows needed l levels below the output so that the output level yields `to`
// rows: to 2^l + (taps - 2)(2^l - 1).
__host__ __device__ inline int rows_needed(int to, int l, int taps) { return (to << l) + (taps - 2) * ((1 << l) - 1); }

struct Taps {
  float h[4];
};

template <typename T>
__device__ __forceinline__ float rd(const T* p) { return to_f32(*p); }

// Shared memory: the gathered rows as loaded (T), then the fp32 levels
// alternating between a second buffer and the first one (which holds at
// least as many fp32 rows as the level after the first needs).
template <typename T, int TAPS, int DS>
__global__ void __launch_bounds__(NTH) approx_kernel(const T* __restrict__ K, int64_t ksb, int64_t ksh, int64_t kss,
                                                     int64_t n, int H, const int32_t* __restrict__ cand,
                                                     int64_t cand_stride, int m, int level, Taps taps,
                                                     T* __restrict__ out, int64_t out_unit, int64_t out_row) {
  extern __shared__ __align__(16) uint8_t sbuf[];
  const int to = outputs_per_cta(level);
  const int nin = rows_needed(to, level, TAPS);
  T* X0 = reinterpret_cast<T*>(sbuf);                                    // [nin][DS] raw
  float* Y = reinterpret_cast<float*>(sbuf + (size_t)nin * DS * sizeof(T));  // [nin / 2 + 1][DS]
  float* X = reinterpret_cast<float*>(sbuf);                             // fp32 levels >= 2
  // The channel slice varies fastest, so the slices of the same rows are read
  // by neighbouring CTAs at about the same time.
  const int u = blockIdx.z;
  const int j0 = blockIdx.y * to;
  const int c0 = blockIdx.x * DS;
  const int64_t bb = u / H, hh = u % H;
  const int len = m << level;  // the gathered sequence (< 2^31 tokens)
  const int blk_mask = (1 << level) - 1;
  const T* kb_src = K + bb * ksb + hh * ksh + c0;
  const int32_t* cd = cand ? cand + (int64_t)u * cand_stride : nullptr;
  const int tid = threadIdx.x;

  // Gather: row r is gathered position (j0 2^b + r) mod len, 16-byte copies.
  constexpr int VEC = Vec<T>::N;
  constexpr int VPR = DS / VEC;  // 16-byte vectors per row
  const uint32_t xs = (uint32_t)__cvta_generic_to_shared(X0);
  const int base = (int)(((int64_t)j0 << level) % len);
  // Copy e = tid + NTH k is vector v = tid % VPR of row tid / VPR + (NTH / VPR) k.
  // The VPR lanes of a row share its token: in each batch of VPR copies,
  // lane v resolves the row of copy kb + v and its group reads them by shuffle.
  static_assert(32 % VPR == 0 && NTH % VPR == 0, "a row's lanes sit in one warp");
  const int v = tid % VPR, r0 = tid / VPR, gbase = (tid & 31) & ~(VPR - 1);
  const int iters = (nin * VPR - tid + NTH - 1) / NTH;  // this thread's copies
  const int iters_w = (nin * VPR - (tid & ~31) + NTH - 1) / NTH;  // the most of any lane in the warp
#pragma unroll 1
  for (int kb = 0; kb < iters_w; kb += VPR) {
    int p = base + r0 + (NTH / VPR) * (kb + v);
    p = p < len ? p : (p - len < len ? p - len : p % len);  // the filter's reach wraps around
    int64_t tl = cd ? (((int64_t)cd[p >> level]) << level) + (p & blk_mask) : p;
    tl = tl < 0 ? 0 : (tl >= n ? n - 1 : tl);  // out-of-range block indices are clamped
#pragma unroll
    for (int k = 0; k < VPR; ++k) {
      const int64_t tok = __shfl_sync(0xffffffffu, tl, gbase | k);
      const int it = kb + k, r = r0 + (NTH / VPR) * it;
      if (it < iters)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(xs + (uint32_t)((r * DS + v * VEC) * sizeof(T))),
                     "l"(kb_src + tok * kss + v * VEC)
                     : "memory");
    }
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();

  // The cascade: a thread owns a channel pair and a run of consecutive
  // outputs, sliding its filter window two rows per output (each output is
  // the same fp32 sequence of products and sums).
  const float c32 = 0.70710678118654752440f;  // fl32(1 / sqrt 2)
  const f32x2 c2 = pk2(c32, c32);
  f32x2 h2[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) h2[k] = pk2(taps.h[k], taps.h[k]);
  constexpr int PAIRS = DS / 2;
  constexpr int GROUPS = NTH / PAIRS;
  const int cp = tid % PAIRS, grp = tid / PAIRS;
#pragma unroll 1
  for (int l = 1; l <= level; ++l) {
    const int nout = rows_needed(to, level - l, TAPS);
    float* dst = (l & 1) ? Y : X;
    const float* src = (l & 1) ? X : Y;  // fp32 input of levels >= 2
    const int per = (nout + GROUPS - 1) / GROUPS;
    const int jb = grp * per, je = min(nout, jb + per);
    auto in = [&](int row) -> f32x2 {
      if (l == 1) {
        const T* p = X0 + row * DS + 2 * cp;
        return pk2(rd(p), rd(p + 1));
      }
      return *reinterpret_cast<const f32x2*>(src + row * DS + 2 * cp);
    };
    if (jb < je) {
      f32x2 x[TAPS];
#pragma unroll
      for (int k = 0; k < TAPS - 2; ++k) x[k + 2] = in(2 * jb + k);
#pragma unroll 1
      for (int j = jb; j < je; ++j) {
#pragma unroll
        for (int k = 0; k < TAPS - 2; ++k) x[k] = x[k + 2];
        x[TAPS - 2] = in(2 * j + TAPS - 2);
        x[TAPS - 1] = in(2 * j + TAPS - 1);
        f32x2 v;
        if (TAPS == 2) {
          v = mul2(add2(x[0], x[1]), c2);
        } else {
          v = mul2(h2[0], x[0]);
#pragma unroll
          for (int k = 1; k < TAPS; ++k) v = fma2(h2[k], x[k], v);
        }
        *reinterpret_cast<f32x2*>(dst + j * DS + 2 * cp) = v;
      }
    }
    __syncthreads();
  }

  // The last level: rows j0 .. j0 + to - 1 (those below m), rounded to T.
  const float* fin = (level & 1) ? Y : X;
  T* ob = out + (int64_t)u * out_unit + c0;
  for (int e = tid; e < to * DS; e += NTH) {
    const int j = e / DS, c = e % DS;
    if (j0 + j < m) from_f32(ob[(int64_t)(j0 + j) * out_row + c], fin[j * DS + c]);
  }
}

// Shared memory of one CTA for DS channels: the raw rows, then the first
// fp32 level (the raw buffer holds the later ones).
template <typename T, int TAPS>
size_t approx_smem(int level, int ds) {
  const int nin = rows_needed(outputs_per_cta(level), level, TAPS);
  return (size_t)nin * ds * sizeof(T) + sizeof(float) * ds * (size_t)(nin / 2 + 1);
}

template <typename T, int TAPS, int DS>
cudaError_t run_ds(const void* K, const wf_tensor& kv, const int32_t* cand, int64_t cand_stride, int m, int level,
                   const Taps& taps, void* out, int64_t out_unit, cudaStream_t s) {
  const int to = outputs_per_cta(level);
  const size_t smem = approx_smem<T, TAPS>(level, DS);
  cudaError_t e =
      cudaFuncSetAttribute(approx_kernel<T, TAPS, DS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const dim3 grid((unsigned)(kv.head_dim / DS), (unsigned)((m + to - 1) / to), (unsigned)(kv.batch * kv.heads));
  approx_kernel<T, TAPS, DS><<<grid, NTH, smem, s>>>(static_cast<const T*>(K), kv.stride_b, kv.stride_h,
                                                     kv.stride_s, kv.seq, kv.heads, cand, cand_stride, m, level, taps,
                                                     static_cast<T*>(out), out_unit, kv.head_dim);
  return cudaGetLastError();
}

// 64 channels per CTA (whole 128-byte lines of bf16) while the shared memory
// allows, else 16 (the deepest scales).
template <typename T, int TAPS>
cudaError_t run(const void* K, const wf_tensor& kv, const int32_t* cand, int64_t cand_stride, int m, int level,
                const Taps& taps, void* out, int64_t out_unit, cudaStream_t s) {
  if (approx_smem<T, TAPS>(level, 64) <= 200 * 1024)
    return run_ds<T, TAPS, 64>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s);
  return run_ds<T, TAPS, 16>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s);
}

}  // namespace

int wavelet_taps(int wavelet) { return wavelet == WF_WAVELET_HAAR ? 2 : (wavelet == WF_WAVELET_DB2 ? 4 : 0); }

int wavelet_max_level(int wavelet) { return wavelet == WF_WAVELET_DB2 ? 8 : 10; }

cudaError_t launch_wavelet_approx(const void* K, const wf_tensor& kv, const int32_t* cand, int64_t cand_stride, int m,
                                  int level, int wavelet, void* out, int64_t out_unit, cudaStream_t s) {
  Taps taps{};
  if (wavelet == WF_WAVELET_DB2) {
    // Daubechies' two-vanishing-moment scaling filter, from its closed form.
    const double r = sqrt(3.0), q = 4.0 * sqrt(2.0);
    const double h[4] = {(1.0 + r) / q, (3.0 + r) / q, (3.0 - r) / q, (1.0 - r) / q};
    for (int k = 0; k < 4; ++k) taps.h[k] = (float)h[k];
    return kv.dtype == WF_BF16 ? run<bf16, 4>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s)
                               : run<float, 4>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s);
  }
  return kv.dtype == WF_BF16 ? run<bf16, 2>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s)
                             : run<float, 2>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s);
}

}  // namespace wf
