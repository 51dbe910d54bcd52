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
// there in fp32.  A thread owns one 16-byte vector of channels (8 for bf16,
// 4 for fp32) and a run of consecutive outputs of each level: it slides its
// filter window two rows per output, so an input row is one 16-byte load
// (plus the widening of its bf16 lanes), and every output is taps packed
// multiply-adds a channel pair.  Intermediate levels stay in shared memory as
// fp32 in 16-byte planes (conflict-free loads); the last level goes from
// registers to global memory.  Arithmetic, the storage rule: Haar:
// fl32(x0 + x1) * fl32(1 / sqrt 2), as the stored pyramid; db2:
// fl32(fl32(h[0]) x0), then fused multiply-adds with fl32(h[1..3]) in order.
// The packed fp32 instructions round each lane as the scalar ones do.  Only
// the last level is rounded to the key dtype.
#include <math.h>

#include <map>
#include <mutex>

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

// A vector of VEC channels as VEC / 2 packed fp32 pairs.
template <typename T>
struct Lanes {
  static constexpr int VEC = Vec<T>::N;
  f32x2 v[VEC / 2];
};

// Widen one 16-byte vector of T (as loaded) to fp32 pairs (exact).
__device__ __forceinline__ void widen(const uint4& w, Lanes<bf16>& o) {
  const uint32_t a[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) o.v[i] = pk2(__uint_as_float(a[i] << 16), __uint_as_float(a[i] & 0xffff0000u));
}
__device__ __forceinline__ void widen(const uint4& w, Lanes<float>& o) {
  o.v[0] = pk2(__uint_as_float(w.x), __uint_as_float(w.y));
  o.v[1] = pk2(__uint_as_float(w.z), __uint_as_float(w.w));
}
// Round to T and pack one 16-byte vector.
__device__ __forceinline__ uint4 narrow(const Lanes<bf16>& x) {
  uint32_t w[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = up2(x.v[i]);
    w[i] = pack_bf16(f.x, f.y);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}
__device__ __forceinline__ uint4 narrow(const Lanes<float>& x) {
  const float2 a = up2(x.v[0]), b = up2(x.v[1]);
  return make_uint4(__float_as_uint(a.x), __float_as_uint(a.y), __float_as_uint(b.x), __float_as_uint(b.y));
}

// Outputs of one unrolled pass of the cascade (longer runs take several
// passes, each reloading the window's first taps - 2 rows).
constexpr int PMAX = 2;

// One level of the cascade for this thread's channel vector vt and its run
// of outputs [jb, jb + cnt), cnt <= PMAX: out[j] = sum_k h[k] in[2 j + k].
// RAW: the input is the gathered rows (T, row-major DS channels); else fp32
// rows in 16-byte planes (plane p of vector vt at byte p * 16 VT + 16 vt of
// the row).  LAST: outputs go to global memory rounded to T (rows below
// `valid` only); else to the fp32 rows at dst.  The run is unrolled, so the
// sliding window lives in renamed registers.
template <typename T, int TAPS, int DS, bool RAW>
__device__ __forceinline__ void cascade_level(const uint8_t* src, uint8_t* dst, int jb, int cnt, int vt, bool last,
                                              int valid, T* ob, int64_t out_row, const f32x2 (&h2)[4], f32x2 c2) {
  constexpr int VEC = Vec<T>::N, VT = DS / VEC, NP = VEC / 4;
  constexpr int IN_ROW = RAW ? DS * (int)sizeof(T) : DS * 4;  // bytes per input row
  const uint8_t* sp = src + (2 * jb) * IN_ROW + 16 * vt;
  auto load = [&](int row, Lanes<T>& o) {
    if (RAW) {
      widen(*reinterpret_cast<const uint4*>(sp + row * IN_ROW), o);
    } else {
#pragma unroll
      for (int p = 0; p < NP; ++p) {
        const ulonglong2 q = *reinterpret_cast<const ulonglong2*>(sp + row * IN_ROW + p * 16 * VT);
        o.v[2 * p] = q.x;
        o.v[2 * p + 1] = q.y;
      }
    }
  };
  Lanes<T> x[2 * PMAX + TAPS - 2];  // rows 2 jb + i of the run's window
#pragma unroll
  for (int i = 0; i < TAPS - 2; ++i) load(i, x[i]);
#pragma unroll
  for (int t = 0; t < PMAX; ++t) {
    if (t < cnt) {
      load(2 * t + TAPS - 2, x[2 * t + TAPS - 2]);
      load(2 * t + TAPS - 1, x[2 * t + TAPS - 1]);
      Lanes<T> y;
#pragma unroll
      for (int i = 0; i < VEC / 2; ++i) {
        if (TAPS == 2) {
          y.v[i] = mul2(add2(x[2 * t].v[i], x[2 * t + 1].v[i]), c2);
        } else {
          f32x2 a = mul2(h2[0], x[2 * t].v[i]);
#pragma unroll
          for (int k = 1; k < TAPS; ++k) a = fma2(h2[k], x[2 * t + k].v[i], a);
          y.v[i] = a;
        }
      }
      const int j = jb + t;
      if (last) {
        if (j < valid) *reinterpret_cast<uint4*>(ob + (int64_t)j * out_row + vt * VEC) = narrow(y);
      } else {
#pragma unroll
        for (int p = 0; p < NP; ++p)
          *reinterpret_cast<ulonglong2*>(dst + j * DS * 4 + p * 16 * VT + 16 * vt) =
              make_ulonglong2(y.v[2 * p], y.v[2 * p + 1]);
      }
    }
  }
}

// Quotient and remainder by an invariant divisor with a multiply and a shift
// (Granlund and Montgomery, "Division by invariant integers using
// multiplication", 1994): for 0 <= x < 2^31 and d >= 1, with
// l = ceil(log2 d) and mul = floor(2^32 (2^l - d) / d) + 1,
// x / d = (umulhi(mul, x) + x) >> l.
struct FastDiv {
  uint32_t d, mul, shift;
};
inline FastDiv make_fastdiv(uint32_t d) {
  FastDiv f;
  f.d = d;
  uint32_t l = 0;
  while ((1ull << l) < d) ++l;
  f.shift = l;
  f.mul = (uint32_t)((((1ull << l) - d) << 32) / d + 1);
  return f;
}
__device__ __forceinline__ uint32_t fastdiv(uint32_t x, const FastDiv& f) {
  return (__umulhi(f.mul, x) + x) >> f.shift;
}

// Shared memory: the gathered rows as loaded (T), then the fp32 levels
// alternating between a second buffer and the first one (which holds at
// least as many fp32 rows as the level after the first needs), then the
// gathered rows' token indices.
template <typename T, int TAPS, int DS>
__global__ void __launch_bounds__(NTH, 3) approx_kernel(const T* __restrict__ K, int64_t ksb, int64_t ksh, int64_t kss,
                                                     int64_t n, FastDiv heads, const int32_t* __restrict__ cand,
                                                     int64_t cand_stride, int m, int level, Taps taps,
                                                     T* __restrict__ out, int64_t out_unit, int64_t out_row) {
  extern __shared__ __align__(16) uint8_t sbuf[];
  constexpr int VEC = Vec<T>::N;
  constexpr int VT = DS / VEC;   // vector threads across a row
  constexpr int RT = NTH / VT;   // run threads
  static_assert(NTH % VT == 0 && (VT & (VT - 1)) == 0, "a row's vectors split evenly");
  const int to = outputs_per_cta(level);
  const int nin = rows_needed(to, level, TAPS);
  uint8_t* X = sbuf;                                                             // raw rows, later fp32 levels
  uint8_t* Y = sbuf + ((size_t)nin * DS * sizeof(T) + 15) / 16 * 16;             // fp32 levels 1, 3, ...
  int* tok = reinterpret_cast<int*>(Y + (size_t)(nin / 2 + 1) * DS * 4);         // token of each gathered row
  // The channel slice varies fastest, so the slices of the same rows are read
  // by neighbouring CTAs at about the same time.
  const int u = blockIdx.z;
  const int j0 = blockIdx.y * to;
  const int c0 = blockIdx.x * DS;
  const uint32_t bb = fastdiv((uint32_t)u, heads), hh = (uint32_t)u - bb * heads.d;
  const int len = m << level;  // the gathered sequence (< 2^31 tokens)
  const int blk_mask = (1 << level) - 1;
  const int32_t* cd = cand ? cand + (int64_t)u * cand_stride : nullptr;
  const int tid = threadIdx.x;
  grid_dep_wait();  // the candidates (and the output's previous readers) come from the grids before
  grid_dep_launch();

  // Row r is gathered position (j0 2^b + r) mod len: its token first, then
  // 16-byte copies, VT a row.
  const int base = j0 << level;  // j0 < m, so base < len
  for (int r = tid; r < nin; r += NTH) {
    int p = base + r;
    if (p >= len) p = p - len < len ? p - len : p % len;  // the filter's reach wraps around
    int64_t tl = cd ? ((int64_t)cd[p >> level] << level) + (p & blk_mask) : p;
    tok[r] = (int)(tl < 0 ? 0 : (tl >= n ? n - 1 : tl));  // out-of-range block indices are clamped
  }
  __syncthreads();
  {
    const T* src = K + (int64_t)bb * ksb + (int64_t)hh * ksh + c0 + (tid % VT) * VEC;
    const uint32_t xs = (uint32_t)__cvta_generic_to_shared(X) + (uint32_t)((tid % VT) * VEC * sizeof(T));
#pragma unroll 4
    for (int r = tid / VT; r < nin; r += RT)
      cp_async16(xs + (uint32_t)(r * DS * sizeof(T)), src + (int64_t)tok[r] * kss);
  }
  cp_async_wait_all();
  __syncthreads();

  const float c32 = 0.70710678118654752440f;  // fl32(1 / sqrt 2)
  const f32x2 c2 = pk2(c32, c32);
  f32x2 h2[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) h2[k] = pk2(taps.h[k], taps.h[k]);
  const int vt = tid % VT, rt = tid / VT;
  // The last level's outputs are rows j0 .. j0 + to - 1, those below m written.
  T* obl = out + (int64_t)u * out_unit + c0 + (int64_t)j0 * out_row;
  const int valid = m - j0;
#pragma unroll 1
  for (int l = 1; l <= level; ++l) {
    const int nout = rows_needed(to, level - l, TAPS);
    const bool last = l == level;
    uint8_t* dst = (l & 1) ? Y : X;
    const int per = (nout + RT - 1) / RT;
    const int je = min(nout, (rt + 1) * per);
#pragma unroll 1
    for (int jb = rt * per; jb < je; jb += PMAX) {
      const int cnt = min(je - jb, PMAX);
      if (l == 1)
        cascade_level<T, TAPS, DS, true>(X, dst, jb, cnt, vt, last, valid, obl, out_row, h2, c2);
      else
        cascade_level<T, TAPS, DS, false>((l & 1) ? X : Y, dst, jb, cnt, vt, last, valid, obl, out_row, h2, c2);
    }
    __syncthreads();
  }
}

// Shared memory of one CTA for DS channels: the raw rows, the first fp32
// level (the raw buffer holds the later ones) and the row tokens.
template <typename T, int TAPS>
size_t approx_smem(int level, int ds) {
  const int nin = rows_needed(outputs_per_cta(level), level, TAPS);
  return ((size_t)nin * ds * sizeof(T) + 15) / 16 * 16 + sizeof(float) * ds * (size_t)(nin / 2 + 1) +
         sizeof(int) * (size_t)nin;
}

template <typename T, int TAPS, int DS>
cudaError_t run_ds(const void* K, const wf_tensor& kv, const int32_t* cand, int64_t cand_stride, int m, int level,
                   const Taps& taps, void* out, int64_t out_unit, cudaStream_t s, bool pdl) {
  const int to = outputs_per_cta(level);
  const size_t smem = approx_smem<T, TAPS>(level, DS);
  // The shared-memory limit, raised per device to the largest size requested
  // so far (not on every launch).
  static std::mutex mu;
  static std::map<int, size_t> raised;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  {
    std::lock_guard<std::mutex> lock(mu);
    size_t& cur = raised[dev];
    if (cur < smem) {
      e = cudaFuncSetAttribute(approx_kernel<T, TAPS, DS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
      cur = smem;
    }
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(kv.head_dim / DS), (unsigned)((m + to - 1) / to), (unsigned)(kv.batch * kv.heads));
  cfg.blockDim = dim3(NTH, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  e = cudaLaunchKernelEx(&cfg, approx_kernel<T, TAPS, DS>, static_cast<const T*>(K), kv.stride_b, kv.stride_h,
                         kv.stride_s, (int64_t)kv.seq, make_fastdiv((uint32_t)kv.heads), cand, cand_stride, m, level,
                         taps, static_cast<T*>(out), out_unit, (int64_t)kv.head_dim);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Whole rows of 128 channels per CTA (each row's token resolved once, 256-byte
// copies of bf16) while the shared memory allows, else 64 channels, else 16
// (the deepest scales).  Measured at 32K (bf16, db2, three scales a step):
// whole rows 265 us a step against 301 with 64 channels.
template <typename T, int TAPS>
cudaError_t run(const void* K, const wf_tensor& kv, const int32_t* cand, int64_t cand_stride, int m, int level,
                const Taps& taps, void* out, int64_t out_unit, cudaStream_t s, bool pdl) {
  if (kv.head_dim == 128 && approx_smem<T, TAPS>(level, 128) <= 200 * 1024)
    return run_ds<T, TAPS, 128>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s, pdl);
  if (approx_smem<T, TAPS>(level, 64) <= 200 * 1024)
    return run_ds<T, TAPS, 64>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s, pdl);
  return run_ds<T, TAPS, 16>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s, pdl);
}

}  // namespace

int wavelet_taps(int wavelet) { return wavelet == WF_WAVELET_HAAR ? 2 : (wavelet == WF_WAVELET_DB2 ? 4 : 0); }

int wavelet_max_level(int wavelet) { return wavelet == WF_WAVELET_DB2 ? 8 : 10; }

cudaError_t launch_wavelet_approx(const void* K, const wf_tensor& kv, const int32_t* cand, int64_t cand_stride, int m,
                                  int level, int wavelet, void* out, int64_t out_unit, cudaStream_t s, bool pdl) {
  Taps taps{};
  if (wavelet == WF_WAVELET_DB2) {
    // Daubechies' two-vanishing-moment scaling filter, from its closed form.
    const double r = sqrt(3.0), q = 4.0 * sqrt(2.0);
    const double h[4] = {(1.0 + r) / q, (3.0 + r) / q, (3.0 - r) / q, (1.0 - r) / q};
    for (int k = 0; k < 4; ++k) taps.h[k] = (float)h[k];
    return kv.dtype == WF_BF16 ? run<bf16, 4>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s, pdl)
                               : run<float, 4>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s, pdl);
  }
  return kv.dtype == WF_BF16 ? run<bf16, 2>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s, pdl)
                             : run<float, 2>(K, kv, cand, cand_stride, m, level, taps, out, out_unit, s, pdl);
}

}  // namespace wf
