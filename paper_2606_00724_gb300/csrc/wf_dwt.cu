// Multi-level Haar DWT of the cached keys (Eq. 5 recursion, Eq. 6).
//
// One thread owns one 16-byte column slice (4 fp32 / 8 bf16 channels) of one
// aligned block of 2^L tokens.  It streams the block in chunks of 2^LC tokens
// (LC = min(L, 3)): a chunk's levels 1..LC are evaluated in registers, and the
// chunk's level-LC value feeds a binary-counter carry for levels LC+1..L, so
// every key row is read once and every pyramid row written once.  Lanes that
// share a row are adjacent, so each warp reads and writes whole 256-byte row
// segments.  The arithmetic is the fp32 add-then-multiply of wf_dwt_build
// (no fused multiply-add: __fadd_rn / __fmul_rn).
#include "wf_internal.cuh"

namespace wf {
namespace {

template <typename T, int L>
__global__ void __launch_bounds__(256) dwt_kernel(const T* __restrict__ K, int64_t sb, int64_t sh, int64_t ss,
                                                  int H, int n, int D, T* __restrict__ coeffs,
                                                  int64_t rows_total, int64_t total_items) {
  constexpr int VEC = Vec<T>::N;
  constexpr int LC = L < 3 ? L : 3;
  constexpr int CH = 1 << LC;
  constexpr int NP = L > LC ? L - LC : 1;
  const int lanes = D / VEC;
  const int64_t nblk = (int64_t)n >> L;
  const int64_t item = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (item >= total_items) return;
  const int lane = (int)(item % lanes);
  const int64_t rest = item / lanes;
  const int64_t blk = rest % nblk;
  const int64_t u = rest / nblk;
  const int64_t bb = u / H, hh = u % H;
  const T* src = K + bb * sb + hh * sh + (blk << L) * ss + (int64_t)lane * VEC;
  T* dst = coeffs + u * rows_total * D + (int64_t)lane * VEC;
  const float c = 0.70710678118654752440f;  // fl32(1/sqrt 2)

  float pend[NP][VEC];
#pragma unroll 1
  for (int ch = 0; ch < (1 << (L - LC)); ++ch) {
    float v[CH][VEC];
#pragma unroll
    for (int t = 0; t < CH; ++t) ld_vec(src + (int64_t)(ch * CH + t) * ss, v[t]);
    const int64_t gc = (blk << (L - LC)) + ch;  // chunk index within the unit
#pragma unroll
    for (int lev = 1; lev <= LC; ++lev) {
      const int cnt = CH >> lev;
      const int64_t off = (int64_t)n - ((int64_t)n >> (lev - 1));
#pragma unroll
      for (int j = 0; j < cnt; ++j) {
#pragma unroll
        for (int e = 0; e < VEC; ++e) v[j][e] = __fmul_rn(__fadd_rn(v[2 * j][e], v[2 * j + 1][e]), c);
        st_vec(dst + (off + gc * cnt + j) * D, v[j]);
      }
    }
    if (L > LC) {
      float x[VEC];
#pragma unroll
      for (int e = 0; e < VEC; ++e) x[e] = v[0][e];
#pragma unroll
      for (int lev = LC + 1; lev <= L; ++lev) {
        const int bit = lev - LC - 1;
        if (((ch >> bit) & 1) == 0) {
#pragma unroll
          for (int e = 0; e < VEC; ++e) pend[bit][e] = x[e];
          break;
        }
#pragma unroll
        for (int e = 0; e < VEC; ++e) x[e] = __fmul_rn(__fadd_rn(pend[bit][e], x[e]), c);
        const int64_t off = (int64_t)n - ((int64_t)n >> (lev - 1));
        st_vec(dst + (off + (gc >> (lev - LC))) * D, x);
      }
    }
  }
}

template <typename T, int L>
cudaError_t run(const void* K, const wf_tensor& kv, void* coeffs, cudaStream_t s) {
  const int U = kv.batch * kv.heads;
  const int lanes = kv.head_dim / Vec<T>::N;
  const int64_t rows_total = (int64_t)kv.seq - ((int64_t)kv.seq >> L);
  const int64_t items = (int64_t)U * ((int64_t)kv.seq >> L) * lanes;
  const int threads = 256;
  const int64_t blocks = (items + threads - 1) / threads;
  dwt_kernel<T, L><<<(unsigned)blocks, threads, 0, s>>>(
      static_cast<const T*>(K), kv.stride_b, kv.stride_h, kv.stride_s, kv.heads, kv.seq, kv.head_dim,
      static_cast<T*>(coeffs), rows_total, items);
  return cudaGetLastError();
}

template <typename T>
cudaError_t dispatch(const void* K, const wf_tensor& kv, int levels, void* coeffs, cudaStream_t s) {
  switch (levels) {
    case 1: return run<T, 1>(K, kv, coeffs, s);
    case 2: return run<T, 2>(K, kv, coeffs, s);
    case 3: return run<T, 3>(K, kv, coeffs, s);
    case 4: return run<T, 4>(K, kv, coeffs, s);
    case 5: return run<T, 5>(K, kv, coeffs, s);
    case 6: return run<T, 6>(K, kv, coeffs, s);
    case 7: return run<T, 7>(K, kv, coeffs, s);
    case 8: return run<T, 8>(K, kv, coeffs, s);
    case 9: return run<T, 9>(K, kv, coeffs, s);
    case 10: return run<T, 10>(K, kv, coeffs, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_dwt(const void* K, const wf_tensor& kv, int levels, void* coeffs, cudaStream_t s) {
  if (kv.dtype == WF_BF16) return dispatch<bf16>(K, kv, levels, coeffs, s);
  return dispatch<float>(K, kv, levels, coeffs, s);
}

}  // namespace wf
