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
//
// The update mode (wf_cache_update) runs the same cascade over only the blocks
// that contain token positions [pos, pos + count): a thread takes its slice of
// a new row from the update buffer, writes it into the cache (and the value
// slice too), and takes every other row of the block from the cache, so the
// coefficients it writes equal those of a full build of the updated keys.
#include "wf_internal.cuh"

namespace wf {
namespace {

// Rows [pos, pos + count) of the cache, replaced by an update buffer.
template <typename T>
struct Update {
  const T* Kn;  // [B, H, count, D] new key rows
  const T* Vn;  // new value rows, or null
  T* V;         // value cache (null with Vn)
  int64_t nsb, nsh, nss;  // strides of the update buffers
  int64_t pos, count;
  int64_t blk0;           // first block of the unit that holds a new row
};

template <typename T, int L, bool UPDATE>
__global__ void __launch_bounds__(256) dwt_kernel(const T* K_in, T* K_out, int64_t sb, int64_t sh,
                                                  int64_t ss, int H, int n, int D, T* __restrict__ coeffs,
                                                  int64_t rows_total, int64_t nblk, int64_t total_items,
                                                  Update<T> up) {
  constexpr int VEC = Vec<T>::N;
  constexpr int LC = L < 3 ? L : 3;
  constexpr int CH = 1 << LC;
  constexpr int NP = L > LC ? L - LC : 1;
  const int lanes = D / VEC;
  const int64_t item = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (item >= total_items) return;
  const int lane = (int)(item % lanes);
  const int64_t rest = item / lanes;
  const int64_t blk = rest % nblk + (UPDATE ? up.blk0 : 0);
  const int64_t u = rest / nblk;
  const int64_t bb = u / H, hh = u % H;
  const int64_t tok0 = blk << L;
  const T* src = K_in + bb * sb + hh * sh + tok0 * ss + (int64_t)lane * VEC;
  T* dst = coeffs + u * rows_total * D + (int64_t)lane * VEC;
  const float c = 0.70710678118654752440f;  // fl32(1/sqrt 2)

  float pend[NP][VEC];
#pragma unroll 1
  for (int ch = 0; ch < (1 << (L - LC)); ++ch) {
    float v[CH][VEC];
#pragma unroll
    for (int t = 0; t < CH; ++t) {
      const int64_t tok = tok0 + ch * CH + t;
      if (UPDATE && tok >= up.pos && tok < up.pos + up.count) {
        // A new row: read it from the update buffer, store it into the cache.
        const int64_t r = tok - up.pos;
        const int64_t no = bb * up.nsb + hh * up.nsh + r * up.nss + (int64_t)lane * VEC;
        const int64_t co = bb * sb + hh * sh + tok * ss + (int64_t)lane * VEC;
        ld_vec(up.Kn + no, v[t]);
        st_vec(K_out + co, v[t]);
        if (up.Vn) {
          float vv[VEC];
          ld_vec(up.Vn + no, vv);
          st_vec(up.V + co, vv);
        }
      } else {
        ld_vec(src + (int64_t)(ch * CH + t) * ss, v[t]);
      }
    }
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

// Full build (up.count == 0) or the update of the blocks holding the new rows.
template <typename T, int L>
cudaError_t run(const void* K, void* K_out, const wf_tensor& kv, void* coeffs, const Update<T>& up, cudaStream_t s) {
  const int U = kv.batch * kv.heads;
  const int lanes = kv.head_dim / Vec<T>::N;
  const int64_t rows_total = (int64_t)kv.seq - ((int64_t)kv.seq >> L);
  const int64_t nblk = up.count > 0 ? ((up.pos + up.count - 1) >> L) - (up.pos >> L) + 1 : ((int64_t)kv.seq >> L);
  const int64_t items = (int64_t)U * nblk * lanes;
  const int threads = 256;
  const int64_t blocks = (items + threads - 1) / threads;
  if (up.count > 0) {
    Update<T> u2 = up;
    u2.blk0 = up.pos >> L;
    dwt_kernel<T, L, true><<<(unsigned)blocks, threads, 0, s>>>(
        static_cast<const T*>(K), static_cast<T*>(K_out), kv.stride_b, kv.stride_h, kv.stride_s, kv.heads, kv.seq,
        kv.head_dim, static_cast<T*>(coeffs), rows_total, nblk, items, u2);
  } else {
    dwt_kernel<T, L, false><<<(unsigned)blocks, threads, 0, s>>>(
        static_cast<const T*>(K), nullptr, kv.stride_b, kv.stride_h, kv.stride_s, kv.heads, kv.seq, kv.head_dim,
        static_cast<T*>(coeffs), rows_total, nblk, items, up);
  }
  return cudaGetLastError();
}

template <typename T>
cudaError_t dispatch(const void* K, void* K_out, const wf_tensor& kv, int levels, void* coeffs, const Update<T>& up,
                     cudaStream_t s) {
  switch (levels) {
    case 1: return run<T, 1>(K, K_out, kv, coeffs, up, s);
    case 2: return run<T, 2>(K, K_out, kv, coeffs, up, s);
    case 3: return run<T, 3>(K, K_out, kv, coeffs, up, s);
    case 4: return run<T, 4>(K, K_out, kv, coeffs, up, s);
    case 5: return run<T, 5>(K, K_out, kv, coeffs, up, s);
    case 6: return run<T, 6>(K, K_out, kv, coeffs, up, s);
    case 7: return run<T, 7>(K, K_out, kv, coeffs, up, s);
    case 8: return run<T, 8>(K, K_out, kv, coeffs, up, s);
    case 9: return run<T, 9>(K, K_out, kv, coeffs, up, s);
    case 10: return run<T, 10>(K, K_out, kv, coeffs, up, s);
    default: return cudaErrorInvalidValue;
  }
}

template <typename T>
Update<T> make_update(const void* Kn, const void* Vn, void* V, const wf_tensor* nt, int64_t pos) {
  Update<T> up{};
  if (nt) {
    up.Kn = static_cast<const T*>(Kn);
    up.Vn = static_cast<const T*>(Vn);
    up.V = static_cast<T*>(V);
    up.nsb = nt->stride_b;
    up.nsh = nt->stride_h;
    up.nss = nt->stride_s;
    up.pos = pos;
    up.count = nt->seq;
  }
  return up;
}

}  // namespace

cudaError_t launch_dwt(const void* K, const wf_tensor& kv, int levels, void* coeffs, cudaStream_t s) {
  if (kv.dtype == WF_BF16) return dispatch<bf16>(K, nullptr, kv, levels, coeffs, make_update<bf16>(0, 0, 0, 0, 0), s);
  return dispatch<float>(K, nullptr, kv, levels, coeffs, make_update<float>(0, 0, 0, 0, 0), s);
}

cudaError_t launch_cache_update(const void* Kn, const void* Vn, const wf_tensor& nt, void* K, void* V,
                                const wf_tensor& kv, int64_t pos, int levels, void* coeffs, cudaStream_t s) {
  if (kv.dtype == WF_BF16)
    return dispatch<bf16>(K, K, kv, levels, coeffs, make_update<bf16>(Kn, Vn, V, &nt, pos), s);
  return dispatch<float>(K, K, kv, levels, coeffs, make_update<float>(Kn, Vn, V, &nt, pos), s);
}

}  // namespace wf
