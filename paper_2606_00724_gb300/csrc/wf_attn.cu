// Sparse attention over the gathered rows (Algorithm 1, final step).
//
// Split-K ("flash-decoding") over the sparse key list of each unit: the list
// is [K[idx[0..k)]; Kg[0..n_g)], cut into chunks of 64 keys.  One CTA per
// (chunk, unit) gathers its K/V rows, computes the 64-key logits for every
// query row, their local max m and sum l of exp, and the un-normalised
// partial output sum_t exp(s_t - m) V_t.  A combine kernel rescales the
// partials to the global max and normalises.  fp32 logits, softmax and
// accumulation; O is rounded once to the output dtype.
#include <math.h>

#include "wf_internal.cuh"

namespace wf {
namespace {

constexpr int CH = kAttnChunk;
constexpr int QMAX = kMaxQ;

template <typename T, int D, int QM>
__global__ void __launch_bounds__(256) attn_split_kernel(
    const T* __restrict__ Q, int64_t qsb, int64_t qsh, int64_t qss, const T* __restrict__ K,
    const T* __restrict__ V, int64_t ksb, int64_t ksh, int64_t kss, int n, const int32_t* __restrict__ idx, int k,
    const T* __restrict__ Kg, const T* __restrict__ Vg, int64_t gsb, int64_t gsh, int64_t gss, int ng, int q, int H,
    int G, float scale, int nsplit, int qstride, float* __restrict__ Opart, float2* __restrict__ ML) {
  constexpr int VEC = Vec<T>::N;
  constexpr int KS = D + 4;
  extern __shared__ __align__(16) float smem[];
  float* Qs = smem;                // [QM][D]
  float* Ks = Qs + QM * D;         // [CH][KS]
  float* Vs = Ks + CH * KS;        // [CH][D]
  float* P = Vs + CH * D;          // [QM][CH + 1]
  const int u = blockIdx.y;
  const int sp = blockIdx.x;
  const int t0 = sp * CH;
  const int total = k + ng;
  const int cnt = min(CH, total - t0);
  const int64_t bb = u / H, hh = u % H;
  const int64_t hk = hh / G;  // the KV head of this query head
  const int tid = threadIdx.x;

  const T* qbase = Q + bb * qsb + hh * qsh;
  for (int e = tid; e < QM * (D / VEC); e += blockDim.x) {
    const int i = e / (D / VEC), c = (e % (D / VEC)) * VEC;
    float v[VEC];
    if (i < q) ld_vec(qbase + (int64_t)i * qss + c, v);
    else
#pragma unroll
      for (int x = 0; x < VEC; ++x) v[x] = 0.f;
#pragma unroll
    for (int x = 0; x < VEC; ++x) Qs[i * D + c + x] = v[x];
  }
  const int32_t* ui = idx + (bb * (H / G) + hk) * k;
  for (int e = tid; e < CH * (D / VEC); e += blockDim.x) {
    const int j = e / (D / VEC), c = (e % (D / VEC)) * VEC;
    float kv[VEC], vv[VEC];
    if (j < cnt) {
      const int t = t0 + j;
      const T *kp, *vp;
      if (t < k) {
        int r = ui[t];
        r = r < 0 ? 0 : (r >= n ? n - 1 : r);
        const int64_t o = bb * ksb + hk * ksh + (int64_t)r * kss + c;
        kp = K + o; vp = V + o;
      } else {
        const int64_t o = bb * gsb + hk * gsh + (int64_t)(t - k) * gss + c;
        kp = Kg + o; vp = Vg + o;
      }
      ld_vec(kp, kv);
      ld_vec(vp, vv);
    } else {
#pragma unroll
      for (int x = 0; x < VEC; ++x) { kv[x] = 0.f; vv[x] = 0.f; }
    }
#pragma unroll
    for (int x = 0; x < VEC; ++x) { Ks[j * KS + c + x] = kv[x]; Vs[j * D + c + x] = vv[x]; }
  }
  __syncthreads();

  // Logits: lane -> keys (lane, lane+32), warp -> query rows warp + 8r.
  const int lane = tid & 31, warp = tid >> 5;
  float acc0[QM / 8], acc1[QM / 8];
#pragma unroll
  for (int r = 0; r < QM / 8; ++r) { acc0[r] = 0.f; acc1[r] = 0.f; }
#pragma unroll 2
  for (int c = 0; c < D; c += 4) {
    const float4 k0 = *reinterpret_cast<const float4*>(&Ks[lane * KS + c]);
    const float4 k1 = *reinterpret_cast<const float4*>(&Ks[(lane + 32) * KS + c]);
#pragma unroll
    for (int r = 0; r < QM / 8; ++r) {
      const float4 qv = *reinterpret_cast<const float4*>(&Qs[(warp + 8 * r) * D + c]);
      acc0[r] = fmaf(qv.x, k0.x, fmaf(qv.y, k0.y, fmaf(qv.z, k0.z, fmaf(qv.w, k0.w, acc0[r]))));
      acc1[r] = fmaf(qv.x, k1.x, fmaf(qv.y, k1.y, fmaf(qv.z, k1.z, fmaf(qv.w, k1.w, acc1[r]))));
    }
  }
  float2* ml = ML + ((int64_t)u * nsplit + sp) * qstride;  // a split's partials: qstride rows
#pragma unroll
  for (int r = 0; r < QM / 8; ++r) {
    const int i = warp + 8 * r;
    if (i >= q) break;
    const float s0 = lane < cnt ? acc0[r] * scale : -INFINITY;
    const float s1 = lane + 32 < cnt ? acc1[r] * scale : -INFINITY;
    float mx = fmaxf(s0, s1);
#pragma unroll
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    const float p0 = lane < cnt ? expf(s0 - mx) : 0.f;
    const float p1 = lane + 32 < cnt ? expf(s1 - mx) : 0.f;
    float z = p0 + p1;
#pragma unroll
    for (int o = 16; o; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    P[i * (CH + 1) + lane] = p0;
    P[i * (CH + 1) + lane + 32] = p1;
    if (lane == 0) ml[i] = make_float2(mx, z);
  }
  __syncthreads();

  // Partial output: thread -> channel c, query rows [qg*QPT, (qg+1)*QPT).
  constexpr int GROUPS = 256 / D;
  constexpr int QPT = QM / GROUPS;
  const int c = tid % D, qg = tid / D;
  float o[QPT];
#pragma unroll
  for (int r = 0; r < QPT; ++r) o[r] = 0.f;
  for (int t = 0; t < cnt; ++t) {
    const float v = Vs[t * D + c];
#pragma unroll
    for (int r = 0; r < QPT; ++r) o[r] = fmaf(P[(qg * QPT + r) * (CH + 1) + t], v, o[r]);
  }
  float* op = Opart + ((int64_t)u * nsplit + sp) * qstride * D;
#pragma unroll
  for (int r = 0; r < QPT; ++r) {
    const int i = qg * QPT + r;
    if (i < q) op[(int64_t)i * D + c] = o[r];
  }
}

// One CTA per (unit, query row): the weight exp(m_s - M) of every split s
// and the denominator are formed once in shared memory, then each output
// element is one pass over the splits' partial outputs.
// The combine of nsplit partials (O, m, l) per query row: one warp per row,
// each lane CPL consecutive channels (CPL = D / 32).  Every lane forms the
// split weights exp(m_s - M) (M the largest m_s) itself, so no shared memory
// or block barrier is needed; the per-element order (weights, then fused
// multiply-adds in split order, then one division) is the one of a plain loop.
template <typename T, int D>
__global__ void __launch_bounds__(256) attn_combine_kernel(const float* __restrict__ Opart,
                                                           const float2* __restrict__ ML, int nsplit, int q, int H,
                                                           int qstride, T* __restrict__ O, int64_t osb, int64_t osh,
                                                           int64_t oss) {
  constexpr int CPL = D / 32;
  const int u = blockIdx.x;
  const int i = blockIdx.y * 8 + (threadIdx.x >> 5);  // query row of this warp
  if (i >= q) return;
  const int lane = threadIdx.x & 31;
  const int64_t bb = u / H, hh = u % H;
  const float2* ml = ML + (int64_t)u * nsplit * qstride + i;
  float mx = -INFINITY;
  for (int s = 0; s < nsplit; ++s) mx = fmaxf(mx, ml[(int64_t)s * qstride].x);
  const float* op = Opart + ((int64_t)u * nsplit * qstride + i) * D + lane * CPL;
  float num[CPL], den = 0.f;
#pragma unroll
  for (int e = 0; e < CPL; ++e) num[e] = 0.f;
#pragma unroll 4
  for (int s = 0; s < nsplit; ++s) {
    const float2 st = ml[(int64_t)s * qstride];
    const float w = expf(st.x - mx);
    den = fmaf(st.y, w, den);
    const float* os = op + (int64_t)s * qstride * D;
    if (CPL == 4) {
      const float4 v = *reinterpret_cast<const float4*>(os);
      num[0] = fmaf(v.x, w, num[0]);
      num[1] = fmaf(v.y, w, num[1]);
      num[2] = fmaf(v.z, w, num[2]);
      num[3] = fmaf(v.w, w, num[3]);
    } else {
#pragma unroll
      for (int e = 0; e < CPL; ++e) num[e] = fmaf(os[e], w, num[e]);
    }
  }
  T* ob = O + bb * osb + hh * osh + (int64_t)i * oss + lane * CPL;
#pragma unroll
  for (int e = 0; e < CPL; ++e) from_f32(ob[e], num[e] / den);
}

// The combine of nsplit partials per query-head unit into O.
template <typename T>
cudaError_t combine(const AttnPlan& p, int nsplit, void* O, const wf_tensor& od, void* ws, cudaStream_t s) {
  float* Opart = reinterpret_cast<float*>(static_cast<char*>(ws) + p.off_o);
  float2* ML = reinterpret_cast<float2*>(static_cast<char*>(ws) + p.off_ml);
  const dim3 grid((unsigned)p.U, (unsigned)((p.q + 7) / 8));
  if (p.d == 128)
    attn_combine_kernel<T, 128><<<grid, 256, 0, s>>>(Opart, ML, nsplit, p.q, p.H, p.qstride, static_cast<T*>(O),
                                                     od.stride_b, od.stride_h, od.stride_s);
  else
    attn_combine_kernel<T, 64><<<grid, 256, 0, s>>>(Opart, ML, nsplit, p.q, p.H, p.qstride, static_cast<T*>(O),
                                                    od.stride_b, od.stride_h, od.stride_s);
  return cudaGetLastError();
}

template <typename T, int D, int QM>
cudaError_t run(const AttnPlan& p, const void* Q, const wf_tensor& qd, const void* K, const void* V,
                const wf_tensor& kv, const int32_t* idx, const void* Kg, const void* Vg, const wf_tensor* g,
                void* O, const wf_tensor& od, float scale, void* ws, cudaStream_t s) {
  float* Opart = reinterpret_cast<float*>(static_cast<char*>(ws) + p.off_o);
  float2* ML = reinterpret_cast<float2*>(static_cast<char*>(ws) + p.off_ml);
  const size_t smem = sizeof(float) * (size_t)(QM * D + CH * (D + 4) + CH * D + QM * (CH + 1));
  cudaError_t e = raise_smem_limit(reinterpret_cast<const void*>(attn_split_kernel<T, D, QM>), smem);
  if (e != cudaSuccess) return e;
  const int64_t gsb = g ? g->stride_b : 0, gsh = g ? g->stride_h : 0, gss = g ? g->stride_s : 0;
  attn_split_kernel<T, D, QM><<<dim3(p.nsplit, p.U), 256, smem, s>>>(
      static_cast<const T*>(Q), qd.stride_b, qd.stride_h, qd.stride_s, static_cast<const T*>(K),
      static_cast<const T*>(V), kv.stride_b, kv.stride_h, kv.stride_s, kv.seq, idx, p.k, static_cast<const T*>(Kg),
      static_cast<const T*>(Vg), gsb, gsh, gss, p.ng, p.q, p.H, p.G, scale, p.nsplit, p.qstride, Opart, ML);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  return combine<T>(p, p.nsplit, O, od, ws, s);
}

}  // namespace

AttnPlan plan_attn(const wf_tensor& q, int k, int ng, int group) {
  AttnPlan p{};
  p.U = q.batch * q.heads;
  p.H = q.heads;
  p.G = group;
  p.q = q.seq;
  p.d = q.head_dim;
  p.k = k;
  p.ng = ng;
  p.dtype = q.dtype;
  p.nsplit = (k + ng + CH - 1) / CH;
  // Partials of a split take q rows rounded up to 32 (every kernel's query
  // tile holds at most that many valid rows).
  p.qstride = (q.seq + 31) / 32 * 32;
  size_t off = 256;  // status block
  p.off_o = off;  off = align_up(off + (size_t)p.U * p.nsplit * p.qstride * p.d * sizeof(float), 256);
  p.off_ml = off; off = align_up(off + (size_t)p.U * p.nsplit * p.qstride * sizeof(float2), 256);
  p.total = off;
  return p;
}

cudaError_t launch_attn(const AttnPlan& p, const void* Q, const wf_tensor& qd, const void* K, const void* V,
                        const wf_tensor& kv, const int32_t* idx, const void* Kg, const void* Vg,
                        const wf_tensor* g, void* O, const wf_tensor& od, float scale, void* ws, int* status,
                        cudaStream_t s) {
  // bf16 with head_dim 128: tensor cores.
  if (tc_attn_supported(p, p.G * p.q)) {
    int nsplit = 0;
    cudaError_t e = launch_tc_attn(p, Q, qd, K, V, kv, idx, Kg, Vg, g, scale, status, ws, &nsplit, s);
    if (e != cudaSuccess) return e;
    return combine<bf16>(p, nsplit, O, od, ws, s);
  }
  // Query blocks of up to 32 rows take the 32-row tile.
#define WF_ATTN_RUN(T, DD)                                                                  \
  (p.q <= 32 ? run<T, DD, 32>(p, Q, qd, K, V, kv, idx, Kg, Vg, g, O, od, scale, ws, s)     \
             : run<T, DD, QMAX>(p, Q, qd, K, V, kv, idx, Kg, Vg, g, O, od, scale, ws, s))
  if (p.dtype == WF_BF16) return p.d == 64 ? WF_ATTN_RUN(bf16, 64) : WF_ATTN_RUN(bf16, 128);
  return p.d == 64 ? WF_ATTN_RUN(float, 64) : WF_ATTN_RUN(float, 128);
#undef WF_ATTN_RUN
}

}  // namespace wf
