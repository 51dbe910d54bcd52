// libwf C ABI: argument checks, workspace planning and stream-ordered
// launches.  Nothing here allocates device memory or synchronises the stream.
#include <math.h>
#include <string.h>

#include <atomic>
#include <map>
#include <mutex>
#include <utility>

#include "wf_internal.cuh"
#include "wf_testing.h"

#define WF_API extern "C" __attribute__((visibility("default")))

namespace {

using wf::align_up;

int elem_size(int dtype) { return dtype == WF_BF16 ? 2 : 4; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Shape, dtype and alignment of one descriptor (seq may be 0 when allow_empty).
wf_status check_desc(const wf_tensor* t, bool allow_empty) {
  if (!t) return WF_ERR_INVALID_ARG;
  if (t->dtype != WF_F32 && t->dtype != WF_BF16) return WF_ERR_DTYPE;
  if (t->batch < 1 || t->heads < 1 || t->seq < (allow_empty ? 0 : 1)) return WF_ERR_SHAPE;
  if (t->head_dim != 64 && t->head_dim != 128) return WF_ERR_SHAPE;
  if (t->stride_b < 0 || t->stride_h < 0 || t->stride_s < 0) return WF_ERR_SHAPE;
  const int64_t es = elem_size(t->dtype);
  if ((t->stride_b * es) % 16 || (t->stride_h * es) % 16 || (t->stride_s * es) % 16) return WF_ERR_ALIGN;
  if (t->seq > 1 && t->stride_s < t->head_dim) return WF_ERR_SHAPE;
  return WF_OK;
}

bool same_units(const wf_tensor* a, const wf_tensor* b) {
  return a->batch == b->batch && a->heads == b->heads && a->head_dim == b->head_dim;
}

// Query heads per KV head (grouped-query attention), or 0 if the query
// descriptor q cannot be grouped onto kv.
int group_of(const wf_tensor* q, const wf_tensor* kv) {
  if (q->batch != kv->batch || q->head_dim != kv->head_dim || q->heads % kv->heads) return 0;
  return q->heads / kv->heads;
}

wf_status check_levels(const wf_tensor* kv, int levels) {
  if (levels < 1 || levels > 10) return WF_ERR_UNSUPPORTED;
  const int64_t n = kv->seq;
  if ((n >> levels) < 1 || ((n >> levels) << levels) != n) return WF_ERR_SHAPE;
  return WF_OK;
}

wf_status check_keep(int64_t n, int levels, const int32_t* keep) {
  if (!keep) return WF_ERR_INVALID_ARG;
  int64_t cnt = n >> levels;
  for (int l = levels; l >= 1; --l) {
    if (keep[l] < 1 || keep[l] > cnt) return WF_ERR_SCHEDULE;
    cnt = 2 * (int64_t)keep[l];
  }
  if (keep[0] < 1 || keep[0] > cnt) return WF_ERR_SCHEDULE;
  return WF_OK;
}

wf_status cuda_status(cudaError_t e) { return e == cudaSuccess ? WF_OK : WF_ERR_CUDA; }

// Number of SMs of the current device.
bool device_sms(int* sms) {
  *sms = wf::sm_count();
  return *sms > 0;
}

int64_t ceil_guarded(double v) { return (int64_t)ceil(v - 1e-9); }

}  // namespace

namespace wf {

cudaError_t raise_smem_limit(const void* kernel, size_t smem) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, size_t> raised;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  size_t& cur = raised[std::make_pair(dev, kernel)];
  if (cur >= smem) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) cur = smem;
  return e;
}

int sm_count() {
  static std::mutex mu;
  static std::map<int, int> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(dev);
  if (it != cache.end()) return it->second;
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) n = 0;
  cache.emplace(dev, n);
  return n;
}

}  // namespace wf

namespace {

wf_status check_filter_args(const wf_tensor* q, const wf_tensor* kv, int levels, const int32_t* keep) {
  wf_status st;
  if ((st = check_desc(q, false)) != WF_OK) return st;
  if ((st = check_desc(kv, false)) != WF_OK) return st;
  const int G = group_of(q, kv);
  if (!G) return WF_ERR_SHAPE;
  if (q->dtype != kv->dtype) return WF_ERR_DTYPE;
  if (q->seq > wf::kMaxQ || (int64_t)G * q->seq > wf::kMaxQR) return WF_ERR_UNSUPPORTED;
  if ((st = check_levels(kv, levels)) != WF_OK) return st;
  return check_keep(kv->seq, levels, keep);
}

wf_status check_attn_args(const wf_tensor* q, const wf_tensor* kv, int k, const wf_tensor* g, int n_g,
                          const wf_tensor* o) {
  wf_status st;
  if ((st = check_desc(q, false)) != WF_OK) return st;
  if ((st = check_desc(kv, false)) != WF_OK) return st;
  if ((st = check_desc(o, false)) != WF_OK) return st;
  if (!group_of(q, kv) || !same_units(q, o) || o->seq != q->seq) return WF_ERR_SHAPE;
  if (q->dtype != kv->dtype || o->dtype != q->dtype) return WF_ERR_DTYPE;
  if (q->seq > wf::kMaxQ) return WF_ERR_UNSUPPORTED;
  if (k < 1 || k > kv->seq || n_g < 0) return WF_ERR_INVALID_ARG;
  if (n_g > 0) {
    if ((st = check_desc(g, true)) != WF_OK) return st;
    if (!same_units(kv, g) || g->seq != n_g) return WF_ERR_SHAPE;
    if (g->dtype != q->dtype) return WF_ERR_DTYPE;
  }
  return WF_OK;
}

}  // namespace

WF_API const char* wf_status_str(int status) {
  switch (status) {
    case WF_OK: return "WF_OK";
    case WF_ERR_INVALID_ARG: return "WF_ERR_INVALID_ARG: missing pointer or bad count";
    case WF_ERR_SHAPE: return "WF_ERR_SHAPE: shapes disagree or are unsupported";
    case WF_ERR_DTYPE: return "WF_ERR_DTYPE: unknown or mixed dtypes";
    case WF_ERR_ALIGN: return "WF_ERR_ALIGN: pointer or stride not 16-byte aligned";
    case WF_ERR_WORKSPACE: return "WF_ERR_WORKSPACE: buffer too small";
    case WF_ERR_CUDA: return "WF_ERR_CUDA: CUDA runtime or launch failure";
    case WF_ERR_TIMEOUT: return "WF_ERR_TIMEOUT: a bounded device wait gave up";
    case WF_ERR_UNSUPPORTED: return "WF_ERR_UNSUPPORTED: outside what this build implements";
    case WF_ERR_SCHEDULE: return "WF_ERR_SCHEDULE: kept counts infeasible";
    default: return "unknown wf_status";
  }
}

WF_API size_t wf_coeffs_bytes(const wf_tensor* kv, int levels) {
  if (check_desc(kv, false) != WF_OK || check_levels(kv, levels) != WF_OK) return 0;
  const int64_t rows = (int64_t)kv->seq - ((int64_t)kv->seq >> levels);
  return (size_t)kv->batch * kv->heads * rows * kv->head_dim * elem_size(kv->dtype);
}

WF_API wf_status wf_dwt_build(const void* K, const void* V, const wf_tensor* kv, int levels, void* coeffs,
                              size_t coeffs_bytes, void* stream) {
  wf_status st;
  if ((st = check_desc(kv, false)) != WF_OK) return st;
  if ((st = check_levels(kv, levels)) != WF_OK) return st;
  if (!K || !coeffs || V) return WF_ERR_INVALID_ARG;
  if (!aligned16(K) || !aligned16(coeffs)) return WF_ERR_ALIGN;
  if (coeffs_bytes < wf_coeffs_bytes(kv, levels)) return WF_ERR_WORKSPACE;
  return cuda_status(wf::launch_dwt(K, *kv, levels, coeffs, static_cast<cudaStream_t>(stream)));
}

WF_API wf_status wf_cache_update(const void* Knew, const void* Vnew, const wf_tensor* nt, void* K, void* V,
                                 const wf_tensor* kv, int64_t pos, int levels, void* coeffs, size_t coeffs_bytes,
                                 void* stream) {
  wf_status st;
  if ((st = check_desc(kv, false)) != WF_OK) return st;
  if ((st = check_desc(nt, false)) != WF_OK) return st;
  if ((st = check_levels(kv, levels)) != WF_OK) return st;
  if (!same_units(kv, nt)) return WF_ERR_SHAPE;
  if (kv->dtype != nt->dtype) return WF_ERR_DTYPE;
  if (!Knew || !K || !coeffs || (!Vnew) != (!V)) return WF_ERR_INVALID_ARG;
  if (pos < 0 || pos + (int64_t)nt->seq > (int64_t)kv->seq) return WF_ERR_INVALID_ARG;
  if (!aligned16(Knew) || !aligned16(K) || !aligned16(coeffs) || (V && (!aligned16(V) || !aligned16(Vnew))))
    return WF_ERR_ALIGN;
  if (coeffs_bytes < wf_coeffs_bytes(kv, levels)) return WF_ERR_WORKSPACE;
  return cuda_status(
      wf::launch_cache_update(Knew, Vnew, *nt, K, V, *kv, pos, levels, coeffs, static_cast<cudaStream_t>(stream)));
}

WF_API wf_status wf_default_schedule(int64_t n, int levels, int64_t k, int32_t* keep) {
  if (!keep || levels < 1 || levels > 30 || n < 1 || k < 1 || k > n) return WF_ERR_INVALID_ARG;
  if ((n >> levels) < 1 || ((n >> levels) << levels) != n) return WF_ERR_SHAPE;
  const double m = pow((double)k / (double)n, 1.0 / levels);
  int64_t cnt = n >> levels;
  for (int l = levels; l >= 2; --l) {
    int64_t kb = ceil_guarded(m * (double)cnt);
    kb = kb < 1 ? 1 : (kb > cnt ? cnt : kb);
    keep[l] = (int32_t)kb;
    cnt = 2 * kb;
  }
  const int64_t k1 = (k + 1) / 2;
  if (k1 > cnt) return WF_ERR_SCHEDULE;
  keep[1] = (int32_t)k1;
  keep[0] = (int32_t)k;
  return WF_OK;
}

WF_API wf_status wf_level0_schedule(int64_t n, int levels, int64_t k, int32_t* keep) {
  if (!keep || levels < 1 || levels > 30 || n < 1 || k < 1 || k > n) return WF_ERR_INVALID_ARG;
  if ((n >> levels) < 1 || ((n >> levels) << levels) != n) return WF_ERR_SHAPE;
  const double m = pow((double)k / (double)n, 1.0 / (levels + 1));  // L pyramid scans + the token scan
  int64_t cnt = n >> levels;
  for (int l = levels; l >= 1; --l) {
    int64_t kb = ceil_guarded(m * (double)cnt);
    kb = kb < 1 ? 1 : (kb > cnt ? cnt : kb);
    keep[l] = (int32_t)kb;
    cnt = 2 * kb;
  }
  if (k > cnt) return WF_ERR_SCHEDULE;
  keep[0] = (int32_t)k;
  return WF_OK;
}

WF_API wf_status wf_schedule_from_proportions(int64_t n, int levels, const double* m, int32_t* keep) {
  if (!keep || !m || levels < 1 || levels > 30 || n < 1) return WF_ERR_INVALID_ARG;
  if ((n >> levels) < 1 || ((n >> levels) << levels) != n) return WF_ERR_SHAPE;
  int64_t cnt = n >> levels;
  for (int l = levels; l >= 1; --l) {
    if (!(m[l] > 0.0 && m[l] <= 1.0)) return WF_ERR_SCHEDULE;
    int64_t kb = ceil_guarded(m[l] * (double)cnt);
    kb = kb < 1 ? 1 : (kb > cnt ? cnt : kb);
    keep[l] = (int32_t)kb;
    cnt = 2 * kb;
  }
  keep[0] = 2 * keep[1];
  return WF_OK;
}

WF_API size_t wf_filter_workspace_bytes(const wf_tensor* q, const wf_tensor* kv, int levels, const int32_t* keep) {
  if (check_filter_args(q, kv, levels, keep) != WF_OK) return 0;
  return wf::plan_filter(*q, *kv, levels, keep).total;
}

WF_API wf_status wf_filter(const void* Q, const wf_tensor* q, const void* coeffs, const void* K,
                           const wf_tensor* kv, int levels, const int32_t* keep, int32_t* idx, int32_t* level_sets,
                           void* ws, size_t ws_bytes, void* stream) {
  wf_status st = check_filter_args(q, kv, levels, keep);
  if (st != WF_OK) return st;
  if (!Q || !coeffs || !K || !idx || !ws) return WF_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(coeffs) || !aligned16(K)) return WF_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return WF_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(idx) & 3u) != 0 || (reinterpret_cast<uintptr_t>(level_sets) & 3u) != 0)
    return WF_ERR_ALIGN;
  const wf::FilterPlan p = wf::plan_filter(*q, *kv, levels, keep);
  if (ws_bytes < p.total) return WF_ERR_WORKSPACE;
  return cuda_status(wf::launch_filter(p, Q, *q, coeffs, K, *kv, idx, level_sets, ws, static_cast<int*>(ws),
                                       static_cast<cudaStream_t>(stream)));
}

WF_API wf_status wf_wavelet_approx(const void* K, const wf_tensor* kv, const int32_t* cand, int m, int level,
                                   int wavelet, void* out, size_t out_bytes, void* stream) {
  wf_status st;
  if ((st = check_desc(kv, false)) != WF_OK) return st;
  if (!wf::wavelet_taps(wavelet) || level < 1 || level > wf::wavelet_max_level(wavelet)) return WF_ERR_UNSUPPORTED;
  if ((st = check_levels(kv, level)) != WF_OK) return st;
  if (!K || !out || m < 1 || (!cand && m != (kv->seq >> level))) return WF_ERR_INVALID_ARG;
  if (!aligned16(K) || !aligned16(out) || (reinterpret_cast<uintptr_t>(cand) & 3u) != 0) return WF_ERR_ALIGN;
  if (out_bytes < (size_t)kv->batch * kv->heads * m * kv->head_dim * elem_size(kv->dtype)) return WF_ERR_WORKSPACE;
  return cuda_status(wf::launch_wavelet_approx(K, *kv, cand, m, m, level, wavelet, out, (int64_t)m * kv->head_dim,
                                               static_cast<cudaStream_t>(stream)));
}

WF_API size_t wf_filter_wavelet_workspace_bytes(const wf_tensor* q, const wf_tensor* kv, int levels,
                                                const int32_t* keep, int wavelet) {
  if (check_filter_args(q, kv, levels, keep) != WF_OK) return 0;
  if (!wf::wavelet_taps(wavelet) || levels > wf::wavelet_max_level(wavelet)) return 0;
  return wf::wavelet_filter_bytes(wf::plan_filter(*q, *kv, levels, keep));
}

WF_API wf_status wf_filter_wavelet(const void* Q, const wf_tensor* q, const void* top, const void* K,
                                   const wf_tensor* kv, int levels, const int32_t* keep, int wavelet, int32_t* idx,
                                   int32_t* level_sets, void* ws, size_t ws_bytes, void* stream) {
  wf_status st = check_filter_args(q, kv, levels, keep);
  if (st != WF_OK) return st;
  if (!wf::wavelet_taps(wavelet) || levels > wf::wavelet_max_level(wavelet)) return WF_ERR_UNSUPPORTED;
  if (!Q || !top || !K || !idx || !ws) return WF_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(top) || !aligned16(K)) return WF_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return WF_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(idx) & 3u) != 0 || (reinterpret_cast<uintptr_t>(level_sets) & 3u) != 0)
    return WF_ERR_ALIGN;
  const wf::FilterPlan p = wf::plan_filter(*q, *kv, levels, keep);
  if (ws_bytes < wf::wavelet_filter_bytes(p)) return WF_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int sms = 0;
  if (!device_sms(&sms)) return WF_ERR_CUDA;
  const wf::FusedPlan fp = wf::plan_fused(*q, *kv, levels, keep, 0, nullptr, sms);
  if (fp.ok && q->heads == kv->heads)
    return cuda_status(wf::launch_literal_fused(fp, p, Q, *q, top, K, nullptr, *kv, nullptr, nullptr, nullptr,
                                                wavelet, idx, level_sets, nullptr, nullptr, ws,
                                                static_cast<int*>(ws), s));
  return cuda_status(wf::launch_filter_wavelet(p, Q, *q, top, K, *kv, wavelet, idx, level_sets, ws,
                                               static_cast<int*>(ws), s));
}

WF_API size_t wf_attn_workspace_bytes(const wf_tensor* q, int k, int n_g) {
  if (check_desc(q, false) != WF_OK || k < 1 || n_g < 0 || q->seq > wf::kMaxQ) return 0;
  return wf::plan_attn(*q, k, n_g, 1).total;  // the size does not depend on the grouping
}

WF_API wf_status wf_sparse_attn(const void* Q, const wf_tensor* q, const void* K, const void* V,
                                const wf_tensor* kv, const int32_t* idx, int k, const void* Kg, const void* Vg,
                                const wf_tensor* g, void* O, const wf_tensor* o, float scale, void* ws,
                                size_t ws_bytes, void* stream) {
  const int n_g = g ? g->seq : 0;
  wf_status st = check_attn_args(q, kv, k, g, n_g, o);
  if (st != WF_OK) return st;
  if (!Q || !K || !V || !idx || !O || !ws) return WF_ERR_INVALID_ARG;
  if (n_g > 0 && (!Kg || !Vg)) return WF_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O)) return WF_ERR_ALIGN;
  if (n_g > 0 && (!aligned16(Kg) || !aligned16(Vg))) return WF_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || (reinterpret_cast<uintptr_t>(idx) & 3u) != 0)
    return WF_ERR_ALIGN;
  if (!(scale >= 0.f) || isinf(scale)) return WF_ERR_INVALID_ARG;
  const wf::AttnPlan p = wf::plan_attn(*q, k, n_g, group_of(q, kv));
  if (ws_bytes < p.total) return WF_ERR_WORKSPACE;
  const float sc = scale == 0.f ? 1.0f / sqrtf((float)q->head_dim) : scale;
  return cuda_status(wf::launch_attn(p, Q, *q, K, V, *kv, idx, Kg, Vg, n_g > 0 ? g : nullptr, O, *o, sc, ws,
                                     static_cast<int*>(ws), static_cast<cudaStream_t>(stream)));
}

// wf_step keeps a 256-byte status block at the start of its workspace (the
// fused kernel's bounded waits report there); the rest is the scratch of the
// per-stage kernels when the fused kernel does not apply.
constexpr size_t kStatusBytes = 256;

WF_API size_t wf_step_workspace_bytes(const wf_tensor* q, const wf_tensor* kv, int levels, const int32_t* keep,
                                      int n_g) {
  if (check_filter_args(q, kv, levels, keep) != WF_OK || n_g < 0) return 0;
  const size_t f = wf::plan_filter(*q, *kv, levels, keep).total;
  const size_t a = wf::plan_attn(*q, keep[0], n_g, 1).total;
  return kStatusBytes + (f > a ? f : a);
}

WF_API wf_status wf_step(const void* Q, const wf_tensor* q, const void* K, const void* V, const wf_tensor* kv,
                         const void* Kg, const void* Vg, const wf_tensor* g, void* coeffs, size_t coeffs_bytes,
                         int refresh_coeffs, int levels, const int32_t* keep, int32_t* idx, int32_t* level_sets,
                         void* O, const wf_tensor* o, void* ws, size_t ws_bytes, void* stream) {
  wf_status st = check_filter_args(q, kv, levels, keep);
  if (st != WF_OK) return st;
  const int n_g = g ? g->seq : 0;
  if ((st = check_attn_args(q, kv, keep[0], g, n_g, o)) != WF_OK) return st;
  if (!Q || !K || !V || !coeffs || !idx || !O || !ws) return WF_ERR_INVALID_ARG;
  if (n_g > 0 && (!Kg || !Vg)) return WF_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O) || !aligned16(coeffs)) return WF_ERR_ALIGN;
  if (n_g > 0 && (!aligned16(Kg) || !aligned16(Vg))) return WF_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || (reinterpret_cast<uintptr_t>(idx) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(level_sets) & 3u) != 0)
    return WF_ERR_ALIGN;
  if (coeffs_bytes < wf_coeffs_bytes(kv, levels)) return WF_ERR_WORKSPACE;
  if (ws_bytes < wf_step_workspace_bytes(q, kv, levels, keep, n_g)) return WF_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int sms = 0;
  if (!device_sms(&sms)) return WF_ERR_CUDA;
  int* status = static_cast<int*>(ws);  // set by the fused kernel on a timeout; read and cleared by wf_workspace_status
  void* scratch = static_cast<char*>(ws) + kStatusBytes;
  cudaError_t e = cudaSuccess;
  if (refresh_coeffs && (e = wf::launch_dwt(K, *kv, levels, coeffs, s)) != cudaSuccess) return WF_ERR_CUDA;
  // The fused kernel takes one query head per KV head; grouped heads run the per-stage kernels.
  const wf::FusedPlan fp = wf::plan_fused(*q, *kv, levels, keep, n_g, n_g > 0 ? g : nullptr, sms);
  if (fp.ok && q->heads == kv->heads) {
    e = wf::launch_fused(fp, Q, *q, K, V, *kv, Kg, Vg, n_g > 0 ? g : nullptr, coeffs, levels, keep, idx,
                         level_sets, O, *o, status, s);
    return cuda_status(e);
  }
  // Grouped query heads: the grouped filter kernel where it applies, else the
  // per-stage filter; then the per-stage attention.
  const wf::GqaPlan gp = wf::plan_gqa(*q, *kv, levels, keep, sms);
  if (gp.ok) {
    if ((e = wf::launch_gqa_filter(gp, Q, *q, K, *kv, coeffs, levels, keep, idx, level_sets, status, s)) !=
        cudaSuccess)
      return WF_ERR_CUDA;
  } else {
    const wf::FilterPlan fl = wf::plan_filter(*q, *kv, levels, keep);
    if ((e = wf::launch_filter(fl, Q, *q, coeffs, K, *kv, idx, level_sets, scratch, status, s)) != cudaSuccess)
      return WF_ERR_CUDA;
  }
  const wf::AttnPlan ap = wf::plan_attn(*q, keep[0], n_g, group_of(q, kv));
  const float sc = 1.0f / sqrtf((float)q->head_dim);
  e = wf::launch_attn(ap, Q, *q, K, V, *kv, idx, Kg, Vg, n_g > 0 ? g : nullptr, O, *o, sc, scratch, status, s);
  return cuda_status(e);
}

WF_API size_t wf_step_wavelet_workspace_bytes(const wf_tensor* q, const wf_tensor* kv, int levels,
                                              const int32_t* keep, int wavelet, int n_g) {
  if (check_filter_args(q, kv, levels, keep) != WF_OK || n_g < 0) return 0;
  if (!wf::wavelet_taps(wavelet) || levels > wf::wavelet_max_level(wavelet)) return 0;
  const size_t f = wf::wavelet_filter_bytes(wf::plan_filter(*q, *kv, levels, keep));
  const size_t a = wf::plan_attn(*q, keep[0], n_g, 1).total;
  return kStatusBytes + (f > a ? f : a);
}

WF_API wf_status wf_step_wavelet(const void* Q, const wf_tensor* q, const void* top, const void* K, const void* V,
                                 const wf_tensor* kv, const void* Kg, const void* Vg, const wf_tensor* g, int levels,
                                 const int32_t* keep, int wavelet, int32_t* idx, int32_t* level_sets, void* O,
                                 const wf_tensor* o, void* ws, size_t ws_bytes, void* stream) {
  wf_status st = check_filter_args(q, kv, levels, keep);
  if (st != WF_OK) return st;
  if (!wf::wavelet_taps(wavelet) || levels > wf::wavelet_max_level(wavelet)) return WF_ERR_UNSUPPORTED;
  const int n_g = g ? g->seq : 0;
  if ((st = check_attn_args(q, kv, keep[0], g, n_g, o)) != WF_OK) return st;
  if (!Q || !top || !K || !V || !idx || !O || !ws) return WF_ERR_INVALID_ARG;
  if (n_g > 0 && (!Kg || !Vg)) return WF_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(top) || !aligned16(K) || !aligned16(V) || !aligned16(O)) return WF_ERR_ALIGN;
  if (n_g > 0 && (!aligned16(Kg) || !aligned16(Vg))) return WF_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || (reinterpret_cast<uintptr_t>(idx) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(level_sets) & 3u) != 0)
    return WF_ERR_ALIGN;
  if (ws_bytes < wf_step_wavelet_workspace_bytes(q, kv, levels, keep, wavelet, n_g)) return WF_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int sms = 0;
  if (!device_sms(&sms)) return WF_ERR_CUDA;
  int* status = static_cast<int*>(ws);
  void* scratch = static_cast<char*>(ws) + kStatusBytes;
  const wf::FilterPlan fl = wf::plan_filter(*q, *kv, levels, keep);
  const wf::FusedPlan fp = wf::plan_fused(*q, *kv, levels, keep, n_g, n_g > 0 ? g : nullptr, sms);
  if (fp.ok && q->heads == kv->heads)
    return cuda_status(wf::launch_literal_fused(fp, fl, Q, *q, top, K, V, *kv, Kg, Vg, n_g > 0 ? g : nullptr, wavelet,
                                                idx, level_sets, O, o, scratch, status, s));
  cudaError_t e = wf::launch_filter_wavelet(fl, Q, *q, top, K, *kv, wavelet, idx, level_sets, scratch, status, s);
  if (e != cudaSuccess) return WF_ERR_CUDA;
  const wf::AttnPlan ap = wf::plan_attn(*q, keep[0], n_g, group_of(q, kv));
  const float sc = 1.0f / sqrtf((float)q->head_dim);
  e = wf::launch_attn(ap, Q, *q, K, V, *kv, idx, Kg, Vg, n_g > 0 ? g : nullptr, O, *o, sc, scratch, status, s);
  return cuda_status(e);
}

WF_API wf_status wf_workspace_status(void* ws, void* stream) {
  if (!ws) return WF_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int h = 0;
  if (cudaMemcpyAsync(&h, ws, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess) return WF_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return WF_ERR_CUDA;
  if (h != 0) {
    if (cudaMemsetAsync(ws, 0, sizeof(int), s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
      return WF_ERR_CUDA;
    return WF_ERR_TIMEOUT;
  }
  return WF_OK;
}

// ---------------------------------------------------------------------------
// Test-only wait-failure controls (include/wf_testing.h).
// ---------------------------------------------------------------------------
namespace {
std::atomic<int> g_test_stall{0};
std::atomic<long long> g_test_wait_limit{0};
}  // namespace

namespace wf {
WaitControls wait_controls() {
  WaitControls c;
  c.stall = g_test_stall.load(std::memory_order_relaxed);
  const long long lim = g_test_wait_limit.load(std::memory_order_relaxed);
  c.limit = lim > 0 ? lim : kDefaultWaitLimit;
  return c;
}
}  // namespace wf

WF_API wf_status wf_testing_set_wait_failure(int stall, long long wait_limit_cycles) {
  if (wait_limit_cycles < 0) return WF_ERR_INVALID_ARG;
  g_test_wait_limit.store(wait_limit_cycles, std::memory_order_relaxed);
  g_test_stall.store(stall != 0, std::memory_order_relaxed);
  return WF_OK;
}
