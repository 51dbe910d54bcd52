// wf_sparse_attn_noalloc: sparse attention for callers that cannot allocate
// device memory.
//
// wf_sparse_attn needs a caller-provided device workspace for its split-K
// partial results.  Some callers cannot obtain one: a plugin inside a host
// engine that owns every device allocation and hands out no scratch, or
// code on a path where allocating after start-up is forbidden.  This entry
// point runs the same kernels with a fixed scratch area that lives in this
// translation unit as a static device array, so the call itself allocates
// nothing.  The array (WF_NOALLOC_SCRATCH_BYTES) is reserved on every device
// that loads this module and stays reserved until the process exits.
#include <mutex>

#include "wf_internal.cuh"

#define WF_API extern "C" __attribute__((visibility("default")))

namespace {

// Shared by every call on a device; see the header for the rules.
static __device__ __align__(256) unsigned char g_noalloc_scratch[WF_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// Host code cannot use g_noalloc_scratch's name as a device address: on the
// host it names a stand-in object.  The device address is looked up once per
// device, with that device current.
wf_status scratch_for_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return WF_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return WF_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return WF_OK;
}

}  // namespace

WF_API wf_status wf_sparse_attn_noalloc(const void* Q, const wf_tensor* q, const void* K, const void* V,
                                        const wf_tensor* kv, const int32_t* idx, int k, const void* Kg,
                                        const void* Vg, const wf_tensor* g, void* O, const wf_tensor* o,
                                        float scale, void* stream) {
  // Size check first, so an oversized request fails before any set-up.
  const int n_g = g ? g->seq : 0;
  const size_t need = wf_attn_workspace_bytes(q, k, n_g);
  if (need > (size_t)WF_NOALLOC_SCRATCH_BYTES) return WF_ERR_WORKSPACE;
  void* scratch = nullptr;
  wf_status st = scratch_for_current_device(&scratch);
  if (st != WF_OK) return st;
  // Every scratch word the kernels read is written earlier in the same call
  // (per-chunk maxima, sums and partial outputs), so nothing is cleared.
  return wf_sparse_attn(Q, q, K, V, kv, idx, k, Kg, Vg, g, O, o, scale, scratch, WF_NOALLOC_SCRATCH_BYTES,
                        stream);
}
