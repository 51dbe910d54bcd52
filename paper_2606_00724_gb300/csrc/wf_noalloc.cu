// wf_sparse_attn_noalloc: sparse attention for callers that cannot allocate
// device memory.
//
// wf_sparse_attn needs a caller-provided device workspace for its split-K
// partial results.  Some callers cannot obtain one: a plugin inside a host
// engine that owns every device allocation and hands out no scratch, or
// code on a path where allocating after start-up is forbidden.  This entry
// point runs the same kernels with a fixed scratch area that lives in this
// translation unit as a static device array, so the call itself allocates
// nothing.  The array (WF_NOALLOC_SCRATCH_BYTES) is reserved in every CUDA
// context that loads this module and stays reserved until the context is
// destroyed (for the primary context: until the process exits).
#include <cuda.h>

#include <map>
#include <mutex>

#include "wf_internal.cuh"

#define WF_API extern "C" __attribute__((visibility("default")))

namespace {

// Shared by every call in a context; see the header for the rules.  Its first
// word is the status word of the tensor-core attention kernels (zero when the
// module loads; wf_noalloc_status reads and clears it).
static __device__ __align__(256) unsigned char g_noalloc_scratch[WF_NOALLOC_SCRATCH_BYTES];

// The array's device address differs between CUDA contexts (each context
// loads its own copy of the module), so it is cached per context.  Contexts
// are told apart by their driver-assigned id, which is never reused within a
// process: a context created after another was destroyed (for example the
// primary context after a device reset) gets a fresh entry even if it reuses
// the old handle.
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

std::mutex g_mu;
std::map<unsigned long long, void*> g_addr_by_ctx;
CtxGetCurrentFn g_ctx_get_current = nullptr;
CtxGetIdFn g_ctx_get_id = nullptr;

// Driver entry points, fetched through the runtime so that the library does
// not link the driver library directly.  Called with g_mu held.
bool driver_entry_points() {
  if (g_ctx_get_current && g_ctx_get_id) return true;
  void* a = nullptr;
  void* b = nullptr;
  cudaDriverEntryPointQueryResult qa{}, qb{};
  if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &a, 12000, cudaEnableDefault, &qa) != cudaSuccess ||
      qa != cudaDriverEntryPointSuccess || !a)
    return false;
  if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &b, 12000, cudaEnableDefault, &qb) != cudaSuccess ||
      qb != cudaDriverEntryPointSuccess || !b)
    return false;
  g_ctx_get_current = reinterpret_cast<CtxGetCurrentFn>(a);
  g_ctx_get_id = reinterpret_cast<CtxGetIdFn>(b);
  return true;
}

// Id of the calling thread's current context (0 if none is current).
bool current_context_id(unsigned long long* id) {
  CUcontext ctx = nullptr;
  if (g_ctx_get_current(&ctx) != CUDA_SUCCESS) return false;
  if (!ctx) {
    *id = 0;
    return true;
  }
  return g_ctx_get_id(ctx, id) == CUDA_SUCCESS;
}

// Host code cannot use g_noalloc_scratch's name as a device address: on the
// host it names a stand-in object.  The device address is looked up with
// cudaGetSymbolAddress the first time a context calls in (which also loads
// the module into that context and, for the runtime's primary context,
// creates and binds the context), then served from the cache.
wf_status scratch_for_current_context(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return WF_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!driver_entry_points()) return WF_ERR_CUDA;
  unsigned long long id = 0;
  if (!current_context_id(&id)) return WF_ERR_CUDA;
  if (id != 0) {
    auto it = g_addr_by_ctx.find(id);
    if (it != g_addr_by_ctx.end()) {
      *out = it->second;
      return WF_OK;
    }
  }
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return WF_ERR_CUDA;
  // With no context current before the lookup, the runtime has just bound the
  // device's primary context: key the entry on that one.
  if (id == 0 && (!current_context_id(&id) || id == 0)) return WF_ERR_CUDA;
  g_addr_by_ctx.emplace(id, p);
  *out = p;
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
  wf_status st = scratch_for_current_context(&scratch);
  if (st != WF_OK) return st;
  // Every scratch word the kernels read is written earlier in the same call
  // (per-chunk maxima, sums and partial outputs), so nothing is cleared.  The
  // status word is only ever set, never cleared, by the kernels.
  return wf_sparse_attn(Q, q, K, V, kv, idx, k, Kg, Vg, g, O, o, scale, scratch, WF_NOALLOC_SCRATCH_BYTES,
                        stream);
}

WF_API wf_status wf_noalloc_status(void* stream) {
  void* scratch = nullptr;
  wf_status st = scratch_for_current_context(&scratch);
  if (st != WF_OK) return st;
  return wf_workspace_status(scratch, stream);
}
