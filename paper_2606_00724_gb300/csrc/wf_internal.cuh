// Internal declarations shared by the libwf translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "wf.h"

namespace wf {

typedef __nv_bfloat16 bf16;

// Elements per 16-byte vector.
template <typename T> struct Vec;
template <> struct Vec<float> { static constexpr int N = 4; };
template <> struct Vec<bf16> { static constexpr int N = 8; };

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Load one 16-byte vector of T and widen it to fp32 (exact).
__device__ __forceinline__ void ld_vec(const float* p, float* o) {
  float4 v = __ldg(reinterpret_cast<const float4*>(p));
  o[0] = v.x; o[1] = v.y; o[2] = v.z; o[3] = v.w;
}
__device__ __forceinline__ void ld_vec(const bf16* p, float* o) {
  uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
  o[0] = bf16_lo(v.x); o[1] = bf16_hi(v.x); o[2] = bf16_lo(v.y); o[3] = bf16_hi(v.y);
  o[4] = bf16_lo(v.z); o[5] = bf16_hi(v.z); o[6] = bf16_lo(v.w); o[7] = bf16_hi(v.w);
}

// Round fp32 to the storage type (bf16: round to nearest even) and store 16 bytes.
__device__ __forceinline__ void st_vec(float* p, const float* v) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
}
__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);  // .x = a (low half), .y = b
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ void st_vec(bf16* p, const float* v) {
  uint4 w;
  w.x = pack_bf16(v[0], v[1]); w.y = pack_bf16(v[2], v[3]);
  w.z = pack_bf16(v[4], v[5]); w.w = pack_bf16(v[6], v[7]);
  *reinterpret_cast<uint4*>(p) = w;
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(bf16 x) { return __bfloat162float(x); }
__device__ __forceinline__ void from_f32(float& d, float x) { d = x; }
__device__ __forceinline__ void from_f32(bf16& d, float x) { d = __float2bfloat16_rn(x); }

// A [B, H, rows, d] row source: element (b, h, r, c) at
// base + b*sb + h*sh + off + r*ss + c.
struct RowSrc {
  const void* base;
  int64_t sb, sh, ss, off;
};

// ---------------------------------------------------------------------------
// Launchers (each returns cudaSuccess or the launch error).
// ---------------------------------------------------------------------------

// DWT pyramid of the keys: see wf_dwt_build.
cudaError_t launch_dwt(const void* K, const wf_tensor& kv, int levels, void* coeffs, cudaStream_t s);
// Cache update with the refresh of the touched pyramid blocks: see wf_cache_update.
cudaError_t launch_cache_update(const void* Kn, const void* Vn, const wf_tensor& nt, void* K, void* V,
                                const wf_tensor& kv, int64_t pos, int levels, void* coeffs, cudaStream_t s);

// Filter workspace plan for one call.  A unit is one (batch, KV head); its
// query block is the qs rows of each of its G query heads, q = G qs rows.
struct FilterPlan {
  int U, H, q, d, n, L, dtype;
  int G, qs;
  int32_t keep[16];
  int cmax;        // largest candidate count over the scales (and the trim)
  int tiles_max;   // ceil(cmax / kScoreTile)
  bool trim;
  size_t off_cand_a, off_cand_b, off_w, off_logits, off_part, total;  // a 256-byte status block precedes off_cand_a
};
constexpr int kScoreTile = 32;
constexpr int kMaxQ = 64;    // query rows per query head
constexpr int kMaxQR = 256;  // query rows per KV head (all heads of a group)
FilterPlan plan_filter(const wf_tensor& q, const wf_tensor& kv, int levels, const int32_t* keep);
// status: the word a tensor-core kernel sets when a bounded wait gives up.
cudaError_t launch_filter(const FilterPlan& p, const void* Q, const wf_tensor& qd, const void* coeffs,
                          const void* K, const wf_tensor& kv, int32_t* idx, int32_t* level_sets, void* ws,
                          int* status, cudaStream_t s);
// The tensor-core skim (bf16, head_dim 128, <= 256 query rows per unit): the
// per-tile softmax partials and the ranking keys log2 W of one scale's m
// candidates (rows from src, gathered through cand when not NULL).
bool tc_skim_supported(const FilterPlan& p);
cudaError_t launch_tc_skim(const FilterPlan& p, const void* Q, const wf_tensor& qd, RowSrc src, const int32_t* cand,
                           int m, float2* part, float* W, float* cvec, int* status, cudaStream_t s);

// Approximation rows at scale `level` of the periodized transform (wavelet
// WF_WAVELET_*) of the keys of blocks [2^level c, 2^level (c + 1)) for the m
// candidates c of every unit (cand: [units][cand_stride], NULL = all blocks),
// into out[unit * out_unit + j * head_dim + channel] in the key dtype.
// pdl: launch as a programmatic dependent of the previous kernel on the stream.
cudaError_t launch_wavelet_approx(const void* K, const wf_tensor& kv, const int32_t* cand, int64_t cand_stride, int m,
                                  int level, int wavelet, void* out, int64_t out_unit, cudaStream_t s,
                                  bool pdl = false);
int wavelet_taps(int wavelet);       // 0 for an unknown basis
int wavelet_max_level(int wavelet);  // deepest scale the approximation kernel supports
// Filtering with a generic basis (Eq. 11 taken literally): the filter plan's
// workspace followed by one block of approximation rows [units][cmax][d].
size_t wavelet_filter_bytes(const FilterPlan& p);
cudaError_t launch_filter_wavelet(const FilterPlan& p, const void* Q, const wf_tensor& qd, const void* top,
                                  const void* K, const wf_tensor& kv, int wavelet, int32_t* idx, int32_t* level_sets,
                                  void* ws, int* status, cudaStream_t s);

// Sparse attention workspace plan.  A unit is one (batch, query head); it
// reads KV head h / G and that head's index row.
struct AttnPlan {
  int U, H, q, d, k, ng, nsplit, dtype;
  int G;
  int qstride;  // query rows a split's partials take: q rounded up to 32
  size_t off_o, off_ml, total;
};
constexpr int kAttnChunk = 64;
AttnPlan plan_attn(const wf_tensor& q, int k, int ng, int group);
// status: the word a tensor-core kernel sets when a bounded wait gives up.
cudaError_t launch_attn(const AttnPlan& p, const void* Q, const wf_tensor& qd, const void* K, const void* V,
                        const wf_tensor& kv, const int32_t* idx, const void* Kg, const void* Vg,
                        const wf_tensor* g, void* O, const wf_tensor& od, float scale, void* ws, int* status,
                        cudaStream_t s);
// The tensor-core split attention (bf16, head_dim 128, <= 256 query rows per
// key unit): partials in the workspace's flash-decoding layout, split count
// into *nsplit_out.
bool tc_attn_supported(const AttnPlan& p, int kv_group_rows);
cudaError_t launch_tc_attn(const AttnPlan& p, const void* Q, const wf_tensor& qd, const void* K, const void* V,
                           const wf_tensor& kv, const int32_t* idx, const void* Kg, const void* Vg,
                           const wf_tensor* g, float scale, int* status, void* ws, int* nsplit_out,
                           cudaStream_t s);

// Fused step (bf16, head_dim 128, <= 32 query rows): one cluster of cs CTAs
// per P units.
struct FusedPlan {
  bool ok;
  int cs, P, clusters, stages, tmem_cols, ucols, ecol, cmax, kmax, U;
  size_t smem;
  bool trim;
  bool wide;  // one unit per cluster served by both compute warpgroups
};
FusedPlan plan_fused(const wf_tensor& q, const wf_tensor& kv, int levels, const int32_t* keep, int n_g,
                     const wf_tensor* g, int num_sms);
// Part of the chain in one launch (the literal-basis path runs one launch per
// scale, with the transform of the candidates' blocks between launches):
// scales lev_top down to lev_bot; the previous selection J_{lev_top+1} as its
// children list jin (when lev_top < L); the children of the last selection to
// jout unless final_sel (then mu^0 goes to idx); the attention if attn.
// Scale lev_top's rows come from lrows ([units][m][d], unit stride lrows_unit
// elements) when not null, else from the pyramid (only when lev_top = L).
// pdl: launch as a programmatic dependent of the previous kernel on the
// stream (its set-up overlaps that kernel's tail).
struct FusedRange {
  int lev_top, lev_bot, final_sel, attn, pdl;
  const int32_t* jin;
  int32_t* jout;
  int64_t jstride;
  const void* lrows;
  int64_t lrows_unit;
};
// range == nullptr: the whole step (every scale, mu^0, the attention).
cudaError_t launch_fused(const FusedPlan& fp, const void* Q, const wf_tensor& qd, const void* K, const void* V,
                         const wf_tensor& kv, const void* Kg, const void* Vg, const wf_tensor* g,
                         const void* coeffs, int levels, const int32_t* keep, int32_t* idx, int32_t* level_sets,
                         void* O, const wf_tensor& od, int* status, cudaStream_t s,
                         const FusedRange* range = nullptr);

// The literal-basis filter on the fused kernel (bf16, d 128, one query head
// per KV head, a fused plan fp for the same shapes): one launch per scale,
// each after the transform of its candidates' gathered blocks
// (launch_wavelet_approx, into the block after the filter plan's workspace);
// the candidate lists pass between launches in the plan's two candidate
// buffers.  With O not null the last launch also runs the attention (od its
// descriptor; Kg/Vg/g the generation rows).
cudaError_t launch_literal_fused(const FusedPlan& fp, const FilterPlan& fl, const void* Q, const wf_tensor& qd,
                                 const void* top, const void* K, const void* V, const wf_tensor& kv, const void* Kg,
                                 const void* Vg, const wf_tensor* g, int wavelet, int32_t* idx, int32_t* level_sets,
                                 void* O, const wf_tensor* od, void* ws, int* status, cudaStream_t s);

// The grouped-query filter on the fused kernel design (one cluster per
// (batch, key head); the stacked query rows of the G query heads as MMA
// columns): mu^0 and the level sets, for the per-stage attention after it.
struct GqaPlan {
  bool ok;
  int cs, stages, tmem_cols, nch, G, cmax, kmax, U;
  size_t smem;
  bool trim;
};
GqaPlan plan_gqa(const wf_tensor& q, const wf_tensor& kv, int levels, const int32_t* keep, int num_sms);
cudaError_t launch_gqa_filter(const GqaPlan& gp, const void* Q, const wf_tensor& qd, const void* K,
                              const wf_tensor& kv, const void* coeffs, int levels, const int32_t* keep, int32_t* idx,
                              int32_t* level_sets, int* status, cudaStream_t s);

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// A kernel's dynamic shared-memory limit, raised once per device and kernel
// to the largest size requested so far (otherwise a host call on every
// launch).
cudaError_t raise_smem_limit(const void* kernel, size_t smem);
// The current device's SM count, looked up once per device (0 on an error).
int sm_count();

// Bounds of the tensor-core kernels' waits.  The default, about one second of
// SM clock cycles, can be lowered (and a stalled first wait requested) only
// through the test-only wf_testing_set_wait_failure.
constexpr long long kDefaultWaitLimit = 1ll << 31;
struct WaitControls {
  int stall;        // the first wait of each CTA waits on a barrier that nothing completes
  long long limit;  // bound of the waits that can give up, in cycles
};
WaitControls wait_controls();

}  // namespace wf
