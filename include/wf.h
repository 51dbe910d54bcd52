/*
 * libwf — WaveFilter hot path on GB300 (sm_103a), C ABI.
 *
 * WaveFilter (Sections 3.1-3.2, Algorithm 1) replaces the cached attention of
 * Eq. 3 for one denoising block by four steps, all implemented here as CUDA
 * kernels:
 *   1. a multi-level Haar DWT of the cached prompt keys along the token axis
 *      (Eq. 5, Eq. 6)                                       -> wf_dwt_build
 *   2. a coarse "skim": perception weights of the query block against the
 *      scale-B approximation coefficients and their column sums (Eq. 7, 8)
 *   3. a multi-scale "scan": Top-K of the weights at each scale, mapped to the
 *      next finer scale (Eq. 9, 10, 11), down to token positions mu^0
 *                                                            -> wf_filter
 *   4. attention of the query block over [K[mu^0]; K[I_g]], [V[mu^0]; V[I_g]]
 *      (Algorithm 1, final step)                             -> wf_sparse_attn
 * and wf_step runs 1 (optionally) + 2-3 + 4 as one stream-ordered call.
 * Around them: wf_cache_update (new rows into the caches with the touched
 * pyramid blocks refreshed), the kept-count schedules (wf_default_schedule,
 * wf_level0_schedule, wf_schedule_from_proportions), other wavelet bases
 * with Eq. 11 taken literally (wf_wavelet_approx, wf_filter_wavelet), grouped
 * query heads (wf_filter, wf_sparse_attn, wf_step), and
 * wf_sparse_attn_noalloc for callers that cannot pass a workspace.
 *
 * Conventions shared by every entry point
 * - A tensor is described by wf_tensor: [batch, heads, seq, head_dim] with
 *   element strides for the first three axes; the head_dim axis is
 *   contiguous.  BHSD and BSHD layouts are both expressible.
 * - Pointers named Q, K, V, Kg, Vg, O, coeffs, idx, level_sets, ws are DEVICE
 *   pointers owned by the caller; libwf allocates no device memory and keeps
 *   no state between calls.  Arrays named keep and m are HOST arrays.
 * - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *   stream).  Every call only enqueues work on that stream and returns; the
 *   outputs are valid once the stream reaches that point.
 * - Every argument is checked on the host before anything is launched; a
 *   failed check returns a negative wf_status and enqueues nothing.  A failed
 *   launch returns WF_ERR_CUDA.  Every device-side wait (the fused kernel's
 *   and the tensor-core kernels') is bounded, so no call can hang the device;
 *   a wait that gives up sets the status word read by wf_workspace_status.
 * - Supported: dtype WF_F32 or WF_BF16 (Q, K, V, Kg, Vg, coeffs and O all of
 *   the same dtype); head_dim 64 or 128; 1 <= query rows <= 64 per query head
 *   (at most 256 per key head when query heads are grouped); prompt length
 *   n a multiple of 2^levels with 1 <= levels <= 10; base pointers and the
 *   three strides (in bytes) 16-byte aligned.
 */
#ifndef WF_H
#define WF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  WF_OK = 0,
  WF_ERR_INVALID_ARG = -1, /* NULL pointer where one is required, bad count */
  WF_ERR_SHAPE = -2,       /* shapes disagree, unsupported head_dim, n % 2^L != 0 */
  WF_ERR_DTYPE = -3,       /* unknown dtype or mixed dtypes */
  WF_ERR_ALIGN = -4,       /* pointer or stride not 16-byte aligned */
  WF_ERR_WORKSPACE = -5,   /* workspace or coefficient buffer too small */
  WF_ERR_CUDA = -6,        /* a CUDA runtime call or launch failed */
  WF_ERR_TIMEOUT = -7,     /* a bounded device-side wait gave up */
  WF_ERR_UNSUPPORTED = -8, /* valid request outside what this build implements */
  WF_ERR_SCHEDULE = -9     /* kept counts infeasible for the shape */
} wf_status;

typedef enum { WF_F32 = 0, WF_BF16 = 1 } wf_dtype;

typedef struct {
  int32_t batch;    /* B */
  int32_t heads;    /* H */
  int32_t seq;      /* rows per (batch, head): n for K/V, q for Q/O, n_g for Kg/Vg */
  int32_t head_dim; /* d */
  int64_t stride_b; /* elements between consecutive batch entries */
  int64_t stride_h; /* elements between consecutive heads */
  int64_t stride_s; /* elements between consecutive rows */
  int32_t dtype;    /* wf_dtype */
} wf_tensor;

/* Human-readable name of a status code (static string). */
const char* wf_status_str(int status);

/* ---------------------------------------------------------------------------
 * 1. DWT pyramid (Eq. 5 recursion of Section 2.2; Eq. 6 keys only).
 *
 * For every (batch b, head h) the level cascade a_0 = K[b,h],
 *   a_l[j] = (a_{l-1}[2j] + a_{l-1}[2j+1]) * (1/sqrt 2),   l = 1..levels,
 * is evaluated in fp32 (one fp32 add, one fp32 multiply by fl32(1/sqrt 2),
 * no fused multiply-add) and each a_l row is stored rounded to the key dtype
 * (bf16: round to nearest even).  Coefficient j of level l pairs tokens
 * [2^l j, 2^l (j+1)) (the blocks of Eq. 10); the taps are the orthonormal Haar
 * pair of Table 3.  Detail coefficients are not stored: filtering only reads
 * approximations.
 *
 * coeffs layout (contiguous, dtype of K): unit u = b*H + h owns
 * R = n - n/2^levels rows of head_dim elements starting at row u*R; inside it
 * level l starts at row n - n/2^(l-1) and has n/2^l rows.
 *
 * V must be NULL: Section 3.1 decomposes the cache keys only.
 * Errors: WF_ERR_WORKSPACE if coeffs_bytes < wf_coeffs_bytes(kv, levels).
 * ------------------------------------------------------------------------- */
size_t wf_coeffs_bytes(const wf_tensor* kv, int levels); /* 0 if invalid */
wf_status wf_dwt_build(const void* K, const void* V, const wf_tensor* kv, int levels, void* coeffs,
                       size_t coeffs_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * Cache update with an incremental pyramid refresh (the step before the build
 * in Algorithm 1 when only part of the cached prompt changed, Eq. 4's cache
 * refresh applied to a window): writes the count = nt->seq new key rows Knew
 * (and value rows Vnew) into K (and V) at token positions [pos, pos + count),
 * and in the same kernel recomputes every pyramid coefficient whose block
 * contains one of those positions (Eq. 5-6): coeffs then equals wf_dwt_build
 * of the updated K, bit for bit.  The kernel reads the aligned 2^L-token
 * blocks that hold the new rows, writes the new rows and those blocks'
 * coefficients, and touches nothing else.
 *   Knew, Vnew: device, [B, H, count, d] (nt: same batch, heads, head_dim and
 *               dtype as kv); Vnew and V are both NULL to update keys only.
 *               They must not overlap K, V or coeffs.
 *   K, V: the caches (kv), updated in place; coeffs: the pyramid of K.
 * Errors: WF_ERR_INVALID_ARG for a missing pointer, Vnew/V given alone, or a
 * window outside [0, n); shape, dtype, alignment and size errors as in
 * wf_dwt_build.  Nothing is enqueued on an error.
 * ------------------------------------------------------------------------- */
wf_status wf_cache_update(const void* Knew, const void* Vnew, const wf_tensor* nt, void* K, void* V,
                          const wf_tensor* kv, int64_t pos, int levels, void* coeffs, size_t coeffs_bytes,
                          void* stream);

/* ---------------------------------------------------------------------------
 * Kept counts (Eq. 9 "proportion m_B").  keep has levels+1 entries: keep[l]
 * = number of level-l coefficients kept (l = 1..levels), keep[0] = final
 * number of prompt tokens k.  Feasible iff 1 <= keep[L] <= n/2^L,
 * 1 <= keep[l] <= 2 keep[l+1], 1 <= keep[0] <= 2 keep[1].
 *
 * wf_default_schedule: one proportion m = (k/n)^(1/L) for every scale:
 *   keep[l] = min(|C_l|, max(1, ceil(m |C_l|))) for l = L..2 with
 *   |C_L| = n/2^L, |C_{l-1}| = 2 keep[l]; keep[1] = ceil(k/2); keep[0] = k.
 * wf_schedule_from_proportions: per-scale proportions m[l] in (0, 1]
 *   (m[0] unused): keep[l] = min(|C_l|, max(1, ceil(m[l] |C_l|))),
 *   keep[0] = 2 keep[1].
 * wf_level0_schedule: the reading in which the token level is a selection
 *   step of its own (Algorithm 1's last scan over raw keys): one proportion
 *   m = (k/n)^(1/(L+1)) for the L pyramid scales and for the tokens,
 *   keep[l] = min(|C_l|, max(1, ceil(m |C_l|))) for l = L..1, keep[0] = k
 *   kept out of the 2 keep[1] token candidates (a level-0 selection
 *   whenever k < 2 keep[1]).
 * "ceil" ignores a product that exceeds an integer by less than 1e-9.
 * Host-only; return WF_ERR_SCHEDULE if no feasible schedule exists.
 * ------------------------------------------------------------------------- */
wf_status wf_default_schedule(int64_t n, int levels, int64_t k, int32_t* keep);
wf_status wf_schedule_from_proportions(int64_t n, int levels, const double* m, int32_t* keep);
wf_status wf_level0_schedule(int64_t n, int levels, int64_t k, int32_t* keep);

/* ---------------------------------------------------------------------------
 * 2-3. Skim and scan (Eq. 7-11, Algorithm 1 inner loop).
 *
 * For every unit, with C_L = {0..n/2^L - 1} and for l = L..1:
 *   logits  s_ij = Q_i . A_l[j] / sqrt(d)           (j in C_l; fp32)
 *   P       = softmax over j in C_l of each query row (Eq. 7)
 *   W_j     = sum_i P_ij                            (Eq. 8)
 *   J_l     = the keep[l] candidates of largest W (ties: lower index)  (Eq. 9)
 *   C_{l-1} = {2j, 2j+1 : j in J_l}                 (Eq. 10-11)
 * C_0 holds 2 keep[1] token positions; if keep[0] < 2 keep[1] the same
 * scoring on the raw keys K[C_0] keeps the top keep[0] of them.
 *
 * Inputs: Q [B,Hq,q,d] (descriptor q), coeffs from wf_dwt_build on K with
 * the same levels, K [B,H,n,d] (descriptor kv; read only by the level-0 trim).
 * Grouped-query attention: Hq may be any multiple G of the H key heads.
 * Query head h G + g (g < G) belongs to key head h. A unit is one (batch,
 * key head), and its query rows i are the q rows of each of its G query
 * heads: Eq. 7's softmax is per row, and Eq. 8's sum runs over all G q rows,
 * so one selection serves the whole group. Limits: q <= 64 and G q <= 256
 * (else WF_ERR_UNSUPPORTED); Hq not a multiple of H gives WF_ERR_SHAPE.
 * keep: host array of levels+1 counts (e.g. from wf_default_schedule).
 * Outputs: idx int32 [B*H][keep[0]] token positions, ascending per unit.
 * level_sets (optional, NULL to skip): int32
 * [B*H][keep[L] + .. + keep[1] + keep[0]] = J_L, .., J_1, mu^0 per unit.
 * ws: device scratch of at least wf_filter_workspace_bytes() bytes,
 * 256-byte aligned.  Its first 4 bytes are a status word: for bf16 keys with
 * head_dim 128 the scores run on the tensor cores, and a kernel whose bounded
 * wait gives up (it never should) sets the word and leaves the outputs
 * undefined; wf_workspace_status() reads and clears it.  Zero the word once
 * before the first call; the rest of ws may hold anything.
 * ------------------------------------------------------------------------- */
size_t wf_filter_workspace_bytes(const wf_tensor* q, const wf_tensor* kv, int levels, const int32_t* keep);
wf_status wf_filter(const void* Q, const wf_tensor* q, const void* coeffs, const void* K, const wf_tensor* kv,
                    int levels, const int32_t* keep, int32_t* idx, int32_t* level_sets, void* ws,
                    size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * 2-3'. Other wavelet bases (Eq. 6 and Eq. 11 with a generic psi).
 *
 * With a basis other than Haar the transform of the gathered sub-sequence in
 * Eq. 11 is no longer the pyramid indexed at the candidates, so these calls
 * take Algorithm 1 literally: at scale b the keys of the candidates' blocks
 * (2^b tokens each, in candidate order) form one sequence, taken as
 * periodic, and b levels of the periodized DWT give one approximation row
 * per candidate.  Periodization keeps the n / 2^B rows of Eq. 6 for every
 * basis.  One analysis level is a[j] = sum_k h[k] x[(2j + k) mod len] with
 *   WF_WAVELET_HAAR: h = (1, 1) / sqrt 2;
 *   WF_WAVELET_DB2:  Daubechies' filter with two vanishing moments,
 *                    h = (1 + r, 3 + r, 3 - r, 1 - r) / (4 sqrt 2), r = sqrt 3.
 * Arithmetic: an fp32 cascade (Haar: fl32(x0 + x1) * fl32(1 / sqrt 2), the
 * rule of wf_dwt_build; db2: fl32(fl32(h[0]) x0), then fused multiply-adds
 * with fl32(h[1]), fl32(h[2]), fl32(h[3]) in that order), the last level
 * rounded to the key dtype.
 *
 * wf_wavelet_approx: the level-`level` rows of the keys of blocks
 * [2^level c, 2^level (c + 1)) for the m candidates c of every unit.
 * cand: device int32 [B*H][m] block indices at that scale (the sequence
 * follows their order; entries outside [0, n >> level) are clamped), or NULL
 * for all m = n >> level blocks in order (the whole prompt, Eq. 6).
 * out: device [B*H][m][d] in the key dtype, at least B*H*m*d elements.
 * level: 1..10 for Haar, 1..8 for db2; n a multiple of 2^level.
 *
 * wf_filter_wavelet: Eq. 7-11 with the basis `wavelet`.  The scale-L rows are
 * `top` (wf_wavelet_approx with cand = NULL and level = levels, i.e.
 * [B*H][n >> levels][d], recomputed whenever K changes); the rows of every
 * finer scale are the transform of its candidates' gathered blocks.  Scores,
 * Top-K, children and the level-0 trim, the query grouping rules, limits and
 * outputs are those of wf_filter; with WF_WAVELET_HAAR the results equal
 * wf_filter's.  ws: at least wf_filter_wavelet_workspace_bytes() bytes,
 * 256-byte aligned, with wf_filter's status word in its first 4 bytes.
 * ------------------------------------------------------------------------- */
#define WF_WAVELET_HAAR 0
#define WF_WAVELET_DB2 1
wf_status wf_wavelet_approx(const void* K, const wf_tensor* kv, const int32_t* cand, int m, int level, int wavelet,
                            void* out, size_t out_bytes, void* stream);
size_t wf_filter_wavelet_workspace_bytes(const wf_tensor* q, const wf_tensor* kv, int levels, const int32_t* keep,
                                         int wavelet);
wf_status wf_filter_wavelet(const void* Q, const wf_tensor* q, const void* top, const void* K, const wf_tensor* kv,
                            int levels, const int32_t* keep, int wavelet, int32_t* idx, int32_t* level_sets,
                            void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * 4. Sparse attention (Algorithm 1, final step; Eq. 3 form).
 *
 * For every query head (b, hq), with key head h = hq / G (G = Hq / H, as in
 * wf_filter): K_s = [K[idx[b H + h][0..k)]; Kg], V_s likewise from V and Vg
 * (both at key head h), and
 *   O = softmax(Q K_s^T * scale) V_s      (fp32 logits, softmax, accumulation)
 * with scale = 1/sqrt(d) when the argument is 0.  No mask (the DLMs attend
 * bidirectionally).  Q: [B,Hq,q,d], q <= 64.  K, V: [B,H,n,d].
 * idx: int32 [B*H][k], each entry in [0, n) (any order).
 * Kg, Vg: [B,H,n_g,d] (descriptor g, may be NULL when n_g = 0).  O: [B,Hq,q,d]
 * (descriptor o: same shape and dtype as Q), written rounded to that dtype.
 * ws: device scratch of at least wf_attn_workspace_bytes() bytes, 256-byte
 * aligned; as for wf_filter, its first 4 bytes are a status word set if a
 * tensor-core kernel's bounded wait gives up (bf16 keys with head_dim 128 run
 * on the tensor cores): zero it once, read it with wf_workspace_status().
 * Out-of-range idx entries are clamped to [0, n) (never read out of bounds).
 * ------------------------------------------------------------------------- */
size_t wf_attn_workspace_bytes(const wf_tensor* q, int k, int n_g);
wf_status wf_sparse_attn(const void* Q, const wf_tensor* q, const void* K, const void* V, const wf_tensor* kv,
                         const int32_t* idx, int k, const void* Kg, const void* Vg, const wf_tensor* g, void* O,
                         const wf_tensor* o, float scale, void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * 4'. Sparse attention without a caller workspace.  The paper has no
 * counterpart to this call: it exists for callers that cannot allocate device
 * memory (for example a plugin inside a host engine that owns every device
 * allocation and offers no scratch, or code on a path where allocating after
 * start-up is not allowed) and therefore cannot pass the ws buffer that
 * wf_sparse_attn needs.
 *
 * Same arguments, semantics and results as wf_sparse_attn, minus ws and
 * ws_bytes.  The split-K scratch comes from one static device array of
 * WF_NOALLOC_SCRATCH_BYTES inside libwf, reserved in every CUDA context that
 * loads the library until that context is destroyed (the runtime's primary
 * context: until the process exits); the call allocates nothing.
 * - Limit: returns WF_ERR_WORKSPACE, and launches nothing, when the call would
 *   need more than WF_NOALLOC_SCRATCH_BYTES (the need is
 *   wf_attn_workspace_bytes(q, k, n_g); e.g. 32 heads with head_dim 128 fit
 *   k + n_g <= 1984 rows with query blocks of at most 32 rows, 960 rows with
 *   33 to 64).
 * - Contexts: the array has its own device address in each CUDA context.  The
 *   first call from a context (the runtime's primary context of the current
 *   device, or any context the caller made current) looks that address up
 *   with cudaGetSymbolAddress and caches it under the context's unique id;
 *   later calls from the same context reuse it.  Make that first call before
 *   any stream capture.  It returns WF_ERR_CUDA if the lookup fails.
 * - All calls in a context share the one array and each call overwrites it:
 *   calls whose kernels may overlap on the GPU (other streams, other host
 *   threads) race and corrupt each other's results.  Serialise them, e.g.
 *   on one stream.  No part of the array has to start at zero, except the
 *   status word below (zero when the library loads).
 * - The array's first word is the status word of the tensor-core kernels: if
 *   one of their bounded waits gives up (it never should), the output is
 *   undefined and the word is set.  wf_noalloc_status() waits for `stream`,
 *   returns WF_ERR_TIMEOUT (and clears the word) if it is set, else WF_OK.
 *   Synchronising; not for the hot loop.
 * ------------------------------------------------------------------------- */
#define WF_NOALLOC_SCRATCH_BYTES (16u << 20)
wf_status wf_sparse_attn_noalloc(const void* Q, const wf_tensor* q, const void* K, const void* V,
                                 const wf_tensor* kv, const int32_t* idx, int k, const void* Kg, const void* Vg,
                                 const wf_tensor* g, void* O, const wf_tensor* o, float scale, void* stream);
wf_status wf_noalloc_status(void* stream);

/* ---------------------------------------------------------------------------
 * One denoising-step layer (Algorithm 1 body): if refresh_coeffs != 0, first
 * rebuild coeffs from K (wf_dwt_build); then the skim/scan filter and the
 * sparse attention with scale 1/sqrt(d), writing idx (and level_sets, if not
 * NULL) and O exactly as wf_filter + wf_sparse_attn define them.  Same
 * arguments and rules as those calls; ws must hold wf_step_workspace_bytes().
 *
 * For bf16 with head_dim 128, at most 32 query rows and one query head per
 * key head, the filter and the attention run as one fused kernel (one
 * thread-block cluster per (batch, head)).  Grouped query heads with bf16,
 * head_dim 128, at most 32 rows a query head and at most 256 stacked rows a
 * key head run the grouped filter kernel (one cluster per (batch, key head),
 * the stacked rows as the MMA columns), then the tensor-core attention.
 * Other shapes run the per-stage kernels.  The fused kernels' waits
 * (on copies, tensor-core completion and the cluster's exchanges) are
 * bounded: if one gives up (it never should), the kernel returns early,
 * outputs are undefined, and a status word in the first 4 bytes of ws is set;
 * wf_workspace_status() reports and clears it.  wf_step never clears the word
 * itself (so a failure stays visible across calls): zero those 4 bytes once
 * before the first call (or call wf_workspace_status once).
 * ------------------------------------------------------------------------- */
size_t wf_step_workspace_bytes(const wf_tensor* q, const wf_tensor* kv, int levels, const int32_t* keep,
                               int n_g);
wf_status wf_step(const void* Q, const wf_tensor* q, const void* K, const void* V, const wf_tensor* kv,
                  const void* Kg, const void* Vg, const wf_tensor* g, void* coeffs, size_t coeffs_bytes,
                  int refresh_coeffs, int levels, const int32_t* keep, int32_t* idx, int32_t* level_sets,
                  void* O, const wf_tensor* o, void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * One layer on the literal path (Eq. 11 with the basis `wavelet`, as
 * wf_filter_wavelet): the filter, then the sparse attention with scale
 * 1/sqrt(d), writing idx (and level_sets, if not NULL) and O exactly as
 * wf_filter_wavelet + wf_sparse_attn define them.  top: the scale-L rows of
 * the whole prompt (wf_wavelet_approx with cand = NULL, level = levels),
 * recomputed by the caller whenever K changes.  Other arguments and rules as
 * for wf_step; ws: at least wf_step_wavelet_workspace_bytes() bytes, 256-byte
 * aligned, with the status word of wf_step in its first 4 bytes.
 *
 * For bf16 with head_dim 128, at most 32 query rows and one query head per
 * key head, every scale runs on wf_step's fused kernel: one launch per scale,
 * after the transform of that scale's candidate blocks, with the previous
 * selection handed over in ws; the last launch also runs the attention.
 * wf_filter_wavelet takes the same fused launches (without the attention)
 * for those shapes.  Other shapes run the per-stage kernels.
 * ------------------------------------------------------------------------- */
size_t wf_step_wavelet_workspace_bytes(const wf_tensor* q, const wf_tensor* kv, int levels, const int32_t* keep,
                                       int wavelet, int n_g);
wf_status wf_step_wavelet(const void* Q, const wf_tensor* q, const void* top, const void* K, const void* V,
                          const wf_tensor* kv, const void* Kg, const void* Vg, const wf_tensor* g, int levels,
                          const int32_t* keep, int wavelet, int32_t* idx, int32_t* level_sets, void* O,
                          const wf_tensor* o, void* ws, size_t ws_bytes, void* stream);

/* Device status of the last wf_step calls that used workspace ws: waits for
 * `stream`, returns WF_ERR_TIMEOUT (and clears the word) if a bounded device
 * wait gave up, else WF_OK.  Synchronising; not for the hot loop. */
wf_status wf_workspace_status(void* ws, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* WF_H */
