/*
 * WaveFilter CPU oracle — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded C implementation of what the WaveFilter hot
 * path computes (Section 3, Eq. 5-11, Algorithm 1), in fp64 unless a function
 * says otherwise.  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg may call it; the product library never links or loads it.
 * It shares no code, header or constant with the CUDA library.
 *
 * Conventions (one (batch, head) unit at a time):
 *   - a key/query/value matrix is row-major [rows][d] (token t is row t);
 *   - the coefficient pyramid stores the approximation rows of levels
 *     1..L back to back: level b starts at row n - n/2^(b-1) and holds n/2^b
 *     rows (pyramid_row_offset());
 *   - keep[b] (b = 1..L) is the number of level-b coefficients kept by the
 *     Top-K of Eq. 9 at scale b; keep[0] is the final token count k.
 *
 * Readings of the paper that the oracle fixes, as visible in these
 * signatures: Haar pairs tokens (2j, 2j+1) (forced by the blocks of
 * Eq. 10); orthonormal Haar taps 1/sqrt(2); the softmax of Eq. 7 runs over the
 * current candidates; W of Eq. 8 sums over the query rows; ties in the Top-K
 * of Eq. 9 go to the lower index; a level-0 trim keeps the top keep[0] tokens
 * when keep[0] < 2*keep[1].
 */
#ifndef WF_ORACLE_H
#define WF_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Row offset of level b (1..L) inside a pyramid of an n-token sequence. */
int64_t orc_pyramid_row_offset(int64_t n, int b);
/* Total pyramid rows for levels 1..L: n - n/2^L. */
int64_t orc_pyramid_rows(int64_t n, int L);

/* Eq. 5 applied L times (Section 2.2 recursion): approximation rows of every
 * level into A (pyramid layout) and detail rows into D (same layout).  fp64. */
int orc_haar_analysis_f64(const double* x, int64_t n, int d, int L, double* A, double* D);

/* Inverse of orc_haar_analysis_f64: rebuild the n x d signal from A_L (the
 * last n/2^L rows of the A pyramid) and the detail pyramid D.  fp64. */
int orc_haar_synthesis_f64(const double* A, const double* D, int64_t n, int d, int L, double* x);

/* The coefficient pyramid as the library stores it: the level cascade of
 * Eq. 5 evaluated in fp32 (one fp32 add of the pair, then one fp32 multiply
 * by fl32(1/sqrt 2), no fused multiply-add), each stored value rounded to the
 * storage type (store_bf16 != 0: bfloat16, round to nearest even, returned
 * widened to float; else fp32).  The cascade itself keeps the unrounded fp32
 * values. */
int orc_haar_pyramid_spec32(const float* x, int64_t n, int d, int L, int store_bf16, float* A);

/* Round an fp32 value to bfloat16 (round to nearest, ties to even) and widen
 * it back to fp32. */
float orc_round_bf16(float f);

/* Eq. 7 and Eq. 8 on an explicit candidate row set: logits Q rows^T / sqrt(d)
 * (q x m), softmax along the m candidates of each query row, W_j = sum over
 * the q query rows.  fp64. */
int orc_skim_weights_f64(const double* Q, int q, int d, const double* rows, int64_t m, double* W);

/* Default kept counts: m = (k/n)^(1/L); for b = L..2, keep[b] =
 * ceil(m * |C_b|) clamped to [1, |C_b|], |C_L| = n/2^L, |C_{b-1}| = 2 keep[b];
 * keep[1] = ceil(k/2); keep[0] = k.  Returns 0, or -1 if infeasible. */
int orc_default_schedule(int64_t n, int L, int64_t k, int32_t* keep);

/* Kept counts from the per-scale proportions m_b of Eq. 9 (m[b], b = 1..L;
 * m[0] unused): keep[b] = ceil(m_b |C_b|) clamped to [1, |C_b|];
 * keep[0] = 2 keep[1] (no trim).  Returns 0, or -1 on a bad proportion. */
/* Token level as its own selection step: m = (k/n)^(1/(L+1)) for the L
 * pyramid scans and the token scan; keep[0] = k of the 2 keep[1] tokens. */
int orc_level0_schedule(int64_t n, int L, int64_t k, int32_t* keep);
int orc_schedule_from_proportions(int64_t n, int L, const double* m, int32_t* keep);

/* Multi-scale recursive filtering (Sections 3.1-3.2, Algorithm 1 inner loop)
 * scoring the stored pyramid `pyr` (fp64 copy of the stored coefficients):
 *   C_L = all level-L coefficients; for b = L..1: W = skim(Q, A_b[C_b]);
 *   J_b = Top-K(W, keep[b]); C_{b-1} = {2j, 2j+1 : j in J_b} (Eq. 10);
 *   then mu0 = C_0, trimmed to keep[0] by scoring raw K[C_0] if smaller.
 * mu0 receives keep[0] token indices ascending.  level_sets (optional)
 * receives J_L.., J_1 and then mu0 back to back (ascending within each).
 * level_w (optional) receives W over C_L, .., C_1 and over C_0 when the trim
 * runs, back to back.  Returns 0, or -1 on invalid arguments. */
int orc_filter_f64(const double* Q, int q, int d, const double* pyr, const double* K, int64_t n,
                   int L, const int32_t* keep, int32_t* mu0, int32_t* level_sets, double* level_w);

/* The same filtering taken literally from Algorithm 1 and Eq. 11: at each
 * scale b the Haar DWT (b levels, fp64) of the gathered token sub-sequence
 * K[mu^b] is recomputed and scored; no pyramid is used.  Same outputs. */
int orc_filter_literal_f64(const double* Q, int q, int d, const double* K, int64_t n, int L,
                           const int32_t* keep, int32_t* mu0, int32_t* level_sets);

/* Other wavelet bases (Eq. 6 and Eq. 11 with a generic psi), periodized.
 * An orthogonal two-channel filter bank of `taps` coefficients: low-pass h,
 * high-pass g.  One analysis level of a periodic signal x of even length len:
 *   a[j] = sum_k h[k] x[(2j + k) mod len],   det[j] = sum_k g[k] x[(2j + k) mod len]
 * (periodization keeps the n / 2^B rows of Eq. 6 for every basis).
 *   ORC_HAAR: h = (1, 1) / sqrt 2, g = (1, -1) / sqrt 2.
 *   ORC_DB2 (Daubechies, two vanishing moments): h = (1 + r, 3 + r, 3 - r, 1 - r) / (4 sqrt 2),
 *     r = sqrt 3, and g[k] = (-1)^k h[3 - k].
 * orc_wavelet_taps fills h and g (4 entries each at most) and returns taps, or -1. */
#define ORC_HAAR 0
#define ORC_DB2 1
int orc_wavelet_taps(int wavelet, double* h, double* g);

/* L periodized analysis levels: A and D in the pyramid layout.  fp64. */
int orc_wavelet_analysis_f64(const double* x, int64_t n, int d, int wavelet, int L, double* A, double* D);
/* Inverse of orc_wavelet_analysis_f64 (each level is an orthogonal map; its
 * inverse is the transpose).  fp64. */
int orc_wavelet_synthesis_f64(const double* A, const double* D, int64_t n, int d, int wavelet, int L,
                              double* x);

/* Level-`level` approximation rows (len >> level of them) of the periodized
 * transform of x under the library's storage rule: an fp32 cascade (Haar:
 * fl32(x0 + x1) * fl32(1 / sqrt 2), as the stored pyramid; other bases:
 * fl32(fl32(h[0]) x0), then fmaf(fl32(h[k]), x_k, acc) for k = 1.. in order,
 * each fused multiply-add rounded once), only the last level rounded
 * (bfloat16, nearest even, when store_bf16; returned widened to float). */
int orc_wavelet_approx_spec32(const float* x, int64_t len, int d, int wavelet, int level, int store_bf16,
                              float* out);

/* Algorithm 1 with a generic psi, taken literally: C_L = all level-L blocks;
 * for b = L..1 the keys of the candidates' blocks, K[mu^b] (2^b tokens per
 * candidate, in candidate order), are transformed (b periodized levels of the
 * gathered sequence, Eq. 11; the whole prompt at b = L, Eq. 6) and the
 * approximation rows scored (Eq. 7-9); C_{b-1} = {2j, 2j+1 : j in J_b}.  Then
 * the level-0 trim as orc_filter_f64.  spec32 = 0: fp64 transform; 1: the
 * storage rule of orc_wavelet_approx_spec32 (keys taken as fp32).  Scoring is
 * fp64.  Outputs as orc_filter_f64 (global block indices per scale). */
int orc_filter_wavelet_f64(const double* Q, int q, int d, const double* K, int64_t n, int L, int wavelet,
                           const int32_t* keep, int spec32, int store_bf16, int32_t* mu0, int32_t* level_sets);

/* softmax(Q Ks^T / sqrt(d)) Vs over m key rows (Eq. 1 / Eq. 3 form).  fp64. */
int orc_attention_f64(const double* Q, int q, int d, const double* Ks, const double* Vs, int64_t m,
                      double* O);

/* Final step of Algorithm 1: K_sparse = [K[mu0]; Kg], V_sparse = [V[mu0]; Vg],
 * O = softmax(Q K_sparse^T / sqrt(d)) V_sparse.  fp64. */
int orc_sparse_attn_f64(const double* Q, int q, int d, const double* K, const double* V,
                        const int32_t* mu0, int64_t k, const double* Kg, const double* Vg,
                        int64_t ng, double* O);

#ifdef __cplusplus
}
#endif
#endif
