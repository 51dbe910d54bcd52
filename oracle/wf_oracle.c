/*
 * WaveFilter CPU oracle — TEST INFRASTRUCTURE ONLY (see wf_oracle.h).
 *
 * Plain single-threaded C, fp64 unless stated.  Written from the paper:
 * Eq. 5 (filter-bank DWT), the recursion of Section 2.2, Eq. 6-11 and
 * Algorithm 1.  Built with -ffp-contract=off so that no multiply-add is
 * fused and results are the same on every host.
 */
#include "wf_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Haar filter bank (Eq. 5, "Haar" of Table 3).                              */
/*                                                                          */
/* Eq. 5 writes A_1[n] = sum_k x[k] g[2n-k].  Eq. 10 fixes the coefficient j */
/* of scale B to the token block [2^B j, 2^B (j+1)), so coefficient n pairs  */
/* tokens (2n, 2n+1); with two-tap filters that is the sum                   */
/* sum_k x[k] f[2n+1-k] over k in {2n, 2n+1}.                                */
/* Orthonormal Haar taps: g = {c, c}, h = {-c, c}, c = 1/sqrt(2), so         */
/* A[n] = c (x[2n] + x[2n+1]) and D[n] = c (x[2n] - x[2n+1]).                */
/* ------------------------------------------------------------------------ */
#define HAAR_C 0.70710678118654752440
static const double HAAR_G[2] = {HAAR_C, HAAR_C};
static const double HAAR_H[2] = {-HAAR_C, HAAR_C};

int64_t orc_pyramid_row_offset(int64_t n, int b) { return n - (n >> (b - 1)); }
int64_t orc_pyramid_rows(int64_t n, int L) { return n - (n >> L); }

static int shape_ok(int64_t n, int d, int L) {
  if (n <= 0 || d <= 0 || L < 1 || L > 30) return 0;
  if ((n >> L) <= 0 || ((n >> L) << L) != n) return 0;
  return 1;
}

/* One analysis step of Eq. 5 on a len x d signal: len/2 approximation and
 * detail rows. */
static void analysis_step(const double* x, int64_t len, int d, double* a, double* det) {
  for (int64_t m = 0; m < len / 2; ++m) {
    for (int c = 0; c < d; ++c) {
      double sa = 0.0, sd = 0.0;
      for (int64_t k = 2 * m; k <= 2 * m + 1; ++k) {
        sa += x[k * d + c] * HAAR_G[2 * m + 1 - k];
        sd += x[k * d + c] * HAAR_H[2 * m + 1 - k];
      }
      a[m * d + c] = sa;
      det[m * d + c] = sd;
    }
  }
}

int orc_haar_analysis_f64(const double* x, int64_t n, int d, int L, double* A, double* D) {
  if (!shape_ok(n, d, L) || !x || !A || !D) return -1;
  /* Section 2.2: level 1 filters the signal; level b filters A_{b-1}. */
  const double* src = x;
  for (int b = 1; b <= L; ++b) {
    int64_t off = orc_pyramid_row_offset(n, b);
    int64_t len_in = n >> (b - 1);
    analysis_step(src, len_in, d, A + off * d, D + off * d);
    src = A + off * d;
  }
  return 0;
}

int orc_haar_synthesis_f64(const double* A, const double* D, int64_t n, int d, int L, double* x) {
  if (!shape_ok(n, d, L) || !A || !D || !x) return -1;
  /* Synthesis bank of the orthonormal Haar pair: x[2m] = c (a[m] + d[m]),
   * x[2m+1] = c (a[m] - d[m]), from scale L down to the signal. */
  int64_t rows_l = n >> L;
  double* cur = (double*)malloc(sizeof(double) * (size_t)n * d);
  double* nxt = (double*)malloc(sizeof(double) * (size_t)n * d);
  if (!cur || !nxt) { free(cur); free(nxt); return -1; }
  memcpy(cur, A + orc_pyramid_row_offset(n, L) * d, sizeof(double) * (size_t)rows_l * d);
  for (int b = L; b >= 1; --b) {
    int64_t len = n >> b;
    const double* det = D + orc_pyramid_row_offset(n, b) * d;
    for (int64_t m = 0; m < len; ++m) {
      for (int c = 0; c < d; ++c) {
        nxt[(2 * m) * d + c] = HAAR_C * (cur[m * d + c] + det[m * d + c]);
        nxt[(2 * m + 1) * d + c] = HAAR_C * (cur[m * d + c] - det[m * d + c]);
      }
    }
    double* t = cur; cur = nxt; nxt = t;
  }
  memcpy(x, cur, sizeof(double) * (size_t)n * d);
  free(cur);
  free(nxt);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Storage precision (the library's stored pyramid).                        */
/* ------------------------------------------------------------------------ */
float orc_round_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  if ((u & 0x7f800000u) == 0x7f800000u) {
    /* Inf stays Inf; NaN stays a (quiet) NaN. */
    if (u & 0x007fffffu) u |= 0x00400000u;
    u &= 0xffff0000u;
  } else {
    /* Round to nearest, ties to even, on the 16 dropped bits. */
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7fffu + lsb;
    u &= 0xffff0000u;
  }
  memcpy(&f, &u, sizeof f);
  return f;
}

int orc_haar_pyramid_spec32(const float* x, int64_t n, int d, int L, int store_bf16, float* A) {
  if (!shape_ok(n, d, L) || !x || !A) return -1;
  const float c32 = (float)HAAR_C; /* fl32(1/sqrt 2) */
  /* Unrounded fp32 cascade values of the previous level. */
  float* prev = (float*)malloc(sizeof(float) * (size_t)n * d);
  float* cur = (float*)malloc(sizeof(float) * (size_t)(n / 2) * d);
  if (!prev || !cur) { free(prev); free(cur); return -1; }
  memcpy(prev, x, sizeof(float) * (size_t)n * d);
  for (int b = 1; b <= L; ++b) {
    int64_t len = n >> b;
    float* out = A + orc_pyramid_row_offset(n, b) * d;
    for (int64_t m = 0; m < len; ++m) {
      for (int c = 0; c < d; ++c) {
        float s = prev[(2 * m) * d + c] + prev[(2 * m + 1) * d + c];
        float v = s * c32;
        cur[m * d + c] = v;
        out[m * d + c] = store_bf16 ? orc_round_bf16(v) : v;
      }
    }
    memcpy(prev, cur, sizeof(float) * (size_t)len * d);
  }
  free(prev);
  free(cur);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Eq. 7 - Eq. 9: perception weights, importance vector, Top-K.             */
/* ------------------------------------------------------------------------ */
int orc_skim_weights_f64(const double* Q, int q, int d, const double* rows, int64_t m, double* W) {
  if (!Q || !rows || !W || q <= 0 || d <= 0 || m <= 0) return -1;
  double* A = (double*)malloc(sizeof(double) * (size_t)q * m);
  if (!A) return -1;
  const double sqrt_d = sqrt((double)d);
  /* Eq. 7: A = Softmax(Q K_low^T / sqrt(d)), one softmax per query row over
   * the candidate columns. */
  for (int i = 0; i < q; ++i) {
    double* row = A + (size_t)i * m;
    for (int64_t j = 0; j < m; ++j) {
      double s = 0.0;
      for (int c = 0; c < d; ++c) s += Q[(size_t)i * d + c] * rows[(size_t)j * d + c];
      row[j] = s / sqrt_d;
    }
    double mx = row[0];
    for (int64_t j = 1; j < m; ++j) if (row[j] > mx) mx = row[j];
    double z = 0.0;
    for (int64_t j = 0; j < m; ++j) { row[j] = exp(row[j] - mx); z += row[j]; }
    for (int64_t j = 0; j < m; ++j) row[j] /= z;
  }
  /* Eq. 8: column-wise sum, i.e. over the query rows. */
  for (int64_t j = 0; j < m; ++j) {
    double w = 0.0;
    for (int i = 0; i < q; ++i) w += A[(size_t)i * m + j];
    W[j] = w;
  }
  free(A);
  return 0;
}

typedef struct {
  double w;
  int32_t idx;
} scored_t;

/* Order of Eq. 9's Top-K: larger W first; equal W -> lower index first. */
static int cmp_score_desc(const void* a, const void* b) {
  const scored_t* x = (const scored_t*)a;
  const scored_t* y = (const scored_t*)b;
  if (x->w > y->w) return -1;
  if (x->w < y->w) return 1;
  return (x->idx > y->idx) - (x->idx < y->idx);
}

static int cmp_i32(const void* a, const void* b) {
  int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
  return (x > y) - (x < y);
}

/* Top-K of Eq. 9 over candidates idx[0..m) with weights W: writes the kk
 * chosen indices, ascending. */
static void topk_ascending(const double* W, const int32_t* idx, int64_t m, int64_t kk, int32_t* out) {
  scored_t* s = (scored_t*)malloc(sizeof(scored_t) * (size_t)m);
  for (int64_t j = 0; j < m; ++j) { s[j].w = W[j]; s[j].idx = idx[j]; }
  qsort(s, (size_t)m, sizeof(scored_t), cmp_score_desc);
  for (int64_t j = 0; j < kk; ++j) out[j] = s[j].idx;
  qsort(out, (size_t)kk, sizeof(int32_t), cmp_i32);
  free(s);
}

/* ------------------------------------------------------------------------ */
/* Kept counts.                                                             */
/* ------------------------------------------------------------------------ */
static int64_t ceil_guarded(double v) {
  /* ceil, with products that land on an integer up to pow() rounding kept
   * exact (e.g. 0.5 * 2048 must give 1024, not 1025). */
  return (int64_t)ceil(v - 1e-9);
}

int orc_default_schedule(int64_t n, int L, int64_t k, int32_t* keep) {
  if (!shape_ok(n, 1, L) || !keep || k < 1 || k > n) return -1;
  double m = pow((double)k / (double)n, 1.0 / (double)L);
  int64_t cnt = n >> L;
  for (int b = L; b >= 2; --b) {
    int64_t kb = ceil_guarded(m * (double)cnt);
    if (kb < 1) kb = 1;
    if (kb > cnt) kb = cnt;
    keep[b] = (int32_t)kb;
    cnt = 2 * kb;
  }
  int64_t k1 = (k + 1) / 2;
  if (k1 > cnt) return -1;
  keep[1] = (int32_t)k1;
  keep[0] = (int32_t)k;
  return 0;
}

/* Token level as a selection step of its own: the same proportion m for the
 * L pyramid scans and for the scan over the 2 k_1 raw-key candidates
 * (Algorithm 1 read with its last scan at level 0), m = (k/n)^(1/(L+1)). */
int orc_level0_schedule(int64_t n, int L, int64_t k, int32_t* keep) {
  if (!shape_ok(n, 1, L) || !keep || k < 1 || k > n) return -1;
  double m = pow((double)k / (double)n, 1.0 / (double)(L + 1));
  int64_t cnt = n >> L;
  for (int b = L; b >= 1; --b) {
    int64_t kb = ceil_guarded(m * (double)cnt);
    if (kb < 1) kb = 1;
    if (kb > cnt) kb = cnt;
    keep[b] = (int32_t)kb;
    cnt = 2 * kb;
  }
  if (k > cnt) return -1;
  keep[0] = (int32_t)k;
  return 0;
}

int orc_schedule_from_proportions(int64_t n, int L, const double* m, int32_t* keep) {
  if (!shape_ok(n, 1, L) || !m || !keep) return -1;
  int64_t cnt = n >> L;
  for (int b = L; b >= 1; --b) {
    if (!(m[b] > 0.0 && m[b] <= 1.0)) return -1;
    int64_t kb = ceil_guarded(m[b] * (double)cnt);
    if (kb < 1) kb = 1;
    if (kb > cnt) kb = cnt;
    keep[b] = (int32_t)kb;
    cnt = 2 * kb;
  }
  keep[0] = 2 * keep[1];
  return 0;
}

static int schedule_ok(int64_t n, int L, const int32_t* keep) {
  int64_t cnt = n >> L;
  for (int b = L; b >= 1; --b) {
    if (keep[b] < 1 || keep[b] > cnt) return 0;
    cnt = 2 * (int64_t)keep[b];
  }
  return keep[0] >= 1 && keep[0] <= cnt;
}

/* ------------------------------------------------------------------------ */
/* Multi-scale recursive filtering.                                         */
/* ------------------------------------------------------------------------ */
int orc_filter_f64(const double* Q, int q, int d, const double* pyr, const double* K, int64_t n,
                   int L, const int32_t* keep, int32_t* mu0, int32_t* level_sets, double* level_w) {
  if (!Q || !pyr || !K || !keep || !mu0 || q <= 0 || !shape_ok(n, d, L)) return -1;
  if (!schedule_ok(n, L, keep)) return -1;
  int64_t cap = n >> L;
  for (int b = L; b >= 1; --b) if (2 * (int64_t)keep[b] > cap) cap = 2 * (int64_t)keep[b];
  int32_t* cand = (int32_t*)malloc(sizeof(int32_t) * (size_t)cap);
  int32_t* chosen = (int32_t*)malloc(sizeof(int32_t) * (size_t)cap);
  double* rows = (double*)malloc(sizeof(double) * (size_t)cap * d);
  double* W = (double*)malloc(sizeof(double) * (size_t)cap);
  if (!cand || !chosen || !rows || !W) { free(cand); free(chosen); free(rows); free(W); return -1; }

  /* mu^B <- I_p: every level-L coefficient is a candidate. */
  int64_t m = n >> L;
  for (int64_t j = 0; j < m; ++j) cand[j] = (int32_t)j;
  int64_t set_pos = 0, w_pos = 0;
  for (int b = L; b >= 1; --b) {
    /* Eq. 11 for Haar: the scale-b approximation of the gathered tokens is
     * the level-b pyramid row of each candidate (an aligned 2^b block). */
    const double* Ab = pyr + orc_pyramid_row_offset(n, b) * d;
    for (int64_t j = 0; j < m; ++j) memcpy(rows + j * d, Ab + (int64_t)cand[j] * d, sizeof(double) * d);
    orc_skim_weights_f64(Q, q, d, rows, m, W);                       /* Eq. 7-8 */
    if (level_w) { memcpy(level_w + w_pos, W, sizeof(double) * (size_t)m); w_pos += m; }
    topk_ascending(W, cand, m, keep[b], chosen);                     /* Eq. 9 */
    if (level_sets) { memcpy(level_sets + set_pos, chosen, sizeof(int32_t) * keep[b]); set_pos += keep[b]; }
    /* Eq. 10: each kept coefficient j covers the two scale-(b-1) units 2j, 2j+1. */
    for (int64_t j = 0; j < keep[b]; ++j) { cand[2 * j] = 2 * chosen[j]; cand[2 * j + 1] = 2 * chosen[j] + 1; }
    m = 2 * (int64_t)keep[b];
  }
  /* mu^0: the 2 keep[1] tokens, trimmed to keep[0] by the same scoring on the
   * raw keys when keep[0] is smaller. */
  if (keep[0] < m) {
    for (int64_t j = 0; j < m; ++j) memcpy(rows + j * d, K + (int64_t)cand[j] * d, sizeof(double) * d);
    orc_skim_weights_f64(Q, q, d, rows, m, W);
    if (level_w) { memcpy(level_w + w_pos, W, sizeof(double) * (size_t)m); w_pos += m; }
    topk_ascending(W, cand, m, keep[0], chosen);
    memcpy(mu0, chosen, sizeof(int32_t) * keep[0]);
  } else {
    memcpy(mu0, cand, sizeof(int32_t) * keep[0]);
  }
  if (level_sets) memcpy(level_sets + set_pos, mu0, sizeof(int32_t) * keep[0]);
  free(cand);
  free(chosen);
  free(rows);
  free(W);
  return 0;
}

int orc_filter_literal_f64(const double* Q, int q, int d, const double* K, int64_t n, int L,
                           const int32_t* keep, int32_t* mu0, int32_t* level_sets) {
  if (!Q || !K || !keep || !mu0 || q <= 0 || !shape_ok(n, d, L)) return -1;
  if (!schedule_ok(n, L, keep)) return -1;
  int32_t* mu = (int32_t*)malloc(sizeof(int32_t) * (size_t)n);       /* token set mu^b */
  double* sub = (double*)malloc(sizeof(double) * (size_t)n * d);      /* K[mu^b] */
  double* A = (double*)malloc(sizeof(double) * (size_t)n * d);
  double* D = (double*)malloc(sizeof(double) * (size_t)n * d);
  int32_t* gidx = (int32_t*)malloc(sizeof(int32_t) * (size_t)n);
  int32_t* chosen = (int32_t*)malloc(sizeof(int32_t) * (size_t)n);
  double* W = (double*)malloc(sizeof(double) * (size_t)n);
  if (!mu || !sub || !A || !D || !gidx || !chosen || !W) {
    free(mu); free(sub); free(A); free(D); free(gidx); free(chosen); free(W);
    return -1;
  }
  /* Algorithm 1: mu^B <- I_p. */
  int64_t len = n;
  for (int64_t t = 0; t < n; ++t) mu[t] = (int32_t)t;
  int64_t set_pos = 0;
  for (int b = L; b >= 1; --b) {
    /* Eq. 11: gather the sub-sequence and take its DWT at scale b. */
    for (int64_t t = 0; t < len; ++t) memcpy(sub + t * d, K + (int64_t)mu[t] * d, sizeof(double) * d);
    orc_haar_analysis_f64(sub, len, d, b, A, D);
    int64_t m = len >> b;
    const double* Ab = A + orc_pyramid_row_offset(len, b) * d;
    /* Coefficient j of the gathered sequence covers mu[2^b j .. 2^b j + 2^b);
     * its index in the scale-b space of the prompt is mu[2^b j] / 2^b. */
    for (int64_t j = 0; j < m; ++j) gidx[j] = mu[j << b] >> b;
    orc_skim_weights_f64(Q, q, d, Ab, m, W);                          /* Eq. 7-8 */
    topk_ascending(W, gidx, m, keep[b], chosen);                      /* Eq. 9 */
    if (level_sets) { memcpy(level_sets + set_pos, chosen, sizeof(int32_t) * keep[b]); set_pos += keep[b]; }
    /* Eq. 10: mu^{b-1} = {2^b j + k : j in J_b, k < 2^b}. */
    len = 0;
    for (int64_t j = 0; j < keep[b]; ++j)
      for (int64_t kk = 0; kk < ((int64_t)1 << b); ++kk) mu[len++] = (int32_t)(((int64_t)chosen[j] << b) + kk);
    /* mu^{b-1} holds 2^b tokens per kept coefficient, i.e. two aligned
     * scale-(b-1) blocks each. */
  }
  /* Algorithm 1 after the loop: mu^0 = the 2 keep[1] tokens, trimmed. */
  if (keep[0] < len) {
    for (int64_t t = 0; t < len; ++t) memcpy(sub + t * d, K + (int64_t)mu[t] * d, sizeof(double) * d);
    orc_skim_weights_f64(Q, q, d, sub, len, W);
    topk_ascending(W, mu, len, keep[0], chosen);
    memcpy(mu0, chosen, sizeof(int32_t) * keep[0]);
  } else {
    memcpy(mu0, mu, sizeof(int32_t) * keep[0]);
  }
  if (level_sets) memcpy(level_sets + set_pos, mu0, sizeof(int32_t) * keep[0]);
  free(mu); free(sub); free(A); free(D); free(gidx); free(chosen); free(W);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Attention (Eq. 1 / Eq. 3 form) and the final step of Algorithm 1.        */
/* ------------------------------------------------------------------------ */
int orc_attention_f64(const double* Q, int q, int d, const double* Ks, const double* Vs, int64_t m,
                      double* O) {
  if (!Q || !Ks || !Vs || !O || q <= 0 || d <= 0 || m <= 0) return -1;
  double* p = (double*)malloc(sizeof(double) * (size_t)m);
  if (!p) return -1;
  const double sqrt_d = sqrt((double)d);
  for (int i = 0; i < q; ++i) {
    for (int64_t t = 0; t < m; ++t) {
      double s = 0.0;
      for (int c = 0; c < d; ++c) s += Q[(size_t)i * d + c] * Ks[(size_t)t * d + c];
      p[t] = s / sqrt_d;
    }
    double mx = p[0];
    for (int64_t t = 1; t < m; ++t) if (p[t] > mx) mx = p[t];
    double z = 0.0;
    for (int64_t t = 0; t < m; ++t) { p[t] = exp(p[t] - mx); z += p[t]; }
    for (int c = 0; c < d; ++c) {
      double acc = 0.0;
      for (int64_t t = 0; t < m; ++t) acc += p[t] * Vs[(size_t)t * d + c];
      O[(size_t)i * d + c] = acc / z;
    }
  }
  free(p);
  return 0;
}

int orc_sparse_attn_f64(const double* Q, int q, int d, const double* K, const double* V,
                        const int32_t* mu0, int64_t k, const double* Kg, const double* Vg,
                        int64_t ng, double* O) {
  if (!Q || !K || !V || !mu0 || !O || k < 0 || ng < 0 || k + ng <= 0) return -1;
  if (ng > 0 && (!Kg || !Vg)) return -1;
  int64_t m = k + ng;
  double* Ks = (double*)malloc(sizeof(double) * (size_t)m * d);
  double* Vs = (double*)malloc(sizeof(double) * (size_t)m * d);
  if (!Ks || !Vs) { free(Ks); free(Vs); return -1; }
  /* K_sparse = [K[mu0]; K[I_g]], V_sparse = [V[mu0]; V[I_g]]. */
  for (int64_t t = 0; t < k; ++t) {
    memcpy(Ks + t * d, K + (int64_t)mu0[t] * d, sizeof(double) * d);
    memcpy(Vs + t * d, V + (int64_t)mu0[t] * d, sizeof(double) * d);
  }
  for (int64_t t = 0; t < ng; ++t) {
    memcpy(Ks + (k + t) * d, Kg + t * d, sizeof(double) * d);
    memcpy(Vs + (k + t) * d, Vg + t * d, sizeof(double) * d);
  }
  int rc = orc_attention_f64(Q, q, d, Ks, Vs, m, O);
  free(Ks);
  free(Vs);
  return rc;
}

/* ------------------------------------------------------------------------ */
/* Other wavelet bases (Eq. 6, Eq. 11 with a generic psi), periodized.      */
/* ------------------------------------------------------------------------ */
int orc_wavelet_taps(int wavelet, double* h, double* g) {
  if (!h || !g) return -1;
  if (wavelet == ORC_HAAR) {
    h[0] = HAAR_C; h[1] = HAAR_C;
    g[0] = HAAR_C; g[1] = -HAAR_C;
    return 2;
  }
  if (wavelet == ORC_DB2) {
    const double r = sqrt(3.0), s = 4.0 * sqrt(2.0);
    h[0] = (1.0 + r) / s; h[1] = (3.0 + r) / s; h[2] = (3.0 - r) / s; h[3] = (1.0 - r) / s;
    for (int k = 0; k < 4; ++k) g[k] = ((k & 1) ? -1.0 : 1.0) * h[3 - k];
    return 4;
  }
  return -1;
}

/* One periodized analysis level: len/2 approximation (and detail) rows. */
static void wavelet_step_f64(const double* x, int64_t len, int d, const double* h, const double* g, int taps,
                             double* a, double* det) {
  for (int64_t j = 0; j < len / 2; ++j) {
    for (int c = 0; c < d; ++c) {
      double sa = 0.0, sd = 0.0;
      for (int k = 0; k < taps; ++k) {
        const double v = x[((2 * j + k) % len) * d + c];
        sa += h[k] * v;
        sd += g[k] * v;
      }
      a[j * d + c] = sa;
      if (det) det[j * d + c] = sd;
    }
  }
}

int orc_wavelet_analysis_f64(const double* x, int64_t n, int d, int wavelet, int L, double* A, double* D) {
  double h[4], g[4];
  const int taps = orc_wavelet_taps(wavelet, h, g);
  if (taps < 0 || !x || !A || !D || !shape_ok(n, d, L)) return -1;
  double* cur = (double*)malloc(sizeof(double) * (size_t)n * d);
  if (!cur) return -1;
  memcpy(cur, x, sizeof(double) * (size_t)n * d);
  int64_t len = n;
  for (int b = 1; b <= L; ++b) {
    double* a = A + orc_pyramid_row_offset(n, b) * d;
    double* det = D + orc_pyramid_row_offset(n, b) * d;
    wavelet_step_f64(cur, len, d, h, g, taps, a, det);
    len /= 2;
    memcpy(cur, a, sizeof(double) * (size_t)len * d);
  }
  free(cur);
  return 0;
}

int orc_wavelet_synthesis_f64(const double* A, const double* D, int64_t n, int d, int wavelet, int L,
                              double* x) {
  double h[4], g[4];
  const int taps = orc_wavelet_taps(wavelet, h, g);
  if (taps < 0 || !x || !A || !D || !shape_ok(n, d, L)) return -1;
  double* cur = (double*)malloc(sizeof(double) * (size_t)n * d);
  double* nxt = (double*)malloc(sizeof(double) * (size_t)n * d);
  if (!cur || !nxt) { free(cur); free(nxt); return -1; }
  memcpy(cur, A + orc_pyramid_row_offset(n, L) * d, sizeof(double) * (size_t)(n >> L) * d);
  for (int b = L; b >= 1; --b) {
    const int64_t half = n >> b, len = 2 * half;
    const double* det = D + orc_pyramid_row_offset(n, b) * d;
    memset(nxt, 0, sizeof(double) * (size_t)len * d);
    /* The transpose of the analysis map: every input row receives h[k] a[j] + g[k] det[j]. */
    for (int64_t j = 0; j < half; ++j)
      for (int k = 0; k < taps; ++k)
        for (int c = 0; c < d; ++c)
          nxt[((2 * j + k) % len) * d + c] += h[k] * cur[j * d + c] + g[k] * det[j * d + c];
    memcpy(cur, nxt, sizeof(double) * (size_t)len * d);
  }
  memcpy(x, cur, sizeof(double) * (size_t)n * d);
  free(cur);
  free(nxt);
  return 0;
}

int orc_wavelet_approx_spec32(const float* x, int64_t len, int d, int wavelet, int level, int store_bf16,
                              float* out) {
  double h[4], g[4];
  const int taps = orc_wavelet_taps(wavelet, h, g);
  if (taps < 0 || !x || !out || !shape_ok(len, d, level)) return -1;
  float h32[4];
  for (int k = 0; k < taps; ++k) h32[k] = (float)h[k];
  const float c32 = (float)HAAR_C;
  float* prev = (float*)malloc(sizeof(float) * (size_t)len * d);
  float* cur = (float*)malloc(sizeof(float) * (size_t)(len / 2) * d);
  if (!prev || !cur) { free(prev); free(cur); return -1; }
  memcpy(prev, x, sizeof(float) * (size_t)len * d);
  int64_t n = len;
  for (int b = 1; b <= level; ++b) {
    const int64_t half = n / 2;
    for (int64_t j = 0; j < half; ++j) {
      for (int c = 0; c < d; ++c) {
        float v;
        if (wavelet == ORC_HAAR) {
          const float s = prev[(2 * j) * d + c] + prev[(2 * j + 1) * d + c];
          v = s * c32;
        } else {
          v = h32[0] * prev[((2 * j) % n) * d + c];
          for (int k = 1; k < taps; ++k) v = fmaf(h32[k], prev[((2 * j + k) % n) * d + c], v);
        }
        cur[j * d + c] = v;
      }
    }
    n = half;
    memcpy(prev, cur, sizeof(float) * (size_t)n * d);
  }
  for (int64_t i = 0; i < n * d; ++i) out[i] = store_bf16 ? orc_round_bf16(prev[i]) : prev[i];
  free(prev);
  free(cur);
  return 0;
}

int orc_filter_wavelet_f64(const double* Q, int q, int d, const double* K, int64_t n, int L, int wavelet,
                           const int32_t* keep, int spec32, int store_bf16, int32_t* mu0, int32_t* level_sets) {
  double h[4], g[4];
  if (orc_wavelet_taps(wavelet, h, g) < 0) return -1;
  if (!Q || !K || !keep || !mu0 || q <= 0 || !shape_ok(n, d, L) || !schedule_ok(n, L, keep)) return -1;
  int64_t cap = n >> L;
  for (int b = 1; b <= L; ++b) cap = cap > 2 * (int64_t)keep[b] ? cap : 2 * (int64_t)keep[b];
  int32_t* cand = (int32_t*)malloc(sizeof(int32_t) * (size_t)cap);
  int32_t* chosen = (int32_t*)malloc(sizeof(int32_t) * (size_t)cap);
  double* sub = (double*)malloc(sizeof(double) * (size_t)n * d);   /* K[mu^b] */
  double* A = (double*)malloc(sizeof(double) * (size_t)n * d);
  double* D = (double*)malloc(sizeof(double) * (size_t)n * d);
  float* sub32 = (float*)malloc(sizeof(float) * (size_t)n * d);
  float* a32 = (float*)malloc(sizeof(float) * (size_t)cap * d);
  double* rows = (double*)malloc(sizeof(double) * (size_t)cap * d);
  double* W = (double*)malloc(sizeof(double) * (size_t)cap);
  if (!cand || !chosen || !sub || !A || !D || !sub32 || !a32 || !rows || !W) {
    free(cand); free(chosen); free(sub); free(A); free(D); free(sub32); free(a32); free(rows); free(W);
    return -1;
  }
  int64_t m = n >> L, set_pos = 0;
  for (int64_t j = 0; j < m; ++j) cand[j] = (int32_t)j;
  for (int b = L; b >= 1; --b) {
    /* Eq. 10-11: the candidates' blocks of 2^b tokens, in candidate order. */
    const int64_t len = m << b, blk = (int64_t)1 << b;
    for (int64_t p = 0; p < len; ++p)
      memcpy(sub + p * d, K + (((int64_t)cand[p >> b] << b) + (p & (blk - 1))) * d, sizeof(double) * d);
    if (spec32) {
      for (int64_t i = 0; i < len * d; ++i) sub32[i] = (float)sub[i];
      orc_wavelet_approx_spec32(sub32, len, d, wavelet, b, store_bf16, a32);
      for (int64_t i = 0; i < m * d; ++i) rows[i] = (double)a32[i];
    } else {
      orc_wavelet_analysis_f64(sub, len, d, wavelet, b, A, D);
      memcpy(rows, A + orc_pyramid_row_offset(len, b) * d, sizeof(double) * (size_t)m * d);
    }
    orc_skim_weights_f64(Q, q, d, rows, m, W);                         /* Eq. 7-8 */
    topk_ascending(W, cand, m, keep[b], chosen);                       /* Eq. 9 */
    if (level_sets) { memcpy(level_sets + set_pos, chosen, sizeof(int32_t) * keep[b]); set_pos += keep[b]; }
    for (int64_t j = 0; j < keep[b]; ++j) { cand[2 * j] = 2 * chosen[j]; cand[2 * j + 1] = 2 * chosen[j] + 1; }
    m = 2 * (int64_t)keep[b];
  }
  /* mu^0: the 2 keep[1] tokens, trimmed to keep[0] on the raw keys. */
  if (keep[0] < m) {
    for (int64_t j = 0; j < m; ++j) memcpy(rows + j * d, K + (int64_t)cand[j] * d, sizeof(double) * d);
    orc_skim_weights_f64(Q, q, d, rows, m, W);
    topk_ascending(W, cand, m, keep[0], chosen);
    memcpy(mu0, chosen, sizeof(int32_t) * keep[0]);
  } else {
    memcpy(mu0, cand, sizeof(int32_t) * keep[0]);
  }
  if (level_sets) memcpy(level_sets + set_pos, mu0, sizeof(int32_t) * keep[0]);
  free(cand); free(chosen); free(sub); free(A); free(D); free(sub32); free(a32); free(rows); free(W);
  return 0;
}
