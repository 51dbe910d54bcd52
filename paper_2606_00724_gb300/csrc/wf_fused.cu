// Fused WaveFilter step (Algorithm 1 body): multi-scale skim/scan filtering
// (Eq. 7-11) and the final sparse attention, in one kernel.
//
// A thread-block cluster of CS CTAs serves P (1 or 2) (batch, head) units;
// every CTA holds one contiguous slice of each unit's candidate list at every
// scale (and finally of its sparse key list).  The warps of a CTA specialise:
//   * producer warps gather candidate rows (pyramid level b, raw keys for the
//     level-0 trim, or K/V rows of mu^0 and the generation rows) with 16-byte
//     cp.async copies into 128-byte-swizzled tiles of 128 rows, through a ring
//     of stages; each copy's completion arrives on the stage's mbarrier;
//   * one MMA thread issues tcgen05.mma (bf16 in, fp32 out) per landed tile,
//     writing S^T = rows . Q^T into the unit's TMEM region (32 columns per
//     tile), and in the attention O^T += V_s^T P^T;
//   * four compute warps per unit (one per TMEM lane quarter, one candidate
//     row per thread; both warpgroups, taking alternate tiles, when a
//     cluster serves one unit with long candidate lists) read the logits
//     back (tcgen05.ld), form the per-query max and
//     sum of exp of the slice, exchange them with the cluster (st.async into
//     every CTA, completion counted on its mbarrier), compute the ranking key
//     log2 W_j (Eq. 8) of each candidate, all-gather the keys the same way,
//     and run the same deterministic Top-K (Eq. 9, lowest position first on
//     ties) in every CTA, giving J_b and hence the next scale's candidates
//     {2j, 2j+1} (Eq. 10).
// The units of a cluster alternate: while the compute warps score, exchange
// and select one unit, the producers already stream the other unit's rows, so
// copies overlap the latency-bound phases.  In the attention the compute warps
// turn S into P = 2^(s - m) (bf16) for the MMA thread, and each CTA's partial
// (m, l, O^T) is reduce-scattered over head-dimension slices: CTA r combines
// rows d of O for its slice and writes them.
//
// A launch may also run part of the chain (a range of scales, the previous
// selection handed in, the last one handed out, the attention optional): the
// literal-basis path runs one launch per scale, each a programmatic dependent
// of the kernel before it (every thread waits for that grid before its first
// global access).
//
// Every wait is bounded (~1 s): on timeout the CTA records a status word,
// stops issuing MMAs and skips the remaining waits, so every thread reaches
// the final cluster barrier.
#include <math.h>
#include <string.h>

#include <map>
#include <mutex>
#include <tuple>

#include "wf_internal.cuh"
#include "wf_sm100.cuh"

namespace wf {
namespace {

using namespace sm100;

constexpr int D = 128;                     // head_dim
constexpr int TM = 128;                    // rows per MMA tile (M)
constexpr int NQ = 32;                     // query rows per MMA (N), zero padded
constexpr int MAXP = 2;                    // units per cluster
constexpr int NCW = 4;                     // compute warps of a unit (one per TMEM lane quarter)
constexpr int NCT = 32 * NCW;              // compute threads of a unit
constexpr int MMA_WARP = MAXP * NCW;       // TMEM allocation and MMA issue (lane 0)
constexpr int NPW = 3;                     // producer warps
constexpr int NPT = 32 * NPW;              // producer threads
constexpr int P0 = 32 * (MMA_WARP + 1);    // first producer thread
constexpr int NT = 32 * (MMA_WARP + 1 + NPW);  // threads per CTA
constexpr int MAXCS = 8;                   // CTAs per cluster
constexpr int HALF_BYTES = TM * 128;       // one 64-column half of a tile, 128-byte rows
constexpr int TILE_BYTES = 2 * HALF_BYTES;
constexpr int QGRP = (D / 8) * 128;        // bytes per 8-row group of a query tile (core matrices)
constexpr int Q_BYTES = NQ * D * 2;
constexpr int P_BYTES = NQ * TM * 2;
constexpr int MAXCS_PAD_BYTES = 8 * NQ * 4;  // the ragged head-dim slices of a cluster of up to 8 CTAs
// A unit's P double buffer; also its Top-K scratch and its combine buffer
// (the partial O rows of this CTA's head-dim slice from every cluster CTA:
// at most (D + cs) rows of 32 fp32 when cs does not divide D).
constexpr int UNIT_P_BYTES = 2 * P_BYTES + MAXCS_PAD_BYTES;
constexpr int kMaxCand = 64 * NCT;         // largest candidate list of the Top-K (64 keys a thread)
constexpr float kLog2e = 1.4426950408889634f;
constexpr uint32_t kCsyncId = 1;           // named barriers 1, 2: the compute warps of unit 0, 1
constexpr uint32_t kSetupSyncId = 3;       // named barrier 3: the set-up threads (all but the producers)

constexpr uint32_t kIdescScore = idesc_bf16(TM, NQ, 0, 0);  // A = rows (K-major), B = Q (K-major)
constexpr uint32_t kIdescPV = idesc_bf16(D, NQ, 1, 1);      // A = V^T (MN-major), B = P^T (MN-major)

constexpr int MAXT = 16;  // TMEM tiles of one unit's region (512 columns / 32)

struct UnitState {
  float2 xstat[MAXCS][NQ];  // (stabiliser, sum of exp) of every cluster CTA's slice
  float2 cstat[MAXCS][NQ];  // attention (max, row sum) of every CTA (d-slice owner side)
  // Per-warp slots (warp w of the unit at slot w; a WIDE unit's warps 4-7 use
  // the second unit's slots, which nothing else uses then).
  float2 kmm[MAXCS][NCW];   // (min, max) of the ranking keys of every cluster warp
  float2 wstat[NCW][NQ];    // (stabiliser, sum of exp) of each compute warp's rows
  float cw[NCW][NQ];        // softmax normaliser c_i, one copy per compute warp
  float fw[NCW][NQ];        // 2^(stabiliser - c_i) of each warp (keys from stored exponentials)
  float mloc[NQ], lacc[NQ];
  float alpha[NQ];          // attention: factor 2^(m_old - m_new) of a raised stabiliser
  float red[NCW][32];
};

struct Misc {
  unsigned long long full[4], empty[4];
  unsigned long long mdone[MAXP], jready[MAXP], xbar[MAXP], kbar[MAXP];
  unsigned long long tdone[MAXP][MAXT];  // scale tile t of a unit scored (one phase per scale)
  unsigned long long pfull[MAXP][2], pempty[MAXP][2], cbar[MAXP], cready[MAXP];
  UnitState us[MAXP];
  unsigned long long qfull;     // the query blocks have landed (the producers' first copies)
  unsigned long long rdone[2], rfree[2];  // grouped filter: a TMEM region's logits are ready / read
  unsigned long long stallbar;  // completed by nothing (the test-only stalled first wait)
  unsigned long long drainbar;  // the MMA thread's final commit
  long long wait_limit;         // bound of the waits that can give up (cycles)
  int abort;
  uint32_t tmem_base;
};

// The UnitState holding the per-warp slots of unit warp w (index w % 4).
template <bool WIDE>
__device__ __forceinline__ UnitState& wslots(Misc& ms, int pp, int w) {
  return WIDE ? ms.us[w >> 2] : ms.us[pp];
}

// Shared-memory layout (byte offsets; the stage ring starts at 0, 1024-byte
// aligned for the 128-byte swizzle).
struct SmemLayout {
  uint32_t q, p, misc, buf, bufw, total;
};
__host__ __device__ inline SmemLayout smem_layout(int stages, int P, int cmax, int kmax) {
  SmemLayout l;
  l.q = (uint32_t)stages * TILE_BYTES;
  l.p = l.q + (uint32_t)P * Q_BYTES;
  l.misc = l.p + (uint32_t)P * UNIT_P_BYTES;
  // Two buffers per unit alternate by scale: one receives the scale's keys and
  // then its selection J_b, the other still holds J_{b+1}.
  l.buf = (l.misc + (uint32_t)sizeof(Misc) + 127u) / 128u * 128u;
  l.bufw = (uint32_t)((max(cmax, kmax) + 3) / 4 * 4);
  l.total = l.buf + (uint32_t)P * 2u * 4u * l.bufw;
  return l;
}

struct FusedParams {
  const bf16* Q;
  int64_t qsb, qsh, qss;
  const bf16* K;
  const bf16* V;
  int64_t ksb, ksh, kss;
  const bf16* Kg;
  const bf16* Vg;
  int64_t gsb, gsh, gss;
  const bf16* coeffs;
  int64_t rows_total;
  bf16* O;
  int64_t osb, osh, oss;
  int32_t* idx;
  int32_t* level_sets;
  int64_t sets_stride;
  int* status;
  int q, n, ng, U, H, L, trim, P, cmax, kmax;
  uint32_t tmem_cols, ucols;  // TMEM allocation; columns per unit region
  uint32_t ecol;              // column of the stored exponentials in a unit region (0: none)
  long long wait_limit;       // bound of the waits that can give up (cycles)
  int stall;                  // test-only: the MMA thread's first wait never completes
  int G, nch;                 // grouped filter: query heads per key head, 32-row chunks of the stacked block
  int32_t keep[12];
  float scale_log2;           // log2(e) / sqrt(d)
  // The scales this launch runs, lev_top down to lev_bot (the whole chain, L
  // down to 1 or 0, for the pyramid step).  A launch that starts below L reads
  // the previous selection J_{lev_top+1} as the children list jin (candidate
  // block indices of scale lev_top, 2 J[i] and 2 J[i] + 1); one that ends
  // above the final scale writes the children of its last selection to jout.
  int lev_top, lev_bot, final_sel, attn;
  const int32_t* jin;
  int32_t* jout;
  int64_t jstride;  // entries per unit of jin and jout
  // Literal-basis rows: scale lev_top's candidate rows in candidate order
  // (row j of unit u at lrows + u lrows_unit + j D); null for the pyramid.
  const bf16* lrows;
  int64_t lrows_unit;
};

// Per-CTA constants and shared-memory addresses.
struct Ctx {
  uint8_t* smem;
  Misc* ms;
  SmemLayout ly;
  uint32_t rank, cs, tmem;
  int np, u0, lev_top, lev_end, stages;
};

// A unit's compute warps: one warpgroup (one per unit of a two-unit cluster),
// or both warpgroups (WIDE) when the cluster serves one unit; then the
// warpgroups take alternate tiles and share the Top-K.  Thread index within
// the unit's compute warps, their count and their barrier.
template <bool WIDE>
__host__ __device__ constexpr int unit_warps() {
  return WIDE ? 2 * NCW : NCW;
}
template <bool WIDE>
__device__ __forceinline__ int ctid() {
  return threadIdx.x & (32 * unit_warps<WIDE>() - 1);
}
template <bool WIDE>
__device__ __forceinline__ void csync() {
  named_sync(kCsyncId + (WIDE ? 0u : (threadIdx.x >> 7)), 32 * unit_warps<WIDE>());
}
// The warpgroup of a compute thread within its unit (0 unless WIDE), the
// first tile it takes and its tile stride.
template <bool WIDE>
__device__ __forceinline__ int unit_wg() {
  return WIDE ? (int)((threadIdx.x >> 7) & 1) : 0;
}
template <bool WIDE>
__host__ __device__ constexpr int tile_step() {
  return WIDE ? 2 : 1;
}

__device__ __forceinline__ bool aborted(const Misc& ms) { return abort_set(smem_u32(&ms.abort)); }

__device__ __forceinline__ void set_abort(Misc& ms, int* status) {
  ms.abort = 1;
  atomicExch(status, 1);
}

__device__ __noinline__ void wait_or_abort(uint32_t bar, uint32_t parity, Misc& ms, int* status) {
  if (!aborted(ms) && !mbar_wait_bounded(bar, parity, ms.wait_limit, smem_u32(&ms.abort))) set_abort(ms, status);
}

// Wait for a phase completed by other CTAs of the cluster (acquire, cluster scope).
__device__ __noinline__ void wait_cluster_or_abort(uint32_t bar, uint32_t parity, Misc& ms, int* status) {
  if (!aborted(ms) && !mbar_wait_cluster_bounded(bar, parity, ms.wait_limit, smem_u32(&ms.abort)))
    set_abort(ms, status);
}

__device__ __forceinline__ uint32_t bar_addr(const unsigned long long& b) { return smem_u32(&b); }

// Candidate count of scale `lev`: the top coefficients, or the children of
// the coefficients kept one scale up (Eq. 10).
__device__ __forceinline__ int m_total(const FusedParams& p, int lev) {
  return lev == p.L ? (p.n >> p.L) : 2 * p.keep[lev + 1];
}

// This CTA's slice [g0, g0 + mc) of a candidate list of m (sibling pairs kept
// together).
__device__ __forceinline__ void scale_slice(int m, uint32_t rank, uint32_t cs, int& g0, int& mc) {
  const int pairs = (m + 1) >> 1;
  // 32-bit arithmetic: rank <= 8 and pairs <= 2^16 (a 64-bit division is a
  // called routine on the path between two scales).
  g0 = min(m, 2 * (int)(rank * (uint32_t)pairs / cs));
  const int g1 = min(m, 2 * (int)((rank + 1u) * (uint32_t)pairs / cs));
  mc = g1 - g0;
}

// This CTA's slice of the sparse key list of `total` rows.
__device__ __forceinline__ void attn_slice(int total, uint32_t rank, uint32_t cs, int& a0, int& mc) {
  a0 = (int)(rank * (uint32_t)total / cs);
  mc = (int)((rank + 1u) * (uint32_t)total / cs) - a0;
}

__device__ __forceinline__ int tiles_of(int mc) { return (mc + TM - 1) / TM; }

// Head-dim slice [dlo(r), dlo(r + 1)) whose output rows CTA r combines.
__device__ __forceinline__ int dlo(int r, int cs) { return r * D / cs; }

// Where the rows of a candidate or key list come from.
//  kind 0: position j -> row j (top scale);
//  kind 1: position j -> row 2 J[j/2] + j%2 (children of the kept coefficients);
//  kind 2: sparse key list, positions < kk -> token 2 J[j/2] + j%2, then
//          generation rows;
//  kind 3: the same with a trimmed level 0, positions < kk -> token J[j].
struct RowSrc {
  const bf16* base;
  int64_t stride;
  const bf16* gbase;
  int64_t gstride;
  uint32_t J;  // shared address of the selection the rows derive from
  int kind, g0, mc, kk;
  int rows;  // rows of the source: indices from a selection are clamped below it
};

// Row r of a slice.  Kinds 0 and 1: the row index in the source; kinds 2
// and 3: the row's address (a key row or a generation row).  Indices read
// from a selection are valid rows; the clamp keeps every address inside the
// source even when a wait gave up and the selection was made from stale data
// (the status word then reports the failure).
template <int KIND>
__device__ __forceinline__ uint32_t row_index(const RowSrc& s, int r) {
  const int pos = s.g0 + (r < s.mc ? r : 0);  // rows past the slice repeat its first row
  const uint32_t row = KIND == 0 ? (uint32_t)pos
                                 : 2u * lds_u32(s.J + 4u * (uint32_t)(pos >> 1)) + (uint32_t)(pos & 1);
  return min(row, (uint32_t)s.rows - 1u);
}
template <int KIND>
__device__ __forceinline__ const bf16* row_ptr(const RowSrc& s, int r) {
  const int pos = s.g0 + (r < s.mc ? r : 0);
  const int pk = min(pos, s.kk - 1);
  const uint32_t tok0 = KIND == 3 ? lds_u32(s.J + 4u * (uint32_t)pk)
                                  : 2u * lds_u32(s.J + 4u * (uint32_t)(pk >> 1)) + (uint32_t)(pk & 1);
  const bf16* key = s.base + (int64_t)min(tok0, (uint32_t)s.rows - 1u) * s.stride;
  const bf16* gen = s.gbase + (int64_t)(pos - s.kk) * s.gstride;
  return pos < s.kk ? key : gen;
}

// Buffer k (0, 1) of unit pp; scale lev's keys and selection use buffer
// (L - lev) % 2.
__device__ __forceinline__ int32_t* unit_buf(const Ctx& c, int pp, int k) {
  return reinterpret_cast<int32_t*>(c.smem + c.ly.buf) + (pp * 2 + k) * (int)c.ly.bufw;
}
// Buffer holding the selection J made at scale lev.
__device__ __forceinline__ int32_t* unit_J(const Ctx& c, const FusedParams& p, int pp, int lev) {
  return unit_buf(c, pp, (p.L - lev) & 1);
}

// Rows of unit u at scale lev (pyramid level lev, or the raw keys at level 0).
__device__ __forceinline__ RowSrc scale_src(const Ctx& c, const FusedParams& p, int pp, int lev, int g0, int mc) {
  const int u = c.u0 + pp;
  const bool lit = p.lrows && lev >= 1 && lev == c.lev_top;  // literal-basis rows of this launch's scale
  RowSrc s;
  if (lit) {
    s.base = p.lrows + (int64_t)u * p.lrows_unit;  // row j: candidate j's transform (kind 0 below)
    s.stride = D;
  } else if (lev >= 1) {
    s.base = p.coeffs + ((int64_t)u * p.rows_total + ((int64_t)p.n - ((int64_t)p.n >> (lev - 1)))) * D;
    s.stride = D;
  } else {
    s.base = p.K + (int64_t)(u / p.H) * p.ksb + (int64_t)(u % p.H) * p.ksh;
    s.stride = p.kss;
  }
  s.gbase = nullptr;
  s.gstride = 0;
  s.J = smem_u32(unit_J(c, p, pp, lev + 1));  // the children of the selection one scale up (unused at the top)
  s.kind = (lev == p.L || lit) ? 0 : 1;
  s.g0 = g0;
  s.mc = mc;
  s.kk = 0;
  s.rows = lit ? m_total(p, lev) : (lev >= 1 ? (int)(p.n >> lev) : (int)p.n);
  return s;
}

// Sparse key list [K[mu^0]; Kg] (or the V rows) of unit pp.
__device__ __forceinline__ RowSrc attn_src(const Ctx& c, const FusedParams& p, int pp, bool values, int a0,
                                           int mc) {
  const int u = c.u0 + pp;
  const int64_t b = u / p.H, h = u % p.H;
  RowSrc s;
  s.base = (values ? p.V : p.K) + b * p.ksb + h * p.ksh;
  s.stride = p.kss;
  s.gbase = (values ? p.Vg : p.Kg) + b * p.gsb + h * p.gsh;
  s.gstride = p.gss;
  s.J = smem_u32(unit_J(c, p, pp, p.trim ? 0 : 1));  // mu^0 from the last selection
  s.kind = p.trim ? 3 : 2;
  s.g0 = a0;
  s.mc = mc;
  s.kk = p.keep[0];
  s.rows = (int)p.n;
  return s;
}

// Top-K scratch.  It lives in the unit's P buffers, which nothing uses before
// the attention.  The histogram and the list counter are zero between calls
// (zeroed at kernel start, cleared again at the end of every call).
constexpr int NB = 2048;     // histogram buckets
constexpr int MAXUW = 2 * NCW;  // most compute warps of a unit
struct SelScratch {
  uint32_t hist[NB];
  float2 blist[32 * MAXUW];  // boundary-bucket keys (key, position)
  float2 sred[2][MAXUW];     // (min, max) per warp, alternating rounds
  int wsum[4][MAXUW];        // per-warp sums of the scans (slot per scan, 32 bytes)
  uint32_t taken[2 * 32 * MAXUW];  // boundary keys taken, as each owner's position mask (zero between uses)
  uint32_t bcnt;
};
static_assert((sizeof(SelScratch) + 15) / 16 * 16 <= UNIT_P_BYTES, "Top-K scratch must fit the P buffers");
static_assert((NB / NCT) % 8 == 0, "buckets are cleared four at a time by up to twice NCT threads");
static_assert(offsetof(SelScratch, wsum) % 16 == 0, "the scan's warp sums are read 16 bytes at a time");

#define SC_ADDR(sc_a, field) ((sc_a) + (uint32_t)offsetof(SelScratch, field))

// Positions a Top-K thread owns for a list of m: the smallest power of two
// (at least 4) with R times the unit's compute threads >= m.
template <bool WIDE>
__host__ __device__ constexpr int topk_run(int m) {
  int R = 4;
  while (R * 32 * unit_warps<WIDE>() < m) R <<= 1;
  return R;
}

// ---------------------------------------------------------------------------
// Producer warps.
// ---------------------------------------------------------------------------

// This producer thread's share of one 128-row tile: 16-byte chunk c = pt % 16
// of rows r0 + RSTEP j (r0 = pt / 16, j < RROWS), written in the
// 128-byte-swizzled K-major layout (row r, chunk c at half c/8, byte
// r*128 + ((c%8) ^ (r%8))*16).  The 16 lanes of a half-warp copy the same
// rows, so each lane forms one row's index or address per 16 rows and the
// half-warp shares them by shuffles.  The swizzle term of a thread's rows
// repeats every 4 rows (RSTEP j mod 8 takes 4 values), so each destination
// is one add.
constexpr int RSTEP = NPT / 16;
constexpr int RROWS = (TM + RSTEP - 1) / RSTEP;  // most rows of one thread
static_assert(RSTEP == 6 && RROWS == 22, "the row schedule below assumes 6 rows a step");
template <int KIND>
__device__ __forceinline__ void load_share(uint32_t st, int t, const RowSrc& src, int pt) {
  const int c = pt & 15, r0 = pt >> 4, half = pt & 16;
  const uint32_t dbase = st + ((c >> 3) << 14) + (uint32_t)r0 * 128u;
  uint32_t xr[4];
#pragma unroll
  for (int m = 0; m < 4; ++m) xr[m] = (uint32_t)((c ^ (r0 + RSTEP * m)) & 7) << 4;
  // Rows j = c and j = 16 + c of this half-warp (clamped into the tile).
  const int ra = t * TM + r0 + RSTEP * c;
  const int rb = t * TM + min(r0 + RSTEP * min(16 + c, RROWS - 1), TM - 1);
  if (KIND <= 1) {
    const char* cb = reinterpret_cast<const char*>(src.base) + c * 16;
    const uint32_t sb = (uint32_t)src.stride * 2u;  // row stride in bytes
    const uint32_t ia = row_index<KIND>(src, ra), ib = row_index<KIND>(src, rb);
#pragma unroll
    for (int j = 0; j < RROWS; ++j) {
      const uint32_t idx = __shfl_sync(0xffffffffu, j < 16 ? ia : ib, half | (j & 15));
      if (RSTEP * j + RSTEP - 1 < TM || r0 + RSTEP * j < TM)
        cp_async16(dbase + 128u * RSTEP * j + xr[j & 3], cb + (size_t)idx * sb);
    }
  } else {
    const unsigned long long pa = reinterpret_cast<unsigned long long>(row_ptr<KIND>(src, ra));
    const unsigned long long pb = reinterpret_cast<unsigned long long>(row_ptr<KIND>(src, rb));
#pragma unroll
    for (int j = 0; j < RROWS; ++j) {
      const unsigned long long ak = __shfl_sync(0xffffffffu, j < 16 ? pa : pb, half | (j & 15));
      if (RSTEP * j + RSTEP - 1 < TM || r0 + RSTEP * j < TM)
        cp_async16(dbase + 128u * RSTEP * j + xr[j & 3], reinterpret_cast<const bf16*>(ak) + c * 8);
    }
  }
}

// Tiles t0 .. t0 + ntl - 1 of the source into ring slots it0, it0 + 1, ...
template <int S>
__device__ __noinline__ void produce(Misc& ms, int* status, uint32_t ring, int it0, int t0, int ntl, const RowSrc src,
                                     int pt) {
#pragma unroll 1
  for (int t = t0; t < t0 + ntl; ++t) {
    const int it = it0 + t - t0, s = it % S, n = it / S;
    if (n > 0) wait_or_abort(bar_addr(ms.empty[s]), (uint32_t)(n - 1) & 1u, ms, status);
    if (!aborted(ms)) {
      const uint32_t st = ring + s * TILE_BYTES;
      switch (src.kind) {
        case 0: load_share<0>(st, t, src, pt); break;
        case 1: load_share<1>(st, t, src, pt); break;
        case 2: load_share<2>(st, t, src, pt); break;
        default: load_share<3>(st, t, src, pt); break;
      }
    }
    cp_async_arrive_noinc(bar_addr(ms.full[s]));
  }
}

template <int S>
__device__ void producer_role(const Ctx& c, const FusedParams& p) {
  Misc& ms = *c.ms;
  const int pt = threadIdx.x - P0;
  // The query blocks go first, ahead of every row copy: they are the MMA
  // thread's first operands, and requests queued behind the whole grid's
  // first burst of rows would reach it only after that burst.  K-major core
  // matrices; rows >= q are zero-filled (no bytes read).
  for (int pp = 0; pp < c.np; ++pp) {
    const int u = c.u0 + pp;
    const bf16* qb = p.Q + (int64_t)(u / p.H) * p.qsb + (int64_t)(u % p.H) * p.qsh;
    const uint32_t sq = smem_u32(c.smem + c.ly.q + pp * Q_BYTES);
    for (int e = pt; e < NQ * (D / 8); e += NPT) {
      const int rr = e & 7, ch = (e >> 3) & (D / 8 - 1), g = e >> 7;
      const int i = g * 8 + rr;
      cp_async16_zfill(sq + (uint32_t)(g * QGRP + ch * 128 + rr * 16), qb + (int64_t)min(i, p.q - 1) * p.qss + ch * 8,
                       i < p.q);
    }
  }
  cp_async_arrive_noinc(bar_addr(ms.qfull));
  int it = 0;
  for (int lev = c.lev_top; lev >= c.lev_end; --lev) {
    for (int pp = 0; pp < c.np; ++pp) {
      // The rows of a lower scale are the children of the unit's last selection.
      if (lev != c.lev_top) wait_or_abort(bar_addr(ms.jready[pp]), (uint32_t)(c.lev_top - lev - 1) & 1u, ms, p.status);
      int g0, mc;
      scale_slice(m_total(p, lev), c.rank, c.cs, g0, mc);
      const int ntl = tiles_of(mc);
      produce<S>(ms, p.status, smem_u32(c.smem), it, 0, ntl, scale_src(c, p, pp, lev, g0, mc), pt);
      it += ntl;
    }
  }
  const int nsel = c.lev_top - c.lev_end + 1;
  for (int pp = 0; pp < c.np && p.attn; ++pp) {
    wait_or_abort(bar_addr(ms.jready[pp]), (uint32_t)(nsel - 1) & 1u, ms, p.status);
    int a0, mc;
    attn_slice(p.keep[0] + p.ng, c.rank, c.cs, a0, mc);
    const int ntl = tiles_of(mc);
    // The key tiles, then the value tiles.  A key tile's slot frees as soon
    // as its S product is done and a value tile's once its PV product is,
    // whose P the compute warps form from each S tile as it lands, so the
    // value stream follows the key stream without waiting for all of S.
    produce<S>(ms, p.status, smem_u32(c.smem), it, 0, ntl, attn_src(c, p, pp, false, a0, mc), pt);
    it += ntl;
    produce<S>(ms, p.status, smem_u32(c.smem), it, 0, ntl, attn_src(c, p, pp, true, a0, mc), pt);
    it += ntl;
  }
  // Copies still in flight (only after a wait gave up) land before the CTA
  // can leave.
  cp_async_wait_all();
}

// ---------------------------------------------------------------------------
// MMA thread.
// ---------------------------------------------------------------------------

// S^T = rows . Q^T of the landed tile in ring slot `it` into TMEM columns
// [dcol, dcol + 32); its completion frees the slot and completes `tbar`, so the
// compute warps start on the tile at once.
template <int S>
__device__ __forceinline__ void mma_score_tile(const Ctx& c, const FusedParams& p, int it, uint32_t dcol, uint32_t sq,
                                               uint32_t tbar) {
  Misc& ms = *c.ms;
  const int s = it % S, n = it / S;
  wait_or_abort(bar_addr(ms.full[s]), (uint32_t)n & 1u, ms, p.status);
  fence_proxy_async();
  if (!aborted(ms)) {
    tc_fence_after();
    const uint32_t st = smem_u32(c.smem) + s * TILE_BYTES;
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        mma_bf16(dcol, smem_desc_sw128(st + h * HALF_BYTES + kk * 32, 16, 1024),
                 smem_desc(sq + (4 * h + kk) * 256, 128, QGRP), kIdescScore, (h | kk) != 0);
  }
  mma_commit(bar_addr(ms.empty[s]));
  mma_commit(tbar);
}

// O^T += V_t^T P_t^T for the value tile in ring slot `it` and unit pp's P tile
// t (the P double buffer t % 2, filled by the compute warps).
template <int S>
__device__ __forceinline__ void mma_pv_tile(const Ctx& c, const FusedParams& p, int pp, int it, int t, uint32_t ocol) {
  Misc& ms = *c.ms;
  const uint32_t pa = smem_u32(c.smem + c.ly.p + pp * UNIT_P_BYTES);
  const int s = it % S, n = it / S;
  const uint32_t pb = (uint32_t)t & 1u, pn = (uint32_t)t >> 1;
  wait_or_abort(bar_addr(ms.full[s]), (uint32_t)n & 1u, ms, p.status);
  wait_or_abort(bar_addr(ms.pfull[pp][pb]), pn & 1u, ms, p.status);
  fence_proxy_async();
  if (!aborted(ms)) {
    tc_fence_after();
    const uint32_t st = smem_u32(c.smem) + s * TILE_BYTES;
#pragma unroll
    for (int kq = 0; kq < TM / 16; ++kq)
      mma_bf16(ocol, smem_desc_sw128(st + kq * 2048, HALF_BYTES, 1024),
               smem_desc(pa + pb * P_BYTES + kq * 1024, 512, 128), kIdescPV, (t > 0 || kq > 0) ? 1u : 0u);
  }
  mma_commit(bar_addr(ms.empty[s]));
  mma_commit(bar_addr(ms.pempty[pp][pb]));
}

template <int S>
__device__ void mma_role_body(const Ctx& c, const FusedParams& p) {
  Misc& ms = *c.ms;
  wait_or_abort(bar_addr(ms.qfull), 0u, ms, p.status);
  fence_proxy_async();
  int it = 0;
  for (int lev = c.lev_top; lev >= c.lev_end; --lev) {
    for (int pp = 0; pp < c.np; ++pp) {
      int g0, mc;
      scale_slice(m_total(p, lev), c.rank, c.cs, g0, mc);
      const int ntl = tiles_of(mc);
      const uint32_t tb = c.tmem + pp * p.ucols, sq = smem_u32(c.smem + c.ly.q + pp * Q_BYTES);
#pragma unroll 1
      for (int t = 0; t < ntl; ++t) mma_score_tile<S>(c, p, it + t, tb + 32 * t, sq, bar_addr(ms.tdone[pp][t]));
      it += ntl;
    }
  }
  for (int pp = 0; pp < c.np && p.attn; ++pp) {
    int a0, mc;
    attn_slice(p.keep[0] + p.ng, c.rank, c.cs, a0, mc);
    const int ntl = tiles_of(mc);
    const uint32_t tb = c.tmem + pp * p.ucols, sq = smem_u32(c.smem + c.ly.q + pp * Q_BYTES);
    if (ntl == 0) continue;
    // S_t as each key tile lands (its completion on the tile's barrier), then
    // the PV products as the value tiles land and their P tiles are formed.
#pragma unroll 1
    for (int t = 0; t < ntl; ++t) mma_score_tile<S>(c, p, it + t, tb + 32 * t, sq, bar_addr(ms.tdone[pp][t]));
    it += ntl;
#pragma unroll 1
    for (int t = 0; t < ntl; ++t) mma_pv_tile<S>(c, p, pp, it + t, t, tb + p.ucols - 32);
    it += ntl;
    mma_commit(bar_addr(ms.mdone[pp]));  // every PV product of the unit is done
  }
}

// The MMA thread: an optional stalled first wait (test-only), the MMAs, then
// a commit that it waits for (default bound), so that no MMA is still
// writing TMEM when it is freed, also after a wait gave up.
template <int S>
__device__ void mma_role(const Ctx& c, const FusedParams& p) {
  Misc& ms = *c.ms;
  if (p.stall) wait_or_abort(bar_addr(ms.stallbar), 0u, ms, p.status);
  mma_role_body<S>(c, p);
  mma_commit(bar_addr(ms.drainbar));
  (void)mbar_wait_bounded(bar_addr(ms.drainbar), 0u, kDefaultWaitLimit);
}

// ---------------------------------------------------------------------------
// Compute warps.
// ---------------------------------------------------------------------------

// Reduce 32 values per lane across the warp's 32 lanes; afterwards lane i
// holds the reduction of column i (31 shuffles).
template <bool MAX>
__device__ __forceinline__ float transpose_reduce32(float (&v)[32], int lane) {
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    const bool up = (lane & off) != 0;
#pragma unroll
    for (int j = 0; j < off; ++j) {
      const float keep = up ? v[j + off] : v[j];
      const float send = up ? v[j] : v[j + off];
      const float recv = __shfl_xor_sync(0xffffffffu, send, off);
      v[j] = MAX ? fmaxf(keep, recv) : keep + recv;
    }
  }
  return v[0];
}


// Exclusive prefix sum over the unit's compute threads (thread order), with
// its per-warp sums in the words at wsum_a.  One barrier: the caller does not
// reuse those words before another barrier has passed.
template <bool WIDE>
__device__ __forceinline__ int cta_excl_scan(int v, uint32_t wsum_a) {
  const int lane = threadIdx.x & 31, warp = ctid<WIDE>() >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) sts_u32(wsum_a + 4u * warp, (uint32_t)incl);
  csync<WIDE>();
  int before = 0;
#pragma unroll
  for (int q = 0; q < unit_warps<WIDE>() / 4; ++q) {
    const uint4 w = lds_v4(wsum_a + 16u * q);
    before += (warp > 4 * q ? (int)w.x : 0) + (warp > 4 * q + 1 ? (int)w.y : 0) + (warp > 4 * q + 2 ? (int)w.z : 0) +
              (warp > 4 * q + 3 ? (int)w.w : 0);
  }
  return before + incl - v;
}

// Bucket of key v in NB buckets linear over [lo, hi): the same fp32
// operations in every pass and every CTA give the same bucket.
__device__ __forceinline__ int bucket_of(float v, float lo, float scale) {
  // floor(x) for 0 <= x < 2^23: adding 2^23 rounded toward -inf leaves
  // floor(x) in the low mantissa bits.
  const float x = fmaxf((v - lo) * scale, 0.f);
  return min(NB - 1, __float_as_int(__fadd_rd(x, 8388608.f)) - 0x4B000000);
}

// Bit counts of the Top-K's position masks (32 or 64 positions a thread).
__device__ __forceinline__ int popc_m(uint32_t x) { return __popc(x); }
__device__ __forceinline__ int popc_m(unsigned long long x) { return __popcll(x); }
__device__ __forceinline__ int ffs_m(uint32_t x) { return __ffs(x); }
__device__ __forceinline__ int ffs_m(unsigned long long x) { return __ffsll((long long)x); }

// (min, max) of the undecided keys (bit i of act: position j0 + i of the key
// array) over the compute threads, via slot `par`.
template <typename MT, bool WIDE>
__device__ __forceinline__ float2 cta_minmax(uint32_t keys_a, int j0, MT act, uint32_t sc_a, int par) {
  const int lane = threadIdx.x & 31, warp = ctid<WIDE>() >> 5;
  float lo = INFINITY, hi = -INFINITY;
#pragma unroll 1
  for (MT a = act; a; a &= a - 1) {
    const float v = lds_f32(keys_a + 4u * (uint32_t)(j0 + ffs_m(a) - 1));
    lo = fminf(lo, v);
    hi = fmaxf(hi, v);
  }
  lo = warp_min_f32(lo);
  hi = warp_max_f32(hi);
  if (lane == 0) sts_v2(SC_ADDR(sc_a, sred) + 8u * (par * MAXUW + warp), __float_as_uint(lo), __float_as_uint(hi));
  csync<WIDE>();
#pragma unroll
  for (int w = 0; w < unit_warps<WIDE>(); ++w) {
    const uint2 r = lds_v2(SC_ADDR(sc_a, sred) + 8u * (par * MAXUW + w));
    lo = fminf(lo, __uint_as_float(r.x));
    hi = fmaxf(hi, __uint_as_float(r.y));
  }
  return make_float2(lo, hi);
}

// Every warp locates the boundary bucket in the histogram by itself, with no
// barrier or broadcast: the bucket holding the need-th largest undecided key
// (buckets ranked high to low), how many of its keys are still needed, and
// how many it holds.  Lane l sums the 64 buckets [NB - 64 (l + 1), NB - 64 l)
// (reading them in a lane-rotated order, free of bank conflicts); a scan over
// the lanes finds the chunk, and a second scan over that chunk's buckets, two
// a lane, the bucket.
__device__ __forceinline__ uint3 warp_boundary(uint32_t hist_a, uint32_t need, int lane) {
  const uint32_t cbase = hist_a + 4u * (uint32_t)(NB - 64 * (lane + 1));
  uint32_t tot = 0;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const uint4 v = lds_v4(cbase + 16u * (uint32_t)((i + lane) & 15));
    tot += v.x + v.y + v.z + v.w;
  }
  uint32_t incl = tot;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  // Some lane always qualifies (need never exceeds the keys counted); the
  // clamp only keeps the reads in the histogram should a wait have given up.
  const int lc = max(0, __ffs(__ballot_sync(0xffffffffu, incl >= need)) - 1);
  const uint32_t above = __shfl_sync(0xffffffffu, incl - tot, lc);
  const int bb = NB - 1 - 64 * lc - 2 * lane;                 // this lane's buckets bb and bb - 1
  const uint2 pr = lds_v2(hist_a + 4u * (uint32_t)(bb - 1));  // .x = bucket bb - 1, .y = bucket bb
  const uint32_t pair = pr.x + pr.y;
  uint32_t inc2 = pair;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t t = __shfl_up_sync(0xffffffffu, inc2, o);
    if (lane >= o) inc2 += t;
  }
  const int l2 = max(0, __ffs(__ballot_sync(0xffffffffu, above + inc2 >= need)) - 1);
  const uint32_t before = above + inc2 - pair;
  const bool upper = before + pr.y >= need;
  const uint32_t b = upper ? (uint32_t)bb : (uint32_t)(bb - 1);
  const uint32_t nd = upper ? need - before : need - before - pr.y;
  const uint32_t ct = upper ? pr.y : pr.x;
  return make_uint3(__shfl_sync(0xffffffffu, b, l2), __shfl_sync(0xffffffffu, nd, l2),
                    __shfl_sync(0xffffffffu, ct, l2));
}

// Top-K of the m keys at keys_a (largest first, lower position wins ties):
// the kk chosen candidate indices, in ascending position order, overwrite the
// key array.  A candidate's index is its position at the top scale, else
// 2 J[j/2] + j%2 with J the previous selection at jprev_a (Eq. 10).
// [lo, hi] is the range of the keys (sent along with them).
// Each thread owns the run of R positions j0 = tid R .. j0 + R - 1 (R a power
// of two, 4 to 64), with one bit per position for "undecided" and "taken" in
// a mask of type MT (32 bits up to R = 32, else 64).
// The keys stay in shared memory; every pass re-reads them four at a time
// (16-byte loads, the G = R / 4 groups of a run visited in a lane-rotated
// order so that the 8 lanes of a quarter warp hit distinct banks).  Each
// round spreads the undecided keys over NB buckets linear in [lo, hi] (fp32
// arithmetic is monotone, so a key in a higher bucket is strictly larger);
// every warp then finds the bucket holding the boundary from the counts: keys
// above it are taken, keys below it dropped.  A boundary bucket of at most
// as many keys as the unit has threads is resolved exactly: its keys go to a
// list, and each is ranked on (key, -position) against the whole list, by its
// owner (one warpgroup) or by the list entry's thread, which marks a winner in
// its owner's position mask (both warpgroups: measured 116.9 -> 110.6 us at
// 128K, while one warpgroup ran slower that way).  A larger bucket is
// bucketed again over its own range.  If only equal keys remain, the lowest
// positions are taken.
template <typename MT, bool WIDE>
__device__ __noinline__ void select_keys(uint32_t keys_a, int m, int kk, uint32_t jprev_a, int top, uint32_t sc_a,
                                         float lo, float hi, int R) {
  constexpr int MB = 8 * (int)sizeof(MT);       // positions a mask holds
  constexpr int TN = 32 * unit_warps<WIDE>();   // the unit's compute threads
  constexpr int BPT = NB / TN;                  // buckets each thread clears
  const int tid = ctid<WIDE>(), lane = tid & 31;
  const int j0 = tid * R;
  const int G = R >> 2;                         // groups of four keys in a run
  const int rotg = ((lane * G) >> 3) & (G - 1);  // first group this lane visits
  const int nv = max(0, min(R, m - j0));        // valid positions of the run
  const uint32_t m4 = (uint32_t)((m + 3) & ~3);  // the key array holds m4 >= 4 words
  MT act = nv >= MB ? ~(MT)0 : (((MT)1 << nv) - 1), took = 0;
  // The four keys of group g (clamped into the array; positions past m are
  // never undecided).
  auto group = [&](int g) {
    const uint4 v = lds_v4(keys_a + 4u * min((uint32_t)(j0 + 4 * g), m4 - 4u));
    return make_float4(__uint_as_float(v.x), __uint_as_float(v.y), __uint_as_float(v.z), __uint_as_float(v.w));
  };
  const uint32_t hist_a = SC_ADDR(sc_a, hist);
  const uint32_t own_a = hist_a + 4u * (uint32_t)(BPT * tid);  // the buckets this thread clears
  uint32_t need = (uint32_t)kk;
  bool resolved = false;
#pragma unroll 1
  for (int iter = 0; iter < 6; ++iter) {
    if (!(hi > lo)) break;  // every undecided key is equal (or none is left)
    const float scale = (float)NB / (hi - lo);
#pragma unroll 4
    for (int gg = 0; gg < G; ++gg) {
      const int g = (gg + rotg) & (G - 1);
      const float4 v = group(g);
      const uint32_t a4 = (uint32_t)(act >> (4 * g));
      const int b0 = bucket_of(v.x, lo, scale), b1 = bucket_of(v.y, lo, scale);
      const int b2 = bucket_of(v.z, lo, scale), b3 = bucket_of(v.w, lo, scale);
      reds_add_if(a4 & 1u, hist_a + 4u * b0, 1u);
      reds_add_if(a4 & 2u, hist_a + 4u * b1, 1u);
      reds_add_if(a4 & 4u, hist_a + 4u * b2, 1u);
      reds_add_if(a4 & 8u, hist_a + 4u * b3, 1u);
    }
    csync<WIDE>();
    const uint3 bd = warp_boundary(hist_a, need, lane);
    const int sb = (int)bd.x;
    need = bd.y;
    const uint32_t cnt = bd.z;
#pragma unroll 4
    for (int gg = 0; gg < G; ++gg) {
      const int g = (gg + rotg) & (G - 1);
      const float4 v = group(g);
      const int bk[4] = {bucket_of(v.x, lo, scale), bucket_of(v.y, lo, scale), bucket_of(v.z, lo, scale),
                         bucket_of(v.w, lo, scale)};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const MT bit = act & ((MT)1 << (4 * g + e));  // 0 for a decided position
        took |= bk[e] > sb ? bit : (MT)0;
        act &= bk[e] != sb ? ~bit : ~(MT)0;
      }
    }
    if (cnt == need) {
      took |= act;
      act = 0;
      resolved = true;
      break;
    }
    if (cnt <= (uint32_t)TN) {
      // Append the boundary keys (one atomic per warp), then every owner
      // ranks its own keys against the list.
      const int nb = popc_m(act);
      int incl = nb;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      uint32_t wbase = 0;
      if (lane == 31 && incl > 0) wbase = atoms_add(SC_ADDR(sc_a, bcnt), (uint32_t)incl);
      wbase = __shfl_sync(0xffffffffu, wbase, 31);
      uint32_t slot = wbase + (uint32_t)(incl - nb);
#pragma unroll 1
      for (MT a = act; a; a &= a - 1, ++slot) {
        const int i = ffs_m(a) - 1;
        // slot < TN always (the list holds cnt <= TN keys); the predicate
        // keeps the store in the list should a wait have given up.
        sts_v2_if(slot < (uint32_t)TN, SC_ADDR(sc_a, blist) + 8u * slot, lds_u32(keys_a + 4u * (uint32_t)(j0 + i)),
                  (uint32_t)(j0 + i));
      }
      csync<WIDE>();
      if (!WIDE) {
        // Every owner ranks its own boundary keys on (key, -position)
        // against the list (measured faster with one warpgroup).
#pragma unroll 1
        for (MT a = act; a; a &= a - 1) {
          const int i = ffs_m(a) - 1;
          const float kx = lds_f32(keys_a + 4u * (uint32_t)(j0 + i));
          const int jx = j0 + i;
          uint32_t rank = 0;
#pragma unroll 1
          for (uint32_t v0 = 0; v0 < cnt; v0 += 4) {
            uint2 o[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) o[k] = lds_v2(SC_ADDR(sc_a, blist) + 8u * min(v0 + k, cnt - 1));
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float ko = __uint_as_float(o[k].x);
              rank += (v0 + k < cnt) && ((ko > kx) || (ko == kx && (int)o[k].y < jx));
            }
          }
          if (rank < need) took |= (MT)1 << i;
        }
        act = 0;
        resolved = true;
        break;
      }
      // WIDE: thread t ranks list entry t on (key, -position) against the
      // whole list (every thread reads the same entry at a time: broadcasts)
      // and marks a winner in its owner's mask; then each owner takes its bits.
      constexpr int MW = (int)sizeof(MT) / 4;  // 32-bit words of a mask
      if ((uint32_t)tid < cnt) {
        const uint2 me = lds_v2(SC_ADDR(sc_a, blist) + 8u * (uint32_t)tid);
        const float kx = __uint_as_float(me.x);
        const int jx = (int)me.y;
        uint32_t rank = 0;
#pragma unroll 1
        for (uint32_t v0 = 0; v0 < cnt; v0 += 4) {
          uint2 o[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) o[k] = lds_v2(SC_ADDR(sc_a, blist) + 8u * min(v0 + k, cnt - 1));
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float ko = __uint_as_float(o[k].x);
            rank += (v0 + k < cnt) && ((ko > kx) || (ko == kx && (int)o[k].y < jx));
          }
        }
        if (rank < need) {
          const int owner = jx / R, bit = jx - owner * R;
          // owner < TN always; the bound keeps the store in the masks should a wait have given up
          const uint32_t w = (uint32_t)min(owner, TN - 1) * MW + (uint32_t)(bit >> 5);
          reds_or(SC_ADDR(sc_a, taken) + 4u * w, 1u << (bit & 31));
        }
      }
      csync<WIDE>();
      {
        const uint32_t ta = SC_ADDR(sc_a, taken) + 4u * (uint32_t)(tid * MW);
        MT mine = (MT)lds_u32(ta);
        if (MW == 2) mine |= (MT)((unsigned long long)lds_u32(ta + 4u) << 32);
        took |= mine & act;
        sts_u32(ta, 0u);
        if (MW == 2) sts_u32(ta + 4u, 0u);
      }
      act = 0;
      resolved = true;
      break;
    }
    // The boundary bucket again over its own range, with a cleared histogram.
    csync<WIDE>();  // every warp has read the histogram
#pragma unroll
    for (int i = 0; i < BPT / 4; ++i) sts_v4(own_a + 16u * i, make_uint4(0, 0, 0, 0));
    const float2 lh = cta_minmax<MT, WIDE>(keys_a, j0, act, sc_a, iter & 1);  // its barrier also publishes the cleared buckets
    lo = lh.x;
    hi = lh.y;
  }
  MT take = took;
  if (!resolved) {
    // Only equal keys are undecided: the first `need` by position are taken.
    const int eq_base = cta_excl_scan<WIDE>(popc_m(act), SC_ADDR(sc_a, wsum) + 96u);
    int remaining = (int)need - eq_base;
    for (MT e = act; e && remaining > 0; --remaining) {
      const MT low = e & (~e + 1);
      take |= low;
      e ^= low;
    }
  }
  // Each winner at its output rank, four positions at a time (positions
  // 4g .. 4g + 3 of the run are the children of the previous selection's
  // entries (j0 + 4g) / 2 and that + 1).  The scan's barrier orders every read
  // of the keys, the histogram and the boundary list before the key array is
  // overwritten and the scratch cleared.
  int r = cta_excl_scan<WIDE>(popc_m(take), SC_ADDR(sc_a, wsum) + 64u);
#pragma unroll 1
  for (int g = 0; g < G; ++g) {
    const uint32_t t4 = (uint32_t)(take >> (4 * g)) & 15u;
    if (!t4) continue;
    const int j = j0 + 4 * g;
    int c[4] = {j, j + 1, j + 2, j + 3};
    if (!top) {
      const uint2 pj = lds_v2(jprev_a + 4u * (uint32_t)(j >> 1));
      c[0] = 2 * (int)pj.x;
      c[1] = 2 * (int)pj.x + 1;
      c[2] = 2 * (int)pj.y;
      c[3] = 2 * (int)pj.y + 1;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      // r < kk <= m always; the bound keeps the store in the array should a
      // wait have given up.
      sts_u32_if(((t4 >> e) & 1u) && (uint32_t)r < (uint32_t)m, keys_a + 4u * (uint32_t)r, (uint32_t)c[e]);
      r += (t4 >> e) & 1u;
    }
  }
#pragma unroll
  for (int i = 0; i < BPT / 4; ++i) sts_v4(own_a + 16u * i, make_uint4(0, 0, 0, 0));
  if (tid == 0) sts_u32(SC_ADDR(sc_a, bcnt), 0u);
  csync<WIDE>();
}

// Top-K dispatch: R = the smallest power of two (at least 4) with R TN >= m
// (m <= 64 NCT, TN the unit's compute threads); 64-bit position masks only
// for R = 64.
template <bool WIDE>
__device__ __forceinline__ void select_topk(uint32_t keys_a, int m, int kk, uint32_t jprev_a, int top, uint32_t sc_a,
                                            float lo, float hi) {
  const int R = topk_run<WIDE>(m);
  if (WIDE || R <= 32) select_keys<uint32_t, WIDE>(keys_a, m, kk, jprev_a, top, sc_a, lo, hi, R);
  else select_keys<unsigned long long, WIDE>(keys_a, m, kk, jprev_a, top, sc_a, lo, hi, R);
}

// The warp's (stabiliser, sum of 2^(l sl2 - stabiliser)) per query over its
// rows of TMEM tiles 0..ntl-1, with the stabiliser the column maximum over
// all those rows: the overflow path of scale_sums, one query column at a
// time (compact code for a path that real inputs never take).
template <bool WIDE>
__device__ __noinline__ float2 warp_sums_exact(uint32_t tb, int ntl, int mc, float sl2) {
  const int tid = ctid<WIDE>(), lane = tid & 31, warp = tid >> 5, row = tid & (TM - 1);
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
  float2 out = make_float2(-INFINITY, 0.f);
#pragma unroll 1
  for (int i = 0; i < 32; ++i) {
    float mx = -INFINITY;
#pragma unroll 1
    for (int t = unit_wg<WIDE>(); t < ntl; t += tile_step<WIDE>()) {
      const float v = tmem_ld1(tb + lane_base + 32 * t + i);
      if (t * TM + row < mc) mx = fmaxf(mx, v);
    }
    const float mi = warp_max_f32(mx) * sl2;
    float sum = 0.f;
#pragma unroll 1
    for (int t = unit_wg<WIDE>(); t < ntl; t += tile_step<WIDE>()) {
      const float v = tmem_ld1(tb + lane_base + 32 * t + i);
      if (t * TM + row < mc) sum += ex2(fmaf(v, sl2, -mi));
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == i) out = make_float2(mi, sum);
  }
  return out;
}

// Softmax statistics of one scale (Eq. 7-8), tile by tile as the MMA thread
// completes them, so that the exponentials of early tiles overlap the
// copies of later ones.  Each compute warp takes as its stabiliser per query
// the largest logit (x sl2, log2 units) of its rows in the first tile (a
// warp with no row there has none in later tiles either) and accumulates the
// sum of 2^(l sl2 - m) over its rows.  A later logit more than ~127 above the
// stabiliser would overflow the sum; the warp then redoes its sums with the
// maximum over all its rows.  The four warps' (m, sum) merge into the CTA's
// (M, S) per query, which goes to slot `rank` of every cluster CTA's xstat.
// tpar holds the parity of each tile barrier's next phase.
template <bool WIDE>
__device__ __noinline__ bool scale_sums(uint32_t rank, uint32_t cs, Misc& ms, int pp, uint32_t tb, int ntl, int mc,
                                        float sl2, uint32_t ecol, uint32_t& tpar, int* status) {
  const int tid = ctid<WIDE>(), lane = tid & 31, warp = tid >> 5, row = tid & (TM - 1);
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
  UnitState& us = ms.us[pp];
  const f32x2 s2 = pk2(sl2, sl2);
  f32x2 nml[16], acc[16];
  float mcol = -INFINITY;  // lane i: this warp's stabiliser of query i
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    acc[k] = pk2(0.f, 0.f);
    nml[k] = pk2(0.f, 0.f);
  }
#pragma unroll 1
  for (int t = unit_wg<WIDE>(); t < ntl; t += tile_step<WIDE>()) {
    wait_or_abort(bar_addr(ms.tdone[pp][t]), (tpar >> t) & 1u, ms, status);
    tpar ^= 1u << t;
    tc_fence_after();
    uint32_t ra[32];
    tmem_ld32_issue(tb + lane_base + 32 * t, ra);
    tmem_wait_ld();
    const bool valid = t * TM + row < mc;
    if (t == unit_wg<WIDE>()) {
      float m2[2];
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        m2[i & 1] = warp_max_f32(valid ? __uint_as_float(ra[i]) : -INFINITY) * sl2;
        mcol = lane == i ? m2[i & 1] : mcol;
        if (i & 1) nml[i >> 1] = pk2(-m2[0], -m2[1]);
      }
    }
    if (valid) {
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        const float2 x = up2(fma2(pk2(__uint_as_float(ra[2 * k]), __uint_as_float(ra[2 * k + 1])), s2, nml[k]));
        const float e0 = ex2(x.x), e1 = ex2(x.y);
        acc[k] = add2(acc[k], pk2(e0, e1));
        ra[2 * k] = __float_as_uint(e0);
        ra[2 * k + 1] = __float_as_uint(e1);
      }
    }
    // The exponentials stay in TMEM for the ranking keys (rows past the
    // slice store whatever they hold; no key is formed for them).
    if (ecol) tmem_st32(tb + ecol + lane_base + 32 * t, ra);
  }
  if (ecol) tmem_wait_st();
  float a[32];
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const float2 v = up2(acc[k]);
    a[2 * k] = v.x;
    a[2 * k + 1] = v.y;
  }
  float2 st = make_float2(mcol, transpose_reduce32<false>(a, lane));
  const bool overflow = __any_sync(0xffffffffu, !(st.y <= 3.0e38f));
  if (overflow) st = warp_sums_exact<WIDE>(tb, ntl, mc, sl2);
  sts_v2(smem_u32(&wslots<WIDE>(ms, pp, warp).wstat[warp & 3][lane]), __float_as_uint(st.x), __float_as_uint(st.y));
  csync<WIDE>();
  if (tid < 32) {
    constexpr int NW = unit_warps<WIDE>();
    float2 w[NW];
#pragma unroll
    for (int k = 0; k < NW; ++k) {
      const uint2 v = lds_v2(smem_u32(&wslots<WIDE>(ms, pp, k).wstat[k & 3][tid]));
      w[k] = make_float2(__uint_as_float(v.x), __uint_as_float(v.y));
    }
    float M = -INFINITY;
#pragma unroll
    for (int k = 0; k < NW; ++k)
      if (w[k].y > 0.f) M = fmaxf(M, w[k].x);
    float S = 0.f;
#pragma unroll
    for (int k = 0; k < NW; ++k)
      if (w[k].y > 0.f) S = fmaf(w[k].y, ex2(w[k].x - M), S);
    const uint32_t dst = smem_u32(&us.xstat[rank][tid]);
    const uint32_t bar = bar_addr(ms.xbar[pp]);
    // After a wait gave up, this CTA sends nothing to the cluster.
    const uint32_t nr = aborted(ms) ? 0u : cs;
#pragma unroll 1
    for (uint32_t r = 0; r < nr; ++r)
      st_async_v2(map_rank(dst, r), __float_as_uint(M), __float_as_uint(S), map_rank(bar, r));
  }
  return ecol != 0 && !overflow;  // the stored exponentials are relative to this warp's stabilisers
}

// Softmax normaliser per query, c_i = M + log2 S over the whole candidate
// set from the cluster's (M, S) pairs (padded query columns get +inf and
// weigh 0), into this warp's slot of cw.  Every warp forms its own copy,
// so no barrier across the warps is needed.
template <bool WIDE>
__device__ __forceinline__ void warp_normaliser(Misc& ms, int pp, uint32_t cs, int q) {
  const int lane = threadIdx.x & 31, warp = ctid<WIDE>() >> 5;
  UnitState& us = ms.us[pp];
  UnitState& ws = wslots<WIDE>(ms, pp, warp);
  float2 st[MAXCS];
#pragma unroll
  for (int r = 0; r < MAXCS; ++r) {
    const uint2 v = lds_v2(smem_u32(&us.xstat[min(r, (int)cs - 1)][lane]));
    st[r] = make_float2(__uint_as_float(v.x), __uint_as_float(v.y));
  }
  float M = -INFINITY;
#pragma unroll
  for (int r = 0; r < MAXCS; ++r)
    if (r < (int)cs && st[r].y > 0.f) M = fmaxf(M, st[r].x);
  float S = 0.f;
#pragma unroll
  for (int r = 0; r < MAXCS; ++r)
    if (r < (int)cs && st[r].y > 0.f) S = fmaf(st[r].y, ex2(st[r].x - M), S);
  const float c = lane < q ? M + lg2(S) : INFINITY;
  ws.cw[warp & 3][lane] = c;
  ws.fw[warp & 3][lane] = ex2(ws.wstat[warp & 3][lane].x - c);  // 0 for padded columns and for a warp without rows
  __syncwarp();
}

// Ranking key log2 W_j of each valid row (Eq. 8), stored at position g0 + j
// of every cluster CTA's key array of the unit; each warp's (min, max) key
// goes to slot (rank, warp) of every CTA's kmm on the same barrier.
// With the scale's exponentials e = 2^(l sl2 - m) stored in TMEM at column
// ecol (eok: the warp's sums used those stabilisers m), W_j = sum_i e_ij f_i
// with f_i = 2^(m_i - c_i) from us.fw: fused multiply-adds, no exponentials.
// Otherwise, and for a row whose W is tiny (below 2^-96, where flushed terms
// could matter), the key is a log-sum-exp of the logits over the query rows
// against the normaliser c_i (us.cw): every exponent l sl2 - c_i is at most 0
// (c_i is the log of a sum that contains the row's own term), so the sum
// cannot overflow; padded query columns have c_i = +inf and add 0; a tiny sum
// is taken again shifted by its largest exponent.
// The exact key of one row from its logits (the slow path of pass_keys):
// the log-sum-exp over the query rows of l sl2 - c_i, with c_i at cw_a
// (+inf for padded columns); a tiny sum is taken again shifted by its largest
// exponent.
__device__ __forceinline__ float key_from_logits(const uint32_t (&ra)[32], uint32_t cw_a, float sl2) {
  const f32x2 s2 = pk2(sl2, sl2);
  f32x2 ncv[16];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const uint4 v = lds_v4(cw_a + 16u * k);
    ncv[2 * k] = pk2(-__uint_as_float(v.x), -__uint_as_float(v.y));
    ncv[2 * k + 1] = pk2(-__uint_as_float(v.z), -__uint_as_float(v.w));
  }
  f32x2 z2 = pk2(0.f, 0.f);
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const float2 v = up2(fma2(pk2(__uint_as_float(ra[2 * k]), __uint_as_float(ra[2 * k + 1])), s2, ncv[k]));
    z2 = add2(z2, pk2(ex2(v.x), ex2(v.y)));
  }
  float2 zz = up2(z2);
  float key = lg2(zz.x + zz.y);
  if (zz.x + zz.y < 0x1p-96f) {
    float mx = -INFINITY;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const float2 v = up2(fma2(pk2(__uint_as_float(ra[2 * k]), __uint_as_float(ra[2 * k + 1])), s2, ncv[k]));
      mx = fmax3(mx, v.x, v.y);
    }
    z2 = pk2(0.f, 0.f);
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const float2 v = up2(fma2(pk2(__uint_as_float(ra[2 * k]), __uint_as_float(ra[2 * k + 1])), s2, ncv[k]));
      z2 = add2(z2, pk2(ex2(v.x - mx), ex2(v.y - mx)));
    }
    zz = up2(z2);
    key = mx + lg2(zz.x + zz.y);
  }
  return key;
}

template <bool WIDE>
__device__ __noinline__ void pass_keys(uint32_t rank, uint32_t cs, Misc& ms, int pp, uint32_t tb, int ntl, int mc,
                                       int g0, float sl2, uint32_t keys_a, uint32_t ecol, bool eok) {
  const int tid = ctid<WIDE>(), lane = tid & 31, warp = tid >> 5, row = tid & (TM - 1);
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
  const uint32_t bar = bar_addr(ms.kbar[pp]);
  UnitState& ws = wslots<WIDE>(ms, pp, warp);
  const uint32_t cw_a = smem_u32(&ws.cw[warp & 3][0]);
  float kmin = INFINITY, kmax = -INFINITY;
  // After a wait gave up, this CTA sends nothing to the cluster.
  const uint32_t nr = aborted(ms) ? 0u : cs;
  auto emit = [&](int j, float key) {
    if (j < mc) {
      kmin = fminf(kmin, key);
      kmax = fmaxf(kmax, key);
      const uint32_t dst = keys_a + 4u * (uint32_t)(g0 + j);
#pragma unroll 1
      for (uint32_t r = 0; r < nr; ++r) st_async_b32(map_rank(dst, r), __float_as_uint(key), map_rank(bar, r));
    }
  };
  if (eok) {
    f32x2 fv[16];
    const uint32_t fw_a = smem_u32(&ws.fw[warp & 3][0]);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const uint4 f = lds_v4(fw_a + 16u * k);
      fv[2 * k] = pk2(__uint_as_float(f.x), __uint_as_float(f.y));
      fv[2 * k + 1] = pk2(__uint_as_float(f.z), __uint_as_float(f.w));
    }
#pragma unroll 1
    for (int t = unit_wg<WIDE>(); t < ntl; t += tile_step<WIDE>()) {
      uint32_t ra[32];
      tmem_ld32_issue(tb + ecol + lane_base + 32 * t, ra);
      tmem_wait_ld();
      f32x2 z2 = pk2(0.f, 0.f);
#pragma unroll
      for (int k = 0; k < 16; ++k) z2 = fma2(pk2(__uint_as_float(ra[2 * k]), __uint_as_float(ra[2 * k + 1])), fv[k], z2);
      const float2 zz = up2(z2);
      float key = lg2(zz.x + zz.y);
      const int j = t * TM + row;
      const bool slow = zz.x + zz.y < 0x1p-96f;
      if (__any_sync(0xffffffffu, slow && j < mc)) {
        // A tiny W: the exact key from the logits (the whole warp reloads them;
        // TMEM loads are warp-wide).
        uint32_t sa[32];
        tmem_ld32_issue(tb + lane_base + 32 * t, sa);
        tmem_wait_ld();
        const float k2 = key_from_logits(sa, cw_a, sl2);
        key = slow ? k2 : key;
      }
      emit(j, key);
    }
  } else {
#pragma unroll 1
    for (int t = unit_wg<WIDE>(); t < ntl; t += tile_step<WIDE>()) {
      uint32_t ra[32];
      tmem_ld32_issue(tb + lane_base + 32 * t, ra);
      tmem_wait_ld();
      emit(t * TM + row, key_from_logits(ra, cw_a, sl2));
    }
  }
  // The warp's key range goes with the keys (the Top-K's first bucket range).
  kmin = warp_min_f32(kmin);
  kmax = warp_max_f32(kmax);
  if (lane == 0) {
    const uint32_t dst = smem_u32(&ws.kmm[rank][warp & 3]);
#pragma unroll 1
    for (uint32_t r = 0; r < nr; ++r)
      st_async_v2(map_rank(dst, r), __float_as_uint(kmin), __float_as_uint(kmax), map_rank(bar, r));
  }
  // Every TMEM read of the scale is done before the Top-K's barriers.
  tc_fence_before();
}

// OR of a predicate over the unit's compute threads (a barrier of theirs).
template <bool WIDE>
__device__ __forceinline__ bool csync_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\tsetp.ne.u32 pi, %1, 0;\n\tbar.red.or.pred po, %2, %3, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v), "r"(kCsyncId + (WIDE ? 0u : (threadIdx.x >> 7))), "r"(32u * unit_warps<WIDE>())
      : "memory");
  return r != 0;
}

// Attention of unit pp over its key slice, tile by tile as the MMA thread
// completes each S tile: P = 2^(s sl2 - m) (bf16, P^T MN-major core matrices)
// into the unit's P double buffer for the MMA thread, so the value tiles are
// consumed while later key tiles still stream.  The stabiliser m_i (x sl2,
// log2 units) is the largest logit of query i in the first step's tiles (one
// tile, or one per warpgroup in the WIDE mode).  A later step whose logits
// exceed m_i by more than kRaise raises m_i to that step's maximum first (a
// decision taken jointly by the unit's threads; real inputs do not take it):
// every PV product issued so far completes, column i of the O^T accumulator
// and the running sums are scaled by 2^(m_old - m_new), and the step's P uses
// the new m.  Otherwise P <= 2^kRaise, which bf16 holds and fp32 sums over
// any key list accumulate without overflow; terms more than 2^126 below the
// stabiliser flush to zero, as they do below the largest term.  Rows past the
// slice get P = 0.  The final m -> us.mloc, the row sums of P -> us.lacc.
// WIDE: warpgroup w forms the P tiles t = w, w + 2, ... (always P buffer w).
constexpr float kRaise = 64.f;
template <bool WIDE>
__device__ __noinline__ void attn_online(Misc& ms, int* status, float sl2, uint8_t* pbase, int pp, uint32_t tb,
                                         int ntl, int mc, uint32_t& tpar, uint32_t ocol) {
  const int tid = ctid<WIDE>(), lane = tid & 31, warp = tid >> 5, row = tid & (TM - 1);
  const int wg = unit_wg<WIDE>();
  constexpr int NW = unit_warps<WIDE>();
  const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
  UnitState& us = ms.us[pp];
  UnitState& ws = wslots<WIDE>(ms, pp, warp);
  const f32x2 s2 = pk2(sl2, sl2);
  f32x2 nml[16], lsum2[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    nml[k] = pk2(0.f, 0.f);
    lsum2[k] = pk2(0.f, 0.f);
  }
  const int nsteps = (ntl + tile_step<WIDE>() - 1) / tile_step<WIDE>();
#pragma unroll 1
  for (int j = 0; j < nsteps; ++j) {
    const int t = j * tile_step<WIDE>() + wg;
    const bool has = t < ntl;  // warp-uniform
    uint32_t ra[32];
    if (has) {
      wait_or_abort(bar_addr(ms.tdone[pp][t]), (tpar >> t) & 1u, ms, status);
      tpar ^= 1u << t;
      tc_fence_after();
      tmem_ld32_issue(tb + lane_base + 32 * t, ra);
      tmem_wait_ld();
    }
    const bool valid = has && t * TM + row < mc;
    bool raise = j == 0;
    if (j > 0) {
      bool over = false;
      if (valid) {
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const float2 x = up2(fma2(pk2(__uint_as_float(ra[2 * k]), __uint_as_float(ra[2 * k + 1])), s2, nml[k]));
          over |= fmaxf(x.x, x.y) > kRaise;
        }
      }
      raise = csync_or<WIDE>(over);
    }
    if (raise) {
      // The step's column maxima: lane i of each warp keeps column i's.
      float mcol = -INFINITY;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float m = warp_max_f32(valid ? __uint_as_float(ra[i]) : -INFINITY);
        mcol = lane == i ? m : mcol;
      }
      ws.red[warp & 3][lane] = mcol;
      csync<WIDE>();
      if (tid < 32) {
        float m = -INFINITY;
#pragma unroll
        for (int w = 0; w < NW; ++w) m = fmaxf(m, wslots<WIDE>(ms, pp, w).red[w & 3][tid]);
        m *= sl2;
        const float mn = j == 0 ? m : fmaxf(us.mloc[tid], m);
        us.alpha[tid] = j == 0 ? 1.f : ex2(us.mloc[tid] - mn);
        us.mloc[tid] = mn;
      }
      csync<WIDE>();
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        nml[k] = pk2(-us.mloc[2 * k], -us.mloc[2 * k + 1]);
        lsum2[k] = mul2(lsum2[k], pk2(us.alpha[2 * k], us.alpha[2 * k + 1]));
      }
      if (j > 0 && wg == 0) {
        // Every PV product issued so far (through tile tl) completes; then the
        // accumulator's columns take the factor.  The tile's P is not
        // announced before, so the next product sees the scaled O^T.
        const int tl = j * tile_step<WIDE>() - 1;
        if (lane == 0) wait_or_abort(bar_addr(ms.pempty[pp][tl & 1]), (uint32_t)(tl >> 1) & 1u, ms, status);
        __syncwarp();
        tc_fence_after();
        uint32_t o[32];
        tmem_ld32_issue(ocol + lane_base, o);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * us.alpha[i]);
        tmem_st32(ocol + lane_base, o);
        tmem_wait_st();
        tc_fence_before();
      }
    }
    if (has) {
      const uint32_t pb = (uint32_t)t & 1u, pn = (uint32_t)t >> 1;
      if (t >= 2) {
        if (lane == 0) wait_or_abort(bar_addr(ms.pempty[pp][pb]), (pn - 1) & 1u, ms, status);
        __syncwarp();
      }
      uint32_t w[16];
      if (valid) {
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const float2 x = up2(fma2(pk2(__uint_as_float(ra[2 * k]), __uint_as_float(ra[2 * k + 1])), s2, nml[k]));
          const __nv_bfloat162 h2 = __floats2bfloat162_rn(ex2(x.x), ex2(x.y));
          lsum2[k] = add2(lsum2[k], pk2(__low2float(h2), __high2float(h2)));
          w[k] = *reinterpret_cast<const uint32_t*>(&h2);
        }
      } else {
#pragma unroll
        for (int k = 0; k < 16; ++k) w[k] = 0u;  // rows past the slice: P = 0
      }
      // P^T, MN-major core matrices: key group r / 8, query chunk ch.
      uint8_t* dst = pbase + pb * P_BYTES + (row >> 3) * 512 + (row & 7) * 16;
#pragma unroll
      for (int ch = 0; ch < 4; ++ch)
        *reinterpret_cast<uint4*>(dst + ch * 128) = make_uint4(w[4 * ch], w[4 * ch + 1], w[4 * ch + 2], w[4 * ch + 3]);
      fence_proxy_async();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_addr(ms.pfull[pp][pb]));
    }
  }
  float lsum[32];
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const float2 v = up2(lsum2[k]);
    lsum[2 * k] = v.x;
    lsum[2 * k + 1] = v.y;
  }
  ws.red[warp & 3][lane] = transpose_reduce32<false>(lsum, lane);
  csync<WIDE>();
  if (tid < 32) {
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < NW; ++w) sum += wslots<WIDE>(ms, pp, w).red[w & 3][tid];
    us.lacc[tid] = sum;
    if (nsteps == 0) us.mloc[tid] = -INFINITY;  // no keys in this CTA's slice
  }
  csync<WIDE>();
}

// Attention combine of unit pp: this CTA's partial O^T rows go to the CTA
// owning their head-dim slice (with the CTA's (m, l) per query), and this
// CTA combines the cluster's partials of its own slice and writes those
// columns of O (bf16).  The partials land in each owner's P buffers of the
// unit, which are free once the owner's own PV products are done; owners
// announce that before any partial is sent.
// (Run by one warpgroup of the unit: four warps, one per TMEM lane quarter.)
__device__ __noinline__ void attn_combine(Misc& ms, const FusedParams& p, uint32_t rank, uint32_t cs, int u,
                                          uint8_t* comb, UnitState& us, int pp, uint32_t ocol) {
  const int tid = threadIdx.x & (NCT - 1), warp = tid >> 5;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  uint32_t orow[32];
  tmem_ld32_issue(ocol + lane_base, orow);
  tmem_wait_ld();
  const uint32_t ready = bar_addr(ms.cready[pp]);
  // One arrival per CTA, each from its own thread (every thread has seen
  // this unit's PV products complete), so the remote arrivals overlap.  A CTA
  // whose wait gave up announces nothing and sends nothing: its P buffers
  // may still be in use, and the partials of others must not land there.
  if (tid < (int)cs && !aborted(ms)) mbar_arrive_cluster(map_rank(ready, (uint32_t)tid));
  wait_cluster_or_abort(ready, 0u, ms, p.status);
  const uint32_t comb_a = smem_u32(comb);
  const uint32_t cbar = bar_addr(ms.cbar[pp]);
  const bool send = !aborted(ms);  // every owner has announced its buffers free
  if (send) {
    // Owner of head-dim row d = tid, and the row's place in its buffer.
    int owner = tid * (int)cs / D;
    while (owner + 1 < (int)cs && dlo(owner + 1, cs) <= tid) ++owner;
    const int orows = dlo(owner + 1, cs) - dlo(owner, cs);
    const int dl = tid - dlo(owner, cs);
    const uint32_t dst = map_rank(comb_a + 4u * (uint32_t)(((int)rank * orows + dl) * NQ), (uint32_t)owner);
    const uint32_t rb = map_rank(cbar, (uint32_t)owner);
#pragma unroll
    for (int i = 0; i < 32; i += 4) st_async_v4(dst + 4u * i, orow[i], orow[i + 1], orow[i + 2], orow[i + 3], rb);
  }
  if (tid < 32 && send) {
    const uint32_t dst = smem_u32(&us.cstat[rank][tid]);
#pragma unroll 1
    for (uint32_t r = 0; r < cs; ++r)
      st_async_v2(map_rank(dst, r), __float_as_uint(us.mloc[tid]), __float_as_uint(us.lacc[tid]),
                  map_rank(cbar, r));
  }
  wait_cluster_or_abort(cbar, 0u, ms, p.status);
  // A thread always serves query qi = tid % 32: the weight 2^(m_r - M) of
  // every source CTA and the denominator are formed once.
  const int qi = tid & (NQ - 1);
  const uint32_t cst_a = smem_u32(&us.cstat[0][qi]);
  float2 st[MAXCS];
#pragma unroll
  for (int r = 0; r < MAXCS; ++r) {
    const uint2 v = lds_v2(cst_a + (uint32_t)(min(r, (int)cs - 1) * NQ * 8));
    st[r] = make_float2(__uint_as_float(v.x), __uint_as_float(v.y));
  }
  float M = -INFINITY;
#pragma unroll
  for (int r = 0; r < MAXCS; ++r)
    if (r < (int)cs && st[r].y > 0.f) M = fmaxf(M, st[r].x);
  float f[MAXCS], den = 0.f;
#pragma unroll
  for (int r = 0; r < MAXCS; ++r) {
    f[r] = (r < (int)cs && st[r].y > 0.f) ? ex2(st[r].x - M) : 0.f;  // a CTA with no keys contributes nothing
    den = fmaf(st[r].y, f[r], den);
  }
  const float inv = 1.f / den;
  bf16* ob = p.O + (int64_t)(u / p.H) * p.osb + (int64_t)(u % p.H) * p.osh;
  const int d0 = dlo((int)rank, cs), rows = dlo((int)rank + 1, cs) - d0;
  auto out = [&](int dl) {
    float n = 0.f;
#pragma unroll
    for (int r = 0; r < MAXCS; ++r)
      if (r < (int)cs) n = fmaf(lds_f32(comb_a + 4u * (uint32_t)((r * rows + dl) * NQ + qi)), f[r], n);
    return n * inv;
  };
  // A slice of 32, 64 or 128 rows (clusters of 4, 2, 1): warp w writes rows
  // [w rows / 4, (w + 1) rows / 4) of its query, 16 bytes a store; otherwise
  // one element a store.
  const bool vec = rows % (NCW * 8) == 0 && d0 % 8 == 0 && p.oss % 8 == 0 &&
                   (reinterpret_cast<uintptr_t>(ob) & 15) == 0;
  if (qi < p.q && vec) {
    const int per = rows / NCW, db = warp * per;
#pragma unroll 1
    for (int c0 = 0; c0 < per; c0 += 8) {
      uint32_t w4[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const __nv_bfloat162 h = __floats2bfloat162_rn(out(db + c0 + 2 * e), out(db + c0 + 2 * e + 1));
        w4[e] = *reinterpret_cast<const uint32_t*>(&h);
      }
      *reinterpret_cast<uint4*>(ob + (int64_t)qi * p.oss + d0 + db + c0) = make_uint4(w4[0], w4[1], w4[2], w4[3]);
    }
  } else if (qi < p.q) {
#pragma unroll 1
    for (int dl = tid >> 5; dl < rows; dl += NCT / NQ) ob[(int64_t)qi * p.oss + d0 + dl] = __float2bfloat16_rn(out(dl));
  }
}

// The compute warps of unit pp = threadIdx.x / NCT of the cluster's units.
// WIDE: both warpgroups serve the cluster's one unit.
template <bool WIDE>
__device__ void compute_role(const Ctx& c, const FusedParams& p) {
  Misc& ms = *c.ms;
  constexpr int TN = 32 * unit_warps<WIDE>();  // the unit's compute threads
  const int tid = ctid<WIDE>();
  const int pp = WIDE ? 0 : threadIdx.x / NCT;
  if (pp >= c.np) return;
  UnitState& us = ms.us[pp];
  uint8_t* ubuf = c.smem + c.ly.p + pp * UNIT_P_BYTES;  // P buffers, Top-K scratch, combine buffer
  const uint32_t sc_a = smem_u32(ubuf);
  const uint32_t tb = c.tmem + pp * p.ucols;
  const int u = c.u0 + pp;
  const float sl2 = p.scale_log2;
  int64_t sets_off = 0;  // the level sets of the scales above this launch's first
  for (int l = p.L; l > c.lev_top; --l) sets_off += p.keep[l];
  // The unit's mdone barrier completes one phase, when the attention's PV
  // products are done (the MMA thread commits it only for a non-empty slice).
  auto wait_mdone = [&]() {
    wait_or_abort(bar_addr(ms.mdone[pp]), 0u, ms, p.status);
    tc_fence_after();
  };
  // A launch that starts below the top scale (its rows dense, so the
  // producers do not need it): the previous selection J_{lev_top+1}, for the
  // first Top-K's winners, from the children list it was handed (halved).
  // The Top-K's first barrier orders it.
  if (c.lev_top < p.L) {
    const int32_t* src = p.jin + (int64_t)u * p.jstride;
    int32_t* Jp = unit_J(c, p, pp, c.lev_top + 1);
#pragma unroll 1
    for (int i = tid; i < p.keep[c.lev_top + 1]; i += TN) Jp[i] = src[2 * i] >> 1;
  }
  // The first pass through the Top-K's code fetches its instructions from
  // memory, where they queue behind the first scale's row streams (several us
  // at 32K).  In a two-unit cluster unit 1's warpgroup, which waits for its
  // first rows until unit 0's have streamed, runs the Top-K once on synthetic
  // keys with the first scale's list length, so unit 0's first selection
  // finds the code cached (measured: 32K step 82.6 -> 80.5 us; in one-unit
  // clusters the warm-up delays the unit's own first scale and the 128K step
  // was 2 us slower).  Its key buffer is the one the scale below receives,
  // which no CTA fills before this one has finished its first selection; the
  // Top-K leaves its scratch cleared.
  if (!WIDE && pp == 1 && c.lev_top == p.L && c.lev_top > c.lev_end) {
    const int m0 = m_total(p, c.lev_top);
    int32_t* wk = unit_J(c, p, pp, c.lev_top - 1);
    // 512 distinct values, each several times: one bucket round whose
    // boundary bucket holds more keys than it needs, like real keys.
#pragma unroll 1
    for (int i = tid; i < m0; i += TN) wk[i] = __float_as_int((float)((((uint32_t)i * 2654435761u) >> 8) & 511u));
    csync<WIDE>();
    select_topk<WIDE>(smem_u32(wk), m0, p.keep[c.lev_top], 0u, 1, sc_a, 0.f, 511.f);
  }
  uint32_t tpar = 0;  // parity of each scale-tile barrier's next phase
#pragma unroll 1
  for (int lev = c.lev_top; lev >= c.lev_end; --lev) {
    const uint32_t ph = (uint32_t)(c.lev_top - lev) & 1u;  // phase of the per-scale barriers
    const int m = m_total(p, lev);
    int g0, mc;
    scale_slice(m, c.rank, c.cs, g0, mc);
    const int ntl = tiles_of(mc);
    const int kb = p.keep[lev];
    int32_t* J = unit_J(c, p, pp, lev);  // receives this scale's keys, then its selection
    const uint32_t keys_a = smem_u32(J);
    const bool eok = scale_sums<WIDE>(c.rank, c.cs, ms, pp, tb, ntl, mc, sl2, p.ecol, tpar, p.status);
    wait_cluster_or_abort(bar_addr(ms.xbar[pp]), ph, ms, p.status);
    // This phase is complete for tid 0, so the arrival arms the next one.
    // After a wait gave up the phase may still be pending (its bytes never
    // came): a second arrival would then underflow the phase's arrival
    // count, so an aborted CTA arms nothing.
    if (tid == 0 && lev > c.lev_end && !aborted(ms)) mbar_arrive_expect_tx(bar_addr(ms.xbar[pp]), c.cs * NQ * 8u);
    warp_normaliser<WIDE>(ms, pp, c.cs, p.q);
    pass_keys<WIDE>(c.rank, c.cs, ms, pp, tb, ntl, mc, g0, sl2, keys_a, p.ecol, eok);
    wait_cluster_or_abort(bar_addr(ms.kbar[pp]), ph, ms, p.status);
    // The keys' range from the cluster warps' (min, max).
    float lo, hi;
    {
      constexpr int NW = unit_warps<WIDE>();
      const int lane = tid & 31;
      float2 mm = make_float2(INFINITY, -INFINITY);
#pragma unroll 1
      for (int e = lane; e < (int)c.cs * NW; e += 32) {  // entry (CTA e / NW, warp e % NW)
        const int w = e % NW;
        const uint2 v = lds_v2(smem_u32(&wslots<WIDE>(ms, pp, w).kmm[e / NW][w & 3]));
        mm = make_float2(fminf(mm.x, __uint_as_float(v.x)), fmaxf(mm.y, __uint_as_float(v.y)));
      }
      lo = warp_min_f32(mm.x);
      hi = warp_max_f32(mm.y);
    }
    // Eq. 9: Top-K (the same result in every CTA of the cluster).
    select_topk<WIDE>(keys_a, m, kb, smem_u32(unit_J(c, p, pp, lev + 1)), lev == p.L, sc_a, lo, hi);
    if (tid == 0) {
      if (lev > c.lev_end && !aborted(ms))  // as for xbar above
        mbar_arrive_expect_tx(bar_addr(ms.kbar[pp]),
                              4u * (uint32_t)m_total(p, lev - 1) + c.cs * unit_warps<WIDE>() * 8u);
      mbar_arrive(bar_addr(ms.jready[pp]));  // the selection is complete (the Top-K ends on a barrier)
    }
    if (c.rank == 0) {
      int32_t* ls = p.level_sets ? p.level_sets + (int64_t)u * p.sets_stride + sets_off : nullptr;
      if (lev >= 1 && ls) {
#pragma unroll 1
        for (int i = tid; i < kb; i += TN) ls[i] = J[i];
      }
      if (lev == c.lev_end && !p.final_sel) {
        // A launch that ends above the final scale hands on the children of
        // its last selection (the next launch's candidates).
        int32_t* out = p.jout + (int64_t)u * p.jstride;
#pragma unroll 1
        for (int t = tid; t < 2 * kb; t += TN) out[t] = 2 * J[t >> 1] + (t & 1);
      } else if (lev == c.lev_end) {
        // mu^0: the children of J^1, or the trimmed level-0 selection.
        const int kk = p.keep[0];
        int32_t* out = p.idx + (int64_t)u * kk;
        int32_t* ls0 = ls ? ls + (lev >= 1 ? kb : 0) : nullptr;
#pragma unroll 1
        for (int t = tid; t < kk; t += TN) {
          const int tok = p.trim ? J[t] : 2 * J[t >> 1] + (t & 1);
          out[t] = tok;
          if (ls0) ls0[t] = tok;
        }
      }
    }
    if (lev >= 1) sets_off += kb;
  }
  if (!p.attn) return;

  // Attention: S of the key slice, P for the MMA thread, then the combine.
  int a0, mc;
  attn_slice(p.keep[0] + p.ng, c.rank, c.cs, a0, mc);
  const int ntl = tiles_of(mc);
  attn_online<WIDE>(ms, p.status, sl2, ubuf, pp, tb, ntl, mc, tpar, tb + p.ucols - 32);
  if (ntl > 0) wait_mdone();  // every PV product of the unit is done
  if (unit_wg<WIDE>() != 0) return;  // one warpgroup combines
  attn_combine(ms, p, c.rank, c.cs, u, ubuf, us, pp, tb + p.ucols - 32);
}

template <int S, bool WIDE>
__global__ void __launch_bounds__(NT, 1) wf_fused_kernel(const __grid_constant__ FusedParams p) {
  extern __shared__ __align__(1024) uint8_t smem[];
  Ctx c;
  c.smem = smem;
  c.ly = smem_layout(S, p.P, p.cmax, p.kmax);
  c.ms = reinterpret_cast<Misc*>(smem + c.ly.misc);
  Misc& ms = *c.ms;
  c.rank = cluster_rank();
  c.cs = cluster_size();
  c.u0 = (int)cluster_id_x() * p.P;
  c.np = min(p.P, p.U - c.u0);
  c.lev_top = p.lev_top;
  c.lev_end = p.lev_bot;
  c.stages = S;
  const int tid = threadIdx.x, warp = tid >> 5;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(bar_addr(ms.full[s]), NPT);
      mbar_init(bar_addr(ms.empty[s]), 1);
    }
    for (int pp = 0; pp < MAXP; ++pp) {
      mbar_init(bar_addr(ms.mdone[pp]), 1);
      mbar_init(bar_addr(ms.jready[pp]), 1);
      mbar_init(bar_addr(ms.xbar[pp]), 1);
      mbar_init(bar_addr(ms.kbar[pp]), 1);
      for (int t = 0; t < MAXT; ++t) mbar_init(bar_addr(ms.tdone[pp][t]), 1);
    }
    for (int pp = 0; pp < MAXP; ++pp) {
      for (int i = 0; i < 2; ++i) {
        mbar_init(bar_addr(ms.pfull[pp][i]), NCW);
        mbar_init(bar_addr(ms.pempty[pp][i]), 1);
      }
      mbar_init(bar_addr(ms.cbar[pp]), 1);
      mbar_init(bar_addr(ms.cready[pp]), c.cs);
    }
    mbar_init(bar_addr(ms.qfull), NPT);
    mbar_init(bar_addr(ms.stallbar), 1);
    mbar_init(bar_addr(ms.drainbar), 1);
    ms.wait_limit = p.wait_limit;
    ms.abort = 0;
    fence_mbar_init();
  }
  __syncthreads();  // this CTA's barriers exist
  if (warp > MMA_WARP) {
    // The producers touch only this CTA's ring and barriers, so they start at
    // once: they join the cluster barrier's first phase now (nothing of theirs
    // needs ordering before other CTAs' remote stores) and wait for it at the
    // end, while the other warps finish the set-up.
    cluster_arrive_relaxed();
    grid_dep_wait();  // the rows come from the grids before a programmatic launch
    producer_role<S>(c, p);
    cluster_wait();
  } else {
    constexpr int NS = NT - NPT;  // the set-up threads: compute warps and the MMA warp
    if (tid == 0) {
      // Arm the first phase of every receive barrier (bytes this CTA expects).
      for (int pp = 0; pp < c.np; ++pp) {
        mbar_arrive_expect_tx(bar_addr(ms.xbar[pp]), c.cs * NQ * 8u);
        mbar_arrive_expect_tx(bar_addr(ms.kbar[pp]),
                              4u * (uint32_t)m_total(p, c.lev_top) + c.cs * unit_warps<WIDE>() * 8u);
        const uint32_t rows = (uint32_t)(dlo((int)c.rank + 1, c.cs) - dlo((int)c.rank, c.cs));
        mbar_arrive_expect_tx(bar_addr(ms.cbar[pp]), c.cs * rows * NQ * 4u + c.cs * NQ * 8u);
      }
    }
    if (warp == MMA_WARP) {
      tmem_alloc(smem_u32(&ms.tmem_base), p.tmem_cols);
      tmem_relinquish();
    }
    // The Top-K scratch starts zeroed (histogram, list counter, masks).
    for (int pp = 0; pp < c.np; ++pp) {
      uint8_t* sc = smem + c.ly.p + pp * UNIT_P_BYTES;
      for (int e = tid; e < (int)((sizeof(SelScratch) + 15) / 16); e += NS)
        *reinterpret_cast<uint4*>(sc + 16 * e) = make_uint4(0, 0, 0, 0);
    }
    // Global memory only after the grids this launch depends on are done (the
    // set-up above overlaps their tail when the launch is programmatic).
    grid_dep_wait();
    grid_dep_launch();
    tc_fence_before();
    named_sync(kSetupSyncId, NS);
    tc_fence_after();
    c.tmem = ms.tmem_base;
    cluster_sync();  // every CTA's barriers are armed before any remote arrival
    if (warp < MMA_WARP) {
      compute_role<WIDE>(c, p);
    } else {
      if ((tid & 31) == 0) mma_role<S>(c, p);
      __syncwarp();
    }
  }

  tc_fence_before();
  __syncthreads();
  // No CTA leaves while another may still address its shared memory.
  cluster_arrive();
  cluster_wait();
  if (warp == MMA_WARP) {
    if (aborted(ms)) {
      // After a wait gave up, asynchronous stores from cluster CTAs that were
      // not waited for may still be landing in this CTA's shared memory:
      // every CTA has issued its last one (all are past the cluster
      // barrier), so a short pause lets them complete before the CTA leaves.
      const unsigned long long t0 = globaltimer_ns();
      while (globaltimer_ns() - t0 < 20000ull) {
      }
    }
    tc_fence_after();
    tmem_dealloc(c.tmem, p.tmem_cols);
  }
}


// ---------------------------------------------------------------------------
// Grouped query heads (reading 21): the filter of one key head for the
// stacked query rows of its G query heads, W_j summed over every row of the
// group (Eq. 7-11; Dream-7B's 7 query heads per key head give 224 rows).
// ---------------------------------------------------------------------------
//
// One cluster of CS CTAs per (batch, key head) unit, both compute warpgroups
// on the unit, the same producers and Top-K as the one-head kernel.  The
// stacked query block (G q rows in chunks of 32) is the N side of the MMAs: a
// tile's logits take 32 nch TMEM columns, so the CTA holds two tiles at a
// time (warpgroup w reads region w, the tiles t = w, w + 2, ...), and every
// scale runs two passes over its rows, the second re-streamed (from L2):
//   1. per query column, a stabiliser (x sl2) and the sum of exponentials
//      over the CTA's rows: each tile's exponentials are taken relative to the
//      largest logit of the query chunk among the warp's rows of that tile
//      (a column whose terms would all flush to zero takes its own maximum),
//      and merged as they come, so nothing overflows; the warps' statistics
//      merge into the CTA's (M, S),
//      which the cluster exchanges into the normalisers c_i = M + log2 S;
//   2. each row's ranking key log2 W_j = log2 sum_i 2^(l_ij sl2 - c_i) over
//      all stacked rows (a running maximum over the chunks keeps tiny sums
//      exact), all-gathered, then the Top-K (Eq. 9).
// The selection is written as mu^0 (and the level sets); the attention runs
// afterwards on the per-stage tensor-core kernels.
constexpr int GQ_MAXCH = 8;  // chunks of 32 stacked query rows (G q <= 256)

struct GqaLayout {
  uint32_t q, sc, misc, wst, xst, cvec, buf, bufw, total;
};
__host__ __device__ inline GqaLayout gqa_layout(int stages, int nch, int cs, int cmax, int kmax) {
  GqaLayout l;
  const uint32_t nq = 32u * (uint32_t)nch;
  l.q = (uint32_t)stages * TILE_BYTES;
  l.sc = l.q + (uint32_t)nch * Q_BYTES;                            // Top-K scratch
  l.misc = (l.sc + (uint32_t)sizeof(SelScratch) + 127u) / 128u * 128u;
  l.wst = (l.misc + (uint32_t)sizeof(Misc) + 15u) / 16u * 16u;     // [8][nq] float2: each warp's column statistics
  l.xst = l.wst + 8u * nq * 8u;                                    // [cs][nq] float2: every CTA's (M, S) per column
  l.cvec = l.xst + (uint32_t)cs * nq * 8u;                         // [nq] float: the normalisers c_i
  l.buf = (l.cvec + nq * 4u + 127u) / 128u * 128u;                 // two key / selection buffers
  l.bufw = (uint32_t)((max(cmax, kmax) + 3) / 4 * 4);
  l.total = l.buf + 2u * 4u * l.bufw;
  return l;
}

// (m, s) pairs of sums of 2^(x - m): the pair of their union.
__device__ __forceinline__ float2 merge_ms(float2 a, float2 b) {
  if (!(b.y > 0.f)) return a;
  if (!(a.y > 0.f)) return b;
  const float M = fmaxf(a.x, b.x);
  return make_float2(M, a.y * ex2(a.x - M) + b.y * ex2(b.x - M));
}

template <int S>
__device__ void gqa_producer_role(const Ctx& c, const FusedParams& p) {
  Misc& ms = *c.ms;
  const int pt = threadIdx.x - P0;
  // The stacked query block first: row i = g q + r is row r of query head
  // h G + g; chunk ch holds rows 32 ch .. 32 ch + 31 (K-major core matrices),
  // rows >= G q zero-filled.
  const int64_t b = c.u0 / p.H, h = c.u0 % p.H;
  const int nq = p.G * p.q;
  for (int ch = 0; ch < p.nch; ++ch) {
    const uint32_t sq = smem_u32(c.smem + c.ly.q + ch * Q_BYTES);
    for (int e = pt; e < NQ * (D / 8); e += NPT) {
      const int rr = e & 7, c16 = (e >> 3) & (D / 8 - 1), g8 = e >> 7;
      const int i = ch * NQ + g8 * 8 + rr;
      const int ic = min(i, nq - 1), hd = ic / p.q, r = ic - hd * p.q;
      const bf16* src = p.Q + b * p.qsb + (h * p.G + hd) * p.qsh + (int64_t)r * p.qss + c16 * 8;
      cp_async16_zfill(sq + (uint32_t)(g8 * QGRP + c16 * 128 + rr * 16), src, i < nq);
    }
  }
  cp_async_arrive_noinc(bar_addr(ms.qfull));
  int it = 0;
  for (int lev = c.lev_top; lev >= c.lev_end; --lev) {
    if (lev != c.lev_top) wait_or_abort(bar_addr(ms.jready[0]), (uint32_t)(c.lev_top - lev - 1) & 1u, ms, p.status);
    int g0, mc;
    scale_slice(m_total(p, lev), c.rank, c.cs, g0, mc);
    const int ntl = tiles_of(mc);
    const RowSrc src = scale_src(c, p, 0, lev, g0, mc);
    produce<S>(ms, p.status, smem_u32(c.smem), it, 0, ntl, src, pt);  // pass 1
    it += ntl;
    // Pass 2: the same rows again, but for the last two tiles, which stay in
    // TMEM from pass 1.
    const int nre = max(ntl - 2, 0);
    produce<S>(ms, p.status, smem_u32(c.smem), it, 0, nre, src, pt);
    it += nre;
  }
  cp_async_wait_all();
}

// Both passes of every scale: tile t's logits for every query chunk into
// TMEM region t % 2 once the warpgroup reading that region has released it.
template <int S>
__device__ void gqa_mma_role(const Ctx& c, const FusedParams& p) {
  Misc& ms = *c.ms;
  if (p.stall) wait_or_abort(bar_addr(ms.stallbar), 0u, ms, p.status);
  wait_or_abort(bar_addr(ms.qfull), 0u, ms, p.status);
  fence_proxy_async();
  const uint32_t sq = smem_u32(c.smem + c.ly.q);
  const uint32_t rcols = 32u * (uint32_t)p.nch;
  const uint32_t idesc = idesc_bf16(TM, 32 * p.nch, 0, 0);  // A = rows (K-major), B = the stacked queries (K-major)
  uint32_t used[2] = {0u, 0u};
  int it = 0;
  for (int lev = c.lev_top; lev >= c.lev_end; --lev) {
    int g0, mc;
    scale_slice(m_total(p, lev), c.rank, c.cs, g0, mc);
    const int ntl = tiles_of(mc);
    // Pass 1: every tile; pass 2: all but the last two, whose logits are
    // still in their regions (each issue into a region is released once by
    // the warpgroup reading it, the kept tiles after their second reading).
    const int nre = max(ntl - 2, 0);
#pragma unroll 1
    for (int k = 0; k < ntl + nre; ++k) {
      const int t = k < ntl ? k : k - ntl, r = t & 1, slot = it + k, s = slot % S;
      if (used[r] > 0) wait_or_abort(bar_addr(ms.rfree[r]), (used[r] - 1u) & 1u, ms, p.status);
      ++used[r];
      wait_or_abort(bar_addr(ms.full[s]), (uint32_t)(slot / S) & 1u, ms, p.status);
      fence_proxy_async();
      if (!aborted(ms)) {
        tc_fence_after();
        const uint32_t st = smem_u32(c.smem) + s * TILE_BYTES;
        // One MMA per K step over every query chunk at once (N = 32 nch: the
        // chunks' 8-row groups follow each other at the same stride).
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_bf16(c.tmem + (uint32_t)r * rcols, smem_desc_sw128(st + h * HALF_BYTES + kk * 32, 16, 1024),
                     smem_desc(sq + (4 * h + kk) * 256, 128, QGRP), idesc, (h | kk) != 0);
      }
      mma_commit(bar_addr(ms.empty[s]));
      mma_commit(bar_addr(ms.rdone[r]));
    }
    it += ntl + nre;
  }
  mma_commit(bar_addr(ms.drainbar));
  (void)mbar_wait_bounded(bar_addr(ms.drainbar), 0u, kDefaultWaitLimit);
}

__device__ void gqa_compute_role(const Ctx& c, const FusedParams& p, const GqaLayout gl) {
  Misc& ms = *c.ms;
  constexpr int TN = 32 * unit_warps<true>();
  const int tid = ctid<true>(), lane = tid & 31, warp = tid >> 5, wg = tid >> 7, qd = warp & 3, row = tid & (TM - 1);
  const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
  const int nch = p.nch, nqp = 32 * nch, nq = p.G * p.q;
  const uint32_t treg = c.tmem + (uint32_t)wg * 32u * (uint32_t)nch;  // this warpgroup's TMEM region
  const uint32_t sc_a = smem_u32(c.smem + gl.sc);
  float2* wst = reinterpret_cast<float2*>(c.smem + gl.wst);
  float2* xst = reinterpret_cast<float2*>(c.smem + gl.xst);
  float* cvec = reinterpret_cast<float*>(c.smem + gl.cvec);  // -c_i
  const uint32_t ncvec_a = smem_u32(cvec);
  const float sl2 = p.scale_log2;
  const int u = c.u0;
  int64_t sets_off = 0;
  uint32_t dpar = 0;  // parity of the next phase of this warpgroup's rdone barrier
  // body(ra, ch) for every query chunk of the tile in the region.
  auto for_chunks = [&](auto&& body) {
#pragma unroll 1
    for (int ch = 0; ch < nch; ++ch) {
      uint32_t ra[32];
      tmem_ld32_issue(treg + 32u * ch + lane_base, ra);
      tmem_wait_ld();
      body(ra, ch);
    }
  };
#pragma unroll 1
  for (int lev = c.lev_top; lev >= c.lev_end; --lev) {
    const uint32_t ph = (uint32_t)(c.lev_top - lev) & 1u;
    const int m = m_total(p, lev);
    int g0, mc;
    scale_slice(m, c.rank, c.cs, g0, mc);
    const int ntl = tiles_of(mc);
    const int kb = p.keep[lev];
    int32_t* J = unit_J(c, p, 0, lev);
    const uint32_t keys_a = smem_u32(J);

    // Pass 1: this warp's (stabiliser, sum) of each query column over its
    // rows, in its own slots (lane l: column 32 ch + l of every chunk).
    float2* wsw = wst + warp * nqp;
#pragma unroll 1
    for (int ch = 0; ch < nch; ++ch) wsw[32 * ch + lane] = make_float2(-INFINITY, 0.f);
    // This warpgroup's last tile stays in its region for pass 2.
    const int tkeep = ntl - 1 - wg >= 0 ? wg + (ntl - 1 - wg) / 2 * 2 : -1;
#pragma unroll 1
    for (int t = wg; t < ntl; t += 2) {
      wait_or_abort(bar_addr(ms.rdone[wg]), dpar, ms, p.status);
      dpar ^= 1u;
      tc_fence_after();
      const bool valid = t * TM + row < mc;
      for_chunks([&](const uint32_t (&ra)[32], int ch) {
        // Exponentials relative to the chunk's largest logit among the warp's
        // rows (one warp-wide max), summed per column across the rows.
        float e[32];
        float vm = -INFINITY;
#pragma unroll
        for (int i = 0; i < 32; i += 2) vm = fmax3(vm, __uint_as_float(ra[i]), __uint_as_float(ra[i + 1]));
        float tm = warp_max_f32(valid ? vm : -INFINITY);
        const float ntm = -tm * sl2;
#pragma unroll
        for (int i = 0; i < 32; ++i) e[i] = valid ? ex2(fmaf(__uint_as_float(ra[i]), sl2, ntm)) : 0.f;
        float ts = transpose_reduce32<false>(e, lane);  // lane l: column l's sum
        // A column whose every term flushed to zero (logits more than ~126
        // below the chunk's largest, in log2 units) is summed again against
        // each column's own maximum (the warp decides together).
        if (__any_sync(0xffffffffu, !(ts > 0.f) && tm > -INFINITY)) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float v = valid ? __uint_as_float(ra[i]) : -INFINITY;
            const float mi = warp_max_f32(v);  // column i's largest logit among the warp's rows
            tm = lane == i ? mi : tm;
            e[i] = valid ? ex2((v - mi) * sl2) : 0.f;
          }
          ts = transpose_reduce32<false>(e, lane);
        }
        wsw[32 * ch + lane] = merge_ms(wsw[32 * ch + lane], make_float2(tm * sl2, ts));
      });
      tc_fence_before();
      __syncwarp();
      if (lane == 0 && t != tkeep) mbar_arrive(bar_addr(ms.rfree[wg]));
    }
    // The eight warps' statistics -> the CTA's (M, S) per column, sent to
    // every cluster CTA.
    csync<true>();
    {
      const uint32_t xbar = bar_addr(ms.xbar[0]);
      const uint32_t nr = aborted(ms) ? 0u : c.cs;  // after a wait gave up, nothing goes to the cluster
#pragma unroll 1
      for (int col = tid; col < nqp; col += TN) {
        float2 a = wst[col];
#pragma unroll
        for (int w8 = 1; w8 < 8; ++w8) a = merge_ms(a, wst[w8 * nqp + col]);
        const uint32_t dst = smem_u32(&xst[c.rank * nqp + col]);
#pragma unroll 1
        for (uint32_t r = 0; r < nr; ++r)
          st_async_v2(map_rank(dst, r), __float_as_uint(a.x), __float_as_uint(a.y), map_rank(xbar, r));
      }
    }
    wait_cluster_or_abort(bar_addr(ms.xbar[0]), ph, ms, p.status);
    if (tid == 0 && lev > c.lev_end && !aborted(ms))
      mbar_arrive_expect_tx(bar_addr(ms.xbar[0]), c.cs * (uint32_t)nqp * 8u);
#pragma unroll 1
    for (int col = tid; col < nqp; col += TN) {
      float2 a = make_float2(-INFINITY, 0.f);
#pragma unroll 1
      for (uint32_t r = 0; r < c.cs; ++r) a = merge_ms(a, xst[r * nqp + col]);
      cvec[col] = col < nq ? -(a.x + lg2(a.y)) : -INFINITY;  // -c_i; padded rows weigh 0
    }
    csync<true>();

    // Pass 2: each row's ranking key over every stacked query row.
    float kmin = INFINITY, kmax = -INFINITY;
    const uint32_t kbar = bar_addr(ms.kbar[0]);
    const uint32_t nr = aborted(ms) ? 0u : c.cs;
    // The kept tile first (its logits are in the region), then the earlier
    // tiles as the MMA thread re-issues them.
#pragma unroll 1
    for (int k = 0; tkeep >= 0 && k <= tkeep / 2; ++k) {
      const int t = k == 0 ? tkeep : wg + 2 * (k - 1);
      if (k > 0) {
        wait_or_abort(bar_addr(ms.rdone[wg]), dpar, ms, p.status);
        dpar ^= 1u;
        tc_fence_after();
      }
      // Every exponent l sl2 - c_i is at most 0 (c_i is the log of a sum that
      // holds the row's own term), so the sum is taken unshifted; a row whose
      // sum is tiny (below 2^-96, where flushed terms could matter) is taken
      // again shifted by its largest exponent (the warp together).
      float rm = 0.f, rs = 0.f;
      for_chunks([&](const uint32_t (&ra)[32], int ch) {
        float z = 0.f;
#pragma unroll
        for (int k4 = 0; k4 < 8; ++k4) {
          const uint4 cv = lds_v4(ncvec_a + 16u * (uint32_t)(8 * ch + k4));
          z += ex2(fmaf(__uint_as_float(ra[4 * k4]), sl2, __uint_as_float(cv.x)));
          z += ex2(fmaf(__uint_as_float(ra[4 * k4 + 1]), sl2, __uint_as_float(cv.y)));
          z += ex2(fmaf(__uint_as_float(ra[4 * k4 + 2]), sl2, __uint_as_float(cv.z)));
          z += ex2(fmaf(__uint_as_float(ra[4 * k4 + 3]), sl2, __uint_as_float(cv.w)));
        }
        rs += z;
      });
      if (__any_sync(0xffffffffu, rs < 0x1p-96f && t * TM + row < mc)) {
        float mxr = -INFINITY;
        for_chunks([&](const uint32_t (&ra)[32], int ch) {
#pragma unroll
          for (int k4 = 0; k4 < 8; ++k4) {
            const uint4 cv = lds_v4(ncvec_a + 16u * (uint32_t)(8 * ch + k4));
            mxr = fmaxf(mxr, fmax3(fmaf(__uint_as_float(ra[4 * k4]), sl2, __uint_as_float(cv.x)),
                                   fmaf(__uint_as_float(ra[4 * k4 + 1]), sl2, __uint_as_float(cv.y)),
                                   fmaxf(fmaf(__uint_as_float(ra[4 * k4 + 2]), sl2, __uint_as_float(cv.z)),
                                         fmaf(__uint_as_float(ra[4 * k4 + 3]), sl2, __uint_as_float(cv.w)))));
          }
        });
        float z2 = 0.f;
        for_chunks([&](const uint32_t (&ra)[32], int ch) {
#pragma unroll
          for (int k4 = 0; k4 < 8; ++k4) {
            const uint4 cv = lds_v4(ncvec_a + 16u * (uint32_t)(8 * ch + k4));
            z2 += ex2(fmaf(__uint_as_float(ra[4 * k4]), sl2, __uint_as_float(cv.x)) - mxr);
            z2 += ex2(fmaf(__uint_as_float(ra[4 * k4 + 1]), sl2, __uint_as_float(cv.y)) - mxr);
            z2 += ex2(fmaf(__uint_as_float(ra[4 * k4 + 2]), sl2, __uint_as_float(cv.z)) - mxr);
            z2 += ex2(fmaf(__uint_as_float(ra[4 * k4 + 3]), sl2, __uint_as_float(cv.w)) - mxr);
          }
        });
        if (rs < 0x1p-96f) {
          rm = mxr;
          rs = z2;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar_addr(ms.rfree[wg]));
      const int j = t * TM + row;
      if (j < mc) {
        const float key = rm + lg2(rs);
        kmin = fminf(kmin, key);
        kmax = fmaxf(kmax, key);
        const uint32_t dst = keys_a + 4u * (uint32_t)(g0 + j);
#pragma unroll 1
        for (uint32_t r = 0; r < nr; ++r) st_async_b32(map_rank(dst, r), __float_as_uint(key), map_rank(kbar, r));
      }
    }
    kmin = warp_min_f32(kmin);
    kmax = warp_max_f32(kmax);
    if (lane == 0) {
      const uint32_t dst = smem_u32(&wslots<true>(ms, 0, warp).kmm[c.rank][warp & 3]);
#pragma unroll 1
      for (uint32_t r = 0; r < nr; ++r)
        st_async_v2(map_rank(dst, r), __float_as_uint(kmin), __float_as_uint(kmax), map_rank(kbar, r));
    }
    wait_cluster_or_abort(kbar, ph, ms, p.status);
    float lo, hi;
    {
      constexpr int NW = unit_warps<true>();
      float2 mm = make_float2(INFINITY, -INFINITY);
#pragma unroll 1
      for (int e = lane; e < (int)c.cs * NW; e += 32) {  // entry (CTA e / NW, warp e % NW)
        const int w = e % NW;
        const uint2 v = lds_v2(smem_u32(&wslots<true>(ms, 0, w).kmm[e / NW][w & 3]));
        mm = make_float2(fminf(mm.x, __uint_as_float(v.x)), fmaxf(mm.y, __uint_as_float(v.y)));
      }
      lo = warp_min_f32(mm.x);
      hi = warp_max_f32(mm.y);
    }
    // Eq. 9: Top-K (the same result in every CTA of the cluster).
    select_topk<true>(keys_a, m, kb, smem_u32(unit_J(c, p, 0, lev + 1)), lev == p.L, sc_a, lo, hi);
    if (tid == 0) {
      if (lev > c.lev_end && !aborted(ms))
        mbar_arrive_expect_tx(kbar, 4u * (uint32_t)m_total(p, lev - 1) + c.cs * unit_warps<true>() * 8u);
      mbar_arrive(bar_addr(ms.jready[0]));
    }
    if (c.rank == 0) {
      int32_t* ls = p.level_sets ? p.level_sets + (int64_t)u * p.sets_stride + sets_off : nullptr;
      if (lev >= 1 && ls) {
#pragma unroll 1
        for (int i = tid; i < kb; i += TN) ls[i] = J[i];
      }
      if (lev == c.lev_end) {
        // mu^0: the children of J^1, or the trimmed level-0 selection.
        const int kk = p.keep[0];
        int32_t* out = p.idx + (int64_t)u * kk;
        int32_t* ls0 = ls ? ls + (lev >= 1 ? kb : 0) : nullptr;
#pragma unroll 1
        for (int t = tid; t < kk; t += TN) {
          const int tok = p.trim ? J[t] : 2 * J[t >> 1] + (t & 1);
          out[t] = tok;
          if (ls0) ls0[t] = tok;
        }
      }
    }
    if (lev >= 1) sets_off += kb;
  }
}

template <int S>
__global__ void __launch_bounds__(NT, 1) wf_gqa_filter_kernel(const __grid_constant__ FusedParams p) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const GqaLayout gl = gqa_layout(S, p.nch, (int)cluster_size(), p.cmax, p.kmax);
  Ctx c;
  c.smem = smem;
  c.ly.q = gl.q;
  c.ly.p = gl.sc;
  c.ly.misc = gl.misc;
  c.ly.buf = gl.buf;
  c.ly.bufw = gl.bufw;
  c.ly.total = gl.total;
  c.ms = reinterpret_cast<Misc*>(smem + gl.misc);
  Misc& ms = *c.ms;
  c.rank = cluster_rank();
  c.cs = cluster_size();
  c.u0 = (int)cluster_id_x();
  c.np = 1;
  c.lev_top = p.L;
  c.lev_end = p.trim ? 0 : 1;
  c.stages = S;
  const int tid = threadIdx.x, warp = tid >> 5;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(bar_addr(ms.full[s]), NPT);
      mbar_init(bar_addr(ms.empty[s]), 1);
    }
    mbar_init(bar_addr(ms.jready[0]), 1);
    mbar_init(bar_addr(ms.xbar[0]), 1);
    mbar_init(bar_addr(ms.kbar[0]), 1);
    for (int r = 0; r < 2; ++r) {
      mbar_init(bar_addr(ms.rdone[r]), 1);
      mbar_init(bar_addr(ms.rfree[r]), NCW);
    }
    mbar_init(bar_addr(ms.qfull), NPT);
    mbar_init(bar_addr(ms.stallbar), 1);
    mbar_init(bar_addr(ms.drainbar), 1);
    ms.wait_limit = p.wait_limit;
    ms.abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (warp > MMA_WARP) {
    cluster_arrive_relaxed();
    gqa_producer_role<S>(c, p);
    cluster_wait();
  } else {
    constexpr int NS = NT - NPT;
    if (tid == 0) {
      mbar_arrive_expect_tx(bar_addr(ms.xbar[0]), c.cs * 32u * (uint32_t)p.nch * 8u);
      mbar_arrive_expect_tx(bar_addr(ms.kbar[0]),
                            4u * (uint32_t)m_total(p, c.lev_top) + c.cs * unit_warps<true>() * 8u);
    }
    if (warp == MMA_WARP) {
      tmem_alloc(smem_u32(&ms.tmem_base), p.tmem_cols);
      tmem_relinquish();
    }
    // The Top-K scratch starts zeroed (histogram, list counter, masks).
    for (int e = tid; e < (int)((sizeof(SelScratch) + 15) / 16); e += NS)
      *reinterpret_cast<uint4*>(smem + gl.sc + 16 * e) = make_uint4(0, 0, 0, 0);
    tc_fence_before();
    named_sync(kSetupSyncId, NS);
    tc_fence_after();
    c.tmem = ms.tmem_base;
    cluster_sync();  // every CTA's barriers are armed before any remote arrival
    if (warp < MMA_WARP) {
      gqa_compute_role(c, p, gl);
    } else {
      if ((tid & 31) == 0) gqa_mma_role<S>(c, p);
      __syncwarp();
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_arrive();
  cluster_wait();
  if (warp == MMA_WARP) {
    if (aborted(ms)) {
      const unsigned long long t0 = globaltimer_ns();
      while (globaltimer_ns() - t0 < 20000ull) {
      }
    }
    tc_fence_after();
    tmem_dealloc(c.tmem, p.tmem_cols);
  }
}
}  // namespace

// ---------------------------------------------------------------------------
// Host side.
// ---------------------------------------------------------------------------
namespace {

// The kernel instance for a stage count and unit width (one-unit plans with
// long candidate lists run the WIDE instance, whose two warpgroups both serve
// the unit).
typedef void (*FusedKernel)(FusedParams);
FusedKernel fused_kernel(int stages, bool wide) {
  if (stages == 4) return wide ? wf_fused_kernel<4, true> : wf_fused_kernel<4, false>;
  return wide ? wf_fused_kernel<3, true> : wf_fused_kernel<3, false>;
}

// The kernel's dynamic shared-memory limit, raised once per device and
// instance to the largest size requested so far instead of on every launch.
cudaError_t ensure_smem_limit(int stages, bool wide, size_t smem) {
  static std::mutex mu;
  static std::map<std::tuple<int, int, bool>, size_t> raised;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  size_t& cur = raised[std::make_tuple(dev, stages, wide)];
  if (cur >= smem) return cudaSuccess;
  e = cudaFuncSetAttribute(fused_kernel(stages, wide), cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) cur = smem;
  return e;
}

// How many clusters of cs CTAs (with `smem` bytes each) can be resident at
// once on the current device; cached per configuration.
int max_active_clusters(int stages, bool wide, int cs, size_t smem) {
  static std::mutex mu;
  static std::map<std::tuple<int, int, bool, int, size_t>, int> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  const auto key = std::make_tuple(dev, stages, wide, cs, smem);
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)cs, 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  cudaError_t e;
  e = ensure_smem_limit(stages, wide, smem);  // only ever raised, so a launch's earlier limit still holds
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&n, fused_kernel(stages, wide), &cfg);
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    n = 0;
  }
  cache.emplace(key, n);
  return n;
}

}  // namespace

FusedPlan plan_fused(const wf_tensor& q, const wf_tensor& kv, int levels, const int32_t* keep, int n_g,
                     const wf_tensor* g, int num_sms) {
  (void)g;
  FusedPlan fp{};
  fp.ok = false;
  if (kv.dtype != WF_BF16 || kv.head_dim != D || q.seq > NQ || levels > 10) return fp;
  const int U = kv.batch * kv.heads;
  const int n = kv.seq;
  const bool trim = keep[0] < 2 * keep[1];
  int cmax = n >> levels, kmax = 0;
  for (int l = 0; l <= levels; ++l) kmax = kmax > keep[l] ? kmax : keep[l];
  for (int l = 1; l <= levels; ++l) cmax = cmax > 2 * keep[l] ? cmax : 2 * keep[l];
  if (cmax > kMaxCand || kmax > kMaxCand) return fp;
  const int total = keep[0] + n_g;
  // TMEM columns of one unit's region at cluster size cs: the widest scale
  // slice, or the attention slice plus the O^T accumulator.
  // TMEM tiles of the widest scale slice at cluster size cs.
  auto scale_tiles = [&](int cs) {
    auto slice_tiles = [&](int m) { return (2 * (((m + 1) / 2 + cs - 1) / cs) + TM - 1) / TM; };
    int tmax = slice_tiles(n >> levels);
    for (int l = levels; l >= 1; --l) {
      const int t = slice_tiles(2 * keep[l]);
      tmax = tmax > t ? tmax : t;
    }
    return tmax;
  };
  auto unit_cols = [&](int cs) {
    int tmax = scale_tiles(cs);
    const int ta = ((total + cs - 1) / cs + TM - 1) / TM + 1;
    tmax = tmax > ta ? tmax : ta;
    return 32 * tmax;
  };
  const size_t kMaxSmem = 227 * 1024;
  // A one-unit plan runs both warpgroups on its unit when the candidate lists
  // are long enough for the halved per-thread work to outweigh the wider
  // barriers (measured: 128K tokens 123.6 -> 116.8 us; 8K tokens, lists of at
  // most 1024, 49.5 -> 51.6 us).
  const bool wide1 = cmax >= 2048;
  // For P units per cluster (1, or 2 so that one unit's copies overlap the
  // other's exchanges and Top-K): the largest cluster (any size up to 8)
  // whose grid fits the SMs in one wave, all clusters resident at once, and
  // whose slices fit TMEM; else the smallest one that fits TMEM.
  struct Choice {
    int P, cs, stages;
    size_t smem;
  };
  auto choose = [&](int P) {
    Choice ch{P, 0, 4, 0};
    const int clusters = (U + P - 1) / P;
    if (smem_layout(4, P, cmax, kmax).total > kMaxSmem) ch.stages = 3;
    ch.smem = smem_layout(ch.stages, P, cmax, kmax).total;
    if (ch.smem > kMaxSmem) return ch;
    for (int c = MAXCS; c >= 1 && ch.cs == 0; --c)
      if (clusters * c <= num_sms && P * unit_cols(c) <= 512 &&
          clusters <= max_active_clusters(ch.stages, P == 1 && wide1, c, ch.smem))
        ch.cs = c;
    for (int c = 1; c <= MAXCS && ch.cs == 0; ++c)
      if (P * unit_cols(c) <= 512) ch.cs = c;
    return ch;
  };
  // Units per SM (P / cs) set each SM's share of the rows: take the smaller,
  // two units per cluster on a tie.
  const Choice c2 = U >= 2 ? choose(2) : Choice{2, 0, 4, 0};
  const Choice c1 = choose(1);
  Choice best = c2;
  if (c2.cs == 0 || (c1.cs > 0 && 1 * c2.cs < 2 * c1.cs)) best = c1;
  if (best.cs == 0) return fp;
  const int P = best.P, cs = best.cs, stages = best.stages;
  const size_t smem = best.smem;
  const int clusters = (U + P - 1) / P;
  int ucols = unit_cols(cs);
  // Room for the scale's exponentials beside its logits (the ranking keys
  // then need no exponentials of their own): the widest scale slice twice.
  const int stiles = scale_tiles(cs);
  int ecol = 0;
  const int ecols = ucols > 64 * stiles ? ucols : 64 * stiles;
  if (P * ecols <= 512) {
    ecol = 32 * stiles;
    ucols = ecols;
  }
  int cols = 32;
  while (cols < P * ucols) cols *= 2;
  fp.ok = true;
  fp.cs = cs;
  fp.P = P;
  fp.wide = P == 1 && wide1;
  fp.stages = stages;
  fp.smem = smem;
  fp.tmem_cols = cols;
  fp.ucols = ucols;
  fp.ecol = ecol;
  fp.cmax = cmax;
  fp.kmax = kmax;
  fp.trim = trim;
  fp.U = U;
  fp.clusters = clusters;
  return fp;
}

cudaError_t launch_fused(const FusedPlan& fp, const void* Q, const wf_tensor& qd, const void* K, const void* V,
                         const wf_tensor& kv, const void* Kg, const void* Vg, const wf_tensor* g,
                         const void* coeffs, int levels, const int32_t* keep, int32_t* idx, int32_t* level_sets,
                         void* O, const wf_tensor& od, int* status, cudaStream_t s, const FusedRange* range) {
  FusedParams p;
  memset(&p, 0, sizeof(p));
  p.Q = static_cast<const bf16*>(Q);
  p.qsb = qd.stride_b; p.qsh = qd.stride_h; p.qss = qd.stride_s;
  p.K = static_cast<const bf16*>(K);
  p.V = static_cast<const bf16*>(V);
  p.ksb = kv.stride_b; p.ksh = kv.stride_h; p.kss = kv.stride_s;
  p.Kg = static_cast<const bf16*>(Kg);
  p.Vg = static_cast<const bf16*>(Vg);
  if (g) { p.gsb = g->stride_b; p.gsh = g->stride_h; p.gss = g->stride_s; }
  p.coeffs = static_cast<const bf16*>(coeffs);
  p.rows_total = (int64_t)kv.seq - ((int64_t)kv.seq >> levels);
  p.O = static_cast<bf16*>(O);
  p.osb = od.stride_b; p.osh = od.stride_h; p.oss = od.stride_s;
  p.idx = idx;
  p.level_sets = level_sets;
  int64_t stride = 0;
  for (int l = 0; l <= levels; ++l) stride += keep[l];
  p.sets_stride = stride;
  p.status = status;
  p.q = qd.seq; p.n = kv.seq; p.ng = g ? g->seq : 0; p.U = fp.U; p.H = kv.heads; p.L = levels;
  p.trim = fp.trim ? 1 : 0;
  p.P = fp.P;
  p.cmax = fp.cmax; p.kmax = fp.kmax;
  p.tmem_cols = (uint32_t)fp.tmem_cols;
  p.ucols = (uint32_t)fp.ucols;
  p.ecol = (uint32_t)fp.ecol;
  const WaitControls wc = wait_controls();
  p.wait_limit = wc.limit;
  p.stall = wc.stall;
  for (int l = 0; l <= levels; ++l) p.keep[l] = keep[l];
  p.scale_log2 = kLog2e / sqrtf((float)D);
  if (range) {
    // A launch below the top scale reads its first scale's rows densely: the
    // producers never wait for the handed-in selection.
    if (range->lev_top < levels && !range->lrows) return cudaErrorInvalidValue;
    p.lev_top = range->lev_top;
    p.lev_bot = range->lev_bot;
    p.final_sel = range->final_sel;
    p.attn = range->attn;
    p.jin = range->jin;
    p.jout = range->jout;
    p.jstride = range->jstride;
    p.lrows = static_cast<const bf16*>(range->lrows);
    p.lrows_unit = range->lrows_unit;
  } else {
    p.lev_top = levels;
    p.lev_bot = fp.trim ? 0 : 1;
    p.final_sel = 1;
    p.attn = 1;
  }

  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(fp.clusters * fp.cs), 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = fp.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = fp.cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = range && range->pdl ? 2 : 1;
  cudaError_t e = ensure_smem_limit(fp.stages, fp.wide, cfg.dynamicSmemBytes);
  if (e != cudaSuccess) return e;
  e = cudaLaunchKernelEx(&cfg, fused_kernel(fp.stages, fp.wide), p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// The grouped filter (wf_gqa_filter_kernel): bf16, d = 128, G >= 2 query
// heads per key head with q <= 32 rows each and G q <= 256, candidate lists
// within the Top-K's 8192.  One unit per cluster; the largest cluster of up
// to 8 CTAs whose grid fits the SMs in one wave with every cluster resident.
GqaPlan plan_gqa(const wf_tensor& q, const wf_tensor& kv, int levels, const int32_t* keep, int num_sms) {
  GqaPlan gp{};
  gp.ok = false;
  if (kv.dtype != WF_BF16 || kv.head_dim != D || q.dtype != WF_BF16 || kv.heads <= 0 || levels > 10) return gp;
  if (q.heads % kv.heads != 0 || q.batch != kv.batch) return gp;
  const int G = q.heads / kv.heads;
  if (G < 2 || q.seq > NQ || G * q.seq > GQ_MAXCH * NQ) return gp;
  const int U = kv.batch * kv.heads;
  int cmax = kv.seq >> levels, kmax = 0;
  for (int l = 0; l <= levels; ++l) kmax = kmax > keep[l] ? kmax : keep[l];
  for (int l = 1; l <= levels; ++l) cmax = cmax > 2 * keep[l] ? cmax : 2 * keep[l];
  if (cmax > kMaxCand || kmax > kMaxCand) return gp;
  const int nch = (G * q.seq + NQ - 1) / NQ;
  constexpr int kStages = 3;
  const size_t kMaxSmem = 227 * 1024;
  int cs = 0;
  size_t smem = 0;
  for (int c = MAXCS; c >= 1 && cs == 0; --c) {
    smem = gqa_layout(kStages, nch, c, cmax, kmax).total;
    if (smem > kMaxSmem || U * c > num_sms) continue;
    static std::mutex mu;
    static std::map<std::tuple<int, int, size_t>, int> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return gp;
    int n = 0;
    {
      std::lock_guard<std::mutex> lock(mu);
      const auto key = std::make_tuple(dev, c, smem);
      auto it = cache.find(key);
      if (it != cache.end()) {
        n = it->second;
      } else {
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)c, 1, 1);
        cfg.blockDim = dim3(NT, 1, 1);
        cfg.dynamicSmemBytes = smem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = c;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        cudaError_t e = cudaFuncSetAttribute(wf_gqa_filter_kernel<kStages>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kMaxSmem);
        if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&n, wf_gqa_filter_kernel<kStages>, &cfg);
        if (e != cudaSuccess) {
          (void)cudaGetLastError();
          n = 0;
        }
        cache.emplace(key, n);
      }
    }
    if (U <= n) cs = c;
  }
  if (cs == 0) {  // more units than one wave holds: single-CTA clusters in several waves
    cs = 1;
    smem = gqa_layout(kStages, nch, 1, cmax, kmax).total;
    if (smem > kMaxSmem) return gp;
  }
  int cols = 32;
  while (cols < 2 * NQ * nch) cols *= 2;
  gp.ok = true;
  gp.cs = cs;
  gp.stages = kStages;
  gp.smem = smem;
  gp.tmem_cols = cols;
  gp.nch = nch;
  gp.G = G;
  gp.cmax = cmax;
  gp.kmax = kmax;
  gp.trim = keep[0] < 2 * keep[1];
  gp.U = U;
  return gp;
}

cudaError_t launch_gqa_filter(const GqaPlan& gp, const void* Q, const wf_tensor& qd, const void* K,
                              const wf_tensor& kv, const void* coeffs, int levels, const int32_t* keep, int32_t* idx,
                              int32_t* level_sets, int* status, cudaStream_t s) {
  FusedParams p;
  memset(&p, 0, sizeof(p));
  p.Q = static_cast<const bf16*>(Q);
  p.qsb = qd.stride_b; p.qsh = qd.stride_h; p.qss = qd.stride_s;
  p.K = static_cast<const bf16*>(K);
  p.ksb = kv.stride_b; p.ksh = kv.stride_h; p.kss = kv.stride_s;
  p.coeffs = static_cast<const bf16*>(coeffs);
  p.rows_total = (int64_t)kv.seq - ((int64_t)kv.seq >> levels);
  p.idx = idx;
  p.level_sets = level_sets;
  int64_t stride = 0;
  for (int l = 0; l <= levels; ++l) stride += keep[l];
  p.sets_stride = stride;
  p.status = status;
  p.q = qd.seq; p.n = kv.seq; p.U = gp.U; p.H = kv.heads; p.L = levels;
  p.trim = gp.trim ? 1 : 0;
  p.P = 1;
  p.cmax = gp.cmax; p.kmax = gp.kmax;
  p.tmem_cols = (uint32_t)gp.tmem_cols;
  const WaitControls wc = wait_controls();
  p.wait_limit = wc.limit;
  p.stall = wc.stall;
  for (int l = 0; l <= levels; ++l) p.keep[l] = keep[l];
  p.scale_log2 = kLog2e / sqrtf((float)D);
  p.lev_top = levels;
  p.lev_bot = gp.trim ? 0 : 1;
  p.final_sel = 1;
  p.G = gp.G;
  p.nch = gp.nch;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)(gp.U * gp.cs), 1, 1);
  cfg.blockDim = dim3(NT, 1, 1);
  cfg.dynamicSmemBytes = gp.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = gp.cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaFuncSetAttribute(wf_gqa_filter_kernel<3>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)gp.smem);
  if (e != cudaSuccess) return e;
  e = cudaLaunchKernelEx(&cfg, wf_gqa_filter_kernel<3>, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_literal_fused(const FusedPlan& fp, const FilterPlan& fl, const void* Q, const wf_tensor& qd,
                                 const void* top, const void* K, const void* V, const wf_tensor& kv, const void* Kg,
                                 const void* Vg, const wf_tensor* g, int wavelet, int32_t* idx, int32_t* level_sets,
                                 void* O, const wf_tensor* od, void* ws, int* status, cudaStream_t s) {
  char* base = static_cast<char*>(ws);
  int32_t* cur = reinterpret_cast<int32_t*>(base + fl.off_cand_a);  // candidates of the scale being filtered
  int32_t* nxt = reinterpret_cast<int32_t*>(base + fl.off_cand_b);
  void* arows = base + align_up(fl.total, 256);
  const int L = fl.L;
  int m = fl.n >> L;
  cudaError_t e;
  for (int l = L; l >= 1; --l) {
    // Scale l's rows: the whole prompt's scale-L rows at the top, else the
    // transform of the candidates' gathered blocks, in candidate order.
    if (l < L && (e = launch_wavelet_approx(K, kv, cur, fl.cmax, m, l, wavelet, arows, (int64_t)fl.cmax * D, s,
                                            true)) != cudaSuccess)
      return e;
    FusedRange r{};
    r.pdl = l < L;  // every launch after the first follows one of this pipeline's own
    r.lev_top = l;
    r.lev_bot = (l == 1 && fl.trim) ? 0 : l;
    r.final_sel = l == 1;
    r.attn = l == 1 && O != nullptr;
    r.jin = cur;
    r.jout = nxt;
    r.jstride = fl.cmax;
    r.lrows = l == L ? top : arows;
    r.lrows_unit = l == L ? (int64_t)m * D : (int64_t)fl.cmax * D;
    if ((e = launch_fused(fp, Q, qd, K, V, kv, Kg, Vg, g, nullptr, L, fl.keep, idx, level_sets, O, od ? *od : qd,
                          status, s, &r)) != cudaSuccess)
      return e;
    m = 2 * fl.keep[l];
    int32_t* t = cur;
    cur = nxt;
    nxt = t;
  }
  return cudaSuccess;
}

}  // namespace wf
