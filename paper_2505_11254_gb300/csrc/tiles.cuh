// tiles.cuh — work decomposition, key-tile lists and visibility predicates of
// the Delta Attention prefill kernels.  Used by the attention kernel and by the
// debug kernels, so the tests check the same code the kernels run.
//
// Definitions (arXiv 2505.11254):
//   * causal visibility (Eq. 1): key j is visible to query row i iff j <= i;
//   * StreamingLLM sparse set (Sec. 2-3, f*): the first n_sink keys and the
//     `window` most recent keys ending at i (diagonal included);
//   * sampled rows (Eq. 4): i = k * gamma, k = 0, 1, ...; row i is corrected
//     with the Delta of sample floor(i / gamma) (Eq. 6, Alg. 1 repeat).
#pragma once
#include <stdint.h>

namespace da {

constexpr int BM = 128;  // query rows per tile = TMEM lanes
constexpr int BN = 128;  // keys per tile

// Which rows a tile holds and which keys it visits.
enum Mode : int {
  MODE_SPARSE = 0,          // contiguous rows of one head, sink + window keys
  MODE_STRIDED_DENSE = 1,   // sampled rows (GQA-packed), all causal keys, split-K
  MODE_STRIDED_SPARSE = 2,  // sampled rows (GQA-packed), sink + window keys
};

// What the epilogue writes.
enum Epi : int {
  EPI_BF16 = 0,          // sparse rows -> bf16 S_i (+ fp32 S at sampled rows if requested)
  EPI_FUSED_INTILE = 1,  // sparse rows -> bf16(S_i + D_k - S_{k gamma}), samples inside the tile
  EPI_FUSED_DELTA = 2,   // sparse rows -> bf16(S_i + Delta_k), Delta precomputed
  EPI_DENSE_F32 = 3,     // sampled rows -> fp32 dense rows D_k
  EPI_DENSE_BF16 = 4,    // sampled rows (gamma = 1: every row) -> bf16 dense rows
  EPI_DELTA_BUILD = 5,   // sampled rows -> fp32 Delta_k = D_k - S_{k gamma}
  EPI_FUSED_SMOOTH = 6,  // sparse rows -> bf16(S_i + sum_j coef[r][j] basis_k[j]), smoothed Delta
};

// Delta smoothing (appendix "Interpolation", Alg. 2): the correction of row
// i = k gamma + r is coef[r][0] basis_k[0] + coef[r][1] basis_k[1].
enum Smooth : int {
  SMOOTH_NONE = 0,
  SMOOTH_LINEAR = 1,  // basis (Delta_k, Delta_{k+1}), coef (1 - r/gamma, r/gamma)
  SMOOTH_EMA = 2,     // basis (e_{k gamma - 1}, Delta_k), coef ((1-beta)^(r+1), 1 - (1-beta)^(r+1))
  SMOOTH_ABG = 3,     // basis (filter output o_k), coef (1)
};
constexpr int kSmoothJ = 2;  // basis vectors per sample (the filter uses the first)

// Order of the strided dense pass's split-K units (plan.h).
enum SplitOrder : int {
  SPLIT_LONGEST_FIRST = 0,  // M-tiles by descending t, each cut into chunks
  SPLIT_LEVELS = 1,         // head group by head group, key-range levels from the top, t descending
};
constexpr int kMaxLevels = 32;

struct Params {
  int B, Hq, Hkv, G;
  long long N;
  int n_sink;
  long long window;
  int gamma;
  long long n_s;           // sampled rows the call computes (ceil((N - q_row0) / gamma); the tail's rows)
  long long row0;          // row of sample 0: q_row0, or N - t for the dense tail block of t rows
  // Rows computed: [q_row0, N).  Q holds exactly these rows (row i at index
  // i - q_row0); K and V hold rows from 0.  A whole-sequence call has
  // q_row0 = 0; a row-range call (one rank's share of a sequence) has q_row0
  // a multiple of BM and of gamma, and the host passes the output and the
  // per-sample buffers the sink + window pass reads by absolute row or sample
  // as base pointers moved back by q_row0 rows (q_row0 / gamma samples).
  long long q_row0;
  long long o_rows;        // rows per (b, head) of the output buffer (its row stride)
  float scale_log2;        // log2(e) / sqrt(d)
  // sampled-row packing: Hp heads x R samples per tile (Hp * R == BM)
  int Hp, R;
  int groups_per_b;        // Hq / Hp
  long long mtiles;        // ceil(n_s / R) tiles per head group
  long long qtiles;        // ceil(N / BM) tiles of contiguous rows per head
  // split-K over keys for MODE_STRIDED_DENSE
  int order;               // SplitOrder
  int n_lev;               // SPLIT_LEVELS: key-range levels of `chunk` tiles
  long long chunk;         // key tiles per unit
  long long n_units;       // units
  long long n_multi;       // units of split M-tiles (partial slots)
  long long units_per_group;   // SPLIT_LEVELS: units of one (b, head group)
  long long split_per_group;   // SPLIT_LEVELS: of which belong to split M-tiles (the group's first units)
  long long lev_cum[kMaxLevels + 1];  // SPLIT_LEVELS: units of a group before step l (level n_lev - 1 - l)
  long long n_items;       // work items of the launched kernel
  // buffers
  void* out_bf16;          // [B,Hq,N,d] bf16
  float* s_sampled;        // [B,Hq,n_s,d] fp32, nullable
  const float* d_in;       // [B,Hq,n_s,d] fp32 dense sampled rows (fused epilogues)
  float* d_out;            // [B,Hq,n_s,d] fp32
  const float* delta_in;   // [B,Hq,n_s,d] fp32
  float* delta_out;        // [B,Hq,n_s,d] fp32
  const float* smooth_basis;  // [B,Hq,n_s,kSmoothJ,d] fp32 (EPI_FUSED_SMOOTH)
  const float* smooth_coef;   // [gamma][kSmoothJ] fp32 (EPI_FUSED_SMOOTH)
  const float* rope;          // RoPE (cos, sin) table [N][d/2][2] fp32: Q rotated on its way to TMEM, or null
  float* partials;         // n_multi slots of BM*(d+2) fp32
  int* tickets;            // n_multi
  unsigned long long* counter;  // dynamic item counter (zeroed before the launch)
  int* err;                // device status word
};

struct Work {
  int b, h0, g;
  long long r0;        // MODE_SPARSE: first row; strided: first sample k0
  long long r_last;    // last valid row / last valid sample
  int n_sink_tiles;    // key tiles [0, n_sink_tiles) visited before the band
  long long kt_lo;     // band tiles [kt_lo, kt_hi]
  long long kt_hi;
  int T;               // number of key tiles visited
  long long unit;      // split-K: this unit's partial slot (when its M-tile is split)
  long long u0;        // split-K: merge ticket of its M-tile
  long long gi, t;     // split-K: (b, head group) index and M-tile index
  int chunk_idx, n_chunks;
};

__host__ __device__ __forceinline__ long long cdiv(long long a, long long b) { return (a + b - 1) / b; }
__host__ __device__ __forceinline__ long long lmin(long long a, long long b) { return a < b ? a : b; }
__host__ __device__ __forceinline__ long long lmax(long long a, long long b) { return a > b ? a : b; }

// --------------------------------------------------------------- predicates
__host__ __device__ __forceinline__ bool visible_causal(long long i, long long j) { return j <= i; }
__host__ __device__ __forceinline__ bool visible_sparse(long long i, long long j, int n_sink, long long window) {
  return j <= i && (j < n_sink || j > i - window);
}
__host__ __device__ __forceinline__ long long sample_of_row(long long i, int gamma) { return (i / gamma) * gamma; }
__host__ __device__ __forceinline__ bool is_sampled_row(long long i, int gamma) { return i % gamma == 0; }

// Visibility word of the key offsets c0 .. c0 + 31 of a tile: bit c - c0 is
// set when lo <= c <= hi (window and causality; hi < lo is an empty range) or
// c < se (sinks).  The kernels mask a tile's scores by one bit test per key.
__host__ __device__ __forceinline__ uint32_t visible_bits(int lo, int hi, int se, int c0) {
  const int a = lo - c0 > 0 ? lo - c0 : 0;
  const int b = hi - c0 < 31 ? hi - c0 : 31;
  const uint32_t upto_b = b < 0 ? 0u : (b >= 31 ? 0xffffffffu : ((2u << b) - 1u));
  const uint32_t below_a = a >= 32 ? 0xffffffffu : ((1u << a) - 1u);
  const uint32_t range = b >= a ? (upto_b & ~below_a) : 0u;
  const int ns = se - c0 < 0 ? 0 : (se - c0 > 32 ? 32 : se - c0);
  const uint32_t sink = ns >= 32 ? 0xffffffffu : ((1u << ns) - 1u);
  return range | sink;
}

// Key tiles covering the sink keys visible to rows up to `last_row`, limited
// to tiles before the band's first tile.
__host__ __device__ __forceinline__ int sink_tiles_before(int n_sink, long long last_row, long long kt_lo) {
  long long s = lmin((long long)n_sink, last_row + 1);
  if (s <= 0) return 0;
  return (int)lmin(kt_lo, cdiv(s, BN));
}

// Number of key tiles an M-tile of sampled rows needs under causal masking.
__host__ __device__ __forceinline__ long long strided_dense_len(const Params& p, long long t) {
  long long k_last = lmin(t * p.R + p.R - 1, p.n_s - 1);
  return (p.row0 + k_last * p.gamma) / BN + 1;
}

// lev_cum[l] for a run-time l, read with constant indices only (the
// parameter block is never indexed dynamically).
__host__ __device__ __forceinline__ long long lev_cum_at(const Params& p, int l) {
  long long v = 0;
#pragma unroll
  for (int i = 0; i <= kMaxLevels; ++i)
    if (i == l) v = p.lev_cum[i];
  return v;
}

// Partial slot of chunk c of the unit's M-tile (its units hold the chunks
// 0 .. n_chunks - 1).
__host__ __device__ __forceinline__ long long partial_slot(const Params& p, const Work& w, int c) {
  if (p.order == SPLIT_LEVELS)
    return w.gi * p.split_per_group + lev_cum_at(p, p.n_lev - 1 - c) + (p.mtiles - 1 - w.t);
  return w.u0 + c;
}

// Split-K units, in the order of p.order (plan.h):
//   SPLIT_LONGEST_FIRST: M-tile index t descending, then (b, head group), then
//     chunk.  Units of M-tiles with more than one chunk come first because the
//     chunk count never decreases with t; a unit's partial slot is its index,
//     its M-tile's ticket the index of its first chunk.
//   SPLIT_LEVELS: (b, head group) outermost; inside a group, level c from
//     n_lev - 1 down to 0 (key tiles [c chunk, (c+1) chunk)), inside a level
//     the M-tiles long enough to reach it by descending t.  The units of
//     split M-tiles are the first split_per_group of each group, which gives
//     their partial slots; the ticket is the slot of the level-0 unit.
__host__ __device__ inline Work decode_strided_dense(const Params& p, long long unit) {
  Work w;
  long long t, nc, mt;
  int c;
  if (p.order == SPLIT_LEVELS) {
    const long long gi = unit / p.units_per_group;
    const long long ul = unit - gi * p.units_per_group;
    int l = 0;
    long long base = 0;
#pragma unroll
    for (int i = 1; i < kMaxLevels; ++i)
      if (i < p.n_lev && p.lev_cum[i] <= ul) {
        l = i;
        base = p.lev_cum[i];
      }
    c = p.n_lev - 1 - l;
    t = p.mtiles - 1 - (ul - base);
    nc = cdiv(strided_dense_len(p, t), p.chunk);
    mt = gi;
    w.gi = gi;
    w.t = t;
    w.unit = gi * p.split_per_group + ul;
    w.u0 = gi * p.split_per_group + lev_cum_at(p, p.n_lev - 1) + (p.mtiles - 1 - t);
  } else {
    long long per_t = (long long)p.B * p.groups_per_b;
    long long cum = 0;
    t = p.mtiles - 1;
    nc = 1;
    for (; t >= 0; --t) {
      nc = cdiv(strided_dense_len(p, t), p.chunk);
      if (unit < cum + nc * per_t) break;
      cum += nc * per_t;
    }
    if (t < 0) t = 0;  // unreachable for unit < n_units
    long long rem = unit - cum;
    mt = rem / nc;
    c = (int)(rem % nc);
    w.gi = mt;
    w.t = t;
    w.unit = unit;
    w.u0 = unit - c;
  }
  w.b = (int)(mt / p.groups_per_b);
  int hg = (int)(mt % p.groups_per_b);
  w.h0 = hg * p.Hp;
  w.g = w.h0 / p.G;
  w.r0 = t * p.R;
  w.r_last = lmin(w.r0 + p.R - 1, p.n_s - 1);
  long long L = strided_dense_len(p, t);
  w.n_sink_tiles = 0;
  w.kt_lo = (long long)c * p.chunk;
  w.kt_hi = lmin(L, (long long)(c + 1) * p.chunk) - 1;
  w.T = (int)(w.kt_hi - w.kt_lo + 1);
  w.chunk_idx = c;
  w.n_chunks = (int)nc;
  return w;
}

// Contiguous rows: CTA order is (kv-head group member fastest, q-tile, kv-head,
// batch) so the G query heads that share K/V run side by side.
__host__ __device__ inline Work decode_sparse(const Params& p, long long lin, long long row_off) {
  Work w;
  int hl;
  long long qt;
  if (lin >= 0 && lin <= 0xffffffffLL && p.qtiles <= 0xffffffffLL) {
    // 32-bit divisions when the values fit, with the same quotients as the
    // 64-bit path below (a 64-bit division by a runtime value is a long
    // software sequence on the item-start path of every role).
    uint32_t l = (uint32_t)lin;
    hl = (int)(l % (uint32_t)p.G);
    l /= (uint32_t)p.G;
    qt = l % (uint32_t)p.qtiles;
    l /= (uint32_t)p.qtiles;
    w.g = (int)(l % (uint32_t)p.Hkv);
    w.b = (int)(l / (uint32_t)p.Hkv);
  } else {
    hl = (int)(lin % p.G);
    lin /= p.G;
    qt = lin % p.qtiles;
    lin /= p.qtiles;
    w.g = (int)(lin % p.Hkv);
    w.b = (int)(lin / p.Hkv);
  }
  w.h0 = w.g * p.G + hl;
  w.r0 = row_off + qt * BM;
  w.r_last = lmin(w.r0 + BM, p.N) - 1;
  long long band_lo = lmax(0, w.r0 - p.window + 1);
  w.kt_lo = band_lo / BN;
  w.kt_hi = w.r_last / BN;
  w.n_sink_tiles = sink_tiles_before(p.n_sink, w.r_last, w.kt_lo);
  w.T = w.n_sink_tiles + (int)(w.kt_hi - w.kt_lo + 1);
  w.unit = w.u0 = w.gi = w.t = 0;
  w.chunk_idx = 0;
  w.n_chunks = 1;
  return w;
}

// Sampled rows with the sparse key set (used when gamma does not divide BM).
__host__ __device__ inline Work decode_strided_sparse(const Params& p, long long lin) {
  Work w;
  int hg = (int)(lin % p.groups_per_b);
  lin /= p.groups_per_b;
  long long t = lin % p.mtiles;
  w.b = (int)(lin / p.mtiles);
  w.h0 = hg * p.Hp;
  w.g = w.h0 / p.G;
  w.r0 = t * p.R;
  w.r_last = lmin(w.r0 + p.R - 1, p.n_s - 1);
  long long row_first = p.row0 + w.r0 * p.gamma, row_last = p.row0 + w.r_last * p.gamma;
  w.kt_lo = lmax(0, row_first - p.window + 1) / BN;
  w.kt_hi = row_last / BN;
  w.n_sink_tiles = sink_tiles_before(p.n_sink, row_last, w.kt_lo);
  w.T = w.n_sink_tiles + (int)(w.kt_hi - w.kt_lo + 1);
  w.unit = w.u0 = w.gi = w.t = 0;
  w.chunk_idx = 0;
  w.n_chunks = 1;
  return w;
}

// ROWS: a row-range call (rows from p.q_row0); whole-sequence kernels are
// compiled with ROWS = false and start at row 0.
template <int MODE, bool ROWS = false>
__host__ __device__ __forceinline__ Work decode_work(const Params& p, long long lin) {
  if (MODE == MODE_SPARSE) return decode_sparse(p, lin, ROWS ? p.q_row0 : 0);
  if (MODE == MODE_STRIDED_DENSE) return decode_strided_dense(p, lin);
  return decode_strided_sparse(p, lin);
}

__host__ __device__ __forceinline__ long long tile_index(const Work& w, int j) {
  return j < w.n_sink_tiles ? (long long)j : w.kt_lo + (j - w.n_sink_tiles);
}

// True when some (row, key) pair of the tile is not visible, so the kernel
// must apply the predicate element by element.
template <int MODE>
__host__ __device__ __forceinline__ bool tile_needs_mask(const Params& p, const Work& w, int j) {
  if (j < w.n_sink_tiles) return true;
  long long kt = tile_index(w, j);
  long long k_first = kt * BN, k_end = k_first + BN - 1;
  if (MODE == MODE_SPARSE) {
    return !(k_end <= w.r0 && k_first > w.r_last - p.window);
  } else if (MODE == MODE_STRIDED_DENSE) {
    return !(k_end <= p.row0 + w.r0 * p.gamma);
  } else {
    return !(k_end <= p.row0 + w.r0 * p.gamma && k_first > p.row0 + w.r_last * p.gamma - p.window);
  }
}

// Floor division (the truncating / of C++ rounds negative quotients up).
__host__ __device__ __forceinline__ long long floor_div(long long a, long long b) {
  return a >= 0 ? a / b : -((-a + b - 1) / b);
}

// The item's tiles j0 <= j < j1 are exactly the ones tile_needs_mask() rejects:
// band tiles whose every key is visible to every row of the item (causal bound
// kt*BN + BN-1 <= first row, window bound kt*BN > last row - window).  Sink
// tiles are never in the range.  Evaluated once per item, so the per-tile test
// is two integer compares.
template <int MODE>
__host__ __device__ __forceinline__ void unmasked_tiles(const Params& p, const Work& w, int& j0, int& j1) {
  const long long rf = (MODE == MODE_SPARSE) ? w.r0 : p.row0 + w.r0 * p.gamma;
  const long long rl = (MODE == MODE_SPARSE) ? w.r_last : p.row0 + w.r_last * p.gamma;
  const long long k_causal = floor_div(rf - (BN - 1), BN);  // last tile all rows see causally
  const long long k_window = (MODE == MODE_STRIDED_DENSE) ? w.kt_lo : floor_div(rl - p.window, BN) + 1;
  const long long lo = lmax(w.kt_lo, k_window), hi = lmin(w.kt_hi, k_causal);
  j0 = w.n_sink_tiles + (int)(lo - w.kt_lo);
  j1 = hi >= lo ? w.n_sink_tiles + (int)(hi - w.kt_lo) + 1 : j0;
}

// Query row and head of TMEM lane t.  Returns false for padding lanes.
template <int MODE>
__host__ __device__ __forceinline__ bool lane_row(const Params& p, const Work& w, int t, long long& row,
                                                  long long& sample, int& head) {
  if (MODE == MODE_SPARSE) {
    row = w.r0 + t;
    sample = row / p.gamma;
    head = w.h0;
    return row < p.N;
  }
  head = w.h0 + t / p.R;
  sample = w.r0 + t % p.R;
  row = p.row0 + sample * p.gamma;
  return sample < p.n_s;
}

}  // namespace da
