// plan.h — host-side planning of the strided dense pass (f(~Q,K,V) of
// Alg. 1 over the sampled rows of Eq. 4): the GQA head packing of its tiles and
// the split of each M-tile's causal key range into units.  Shared by the
// library (api.cu) and the host geometry check, so the check runs the planner
// the library runs.
//
// An M-tile packs Hp query heads of one KV head x R samples into the 128 TMEM
// lanes; its causal key range is L(t) key tiles.  Units are claimed by the
// CTAs from an atomic counter in unit order.  Two orders:
//
//   SPLIT_LONGEST_FIRST  M-tiles in descending t, each cut into `chunk`-tile
//     units: unit lengths shrink as the schedule runs, which balances the
//     CTAs, but every KV head's key range is streamed at once.
//   SPLIT_LEVELS  the key range is cut at multiples of `chunk` into levels;
//     units run head group by head group, inside a group level by level from
//     the top, inside a level M-tiles in descending t.  The units that run at
//     the same time read the same few key tiles of one KV head, so K and V are
//     read from L2 by all but the first of them; every unit is at most `chunk`
//     tiles, which bounds the tail of the schedule.  Each unit of a split
//     M-tile writes a partial (unnormalised O, row max, row sum) that the last
//     unit of the M-tile to finish merges.
//
// The level order is used unless its partials would not fit the budget even
// with two levels (very long problems with every row dense, gamma = 1 at 1M
// tokens), where the longest-first order is balanced without splitting.
#pragma once
#include <stddef.h>

#include <algorithm>

#include "tiles.cuh"

namespace da {

// The planner's choices (SplitPolicy): units of about kUnitTiles key tiles
// (long enough that a unit's fixed costs, its Q load and its partial, stay
// small), fewer when the problem is too small to give every SM two of them;
// at most kMaxLevelsUsed levels (the chunk grows with the sequence); and a
// partial buffer of at most max(kLevelPartialBytes, 3 x the dense rows' bf16
// output), doubling the chunk until it fits.
constexpr int kMaxLevelsUsed = 16;
constexpr long long kUnitTiles = 128;
constexpr long long kMinChunk = 8;
constexpr size_t kLevelPartialBytes = size_t(4) << 30;

// Hp query heads of one KV group share a dense tile when G is a power of two
// up to 16 (R = 128 / Hp samples each); otherwise one head per tile.
inline void packing(int G, int* Hp, int* R) {
  int hp = 1;
  if (G >= 2 && G <= 16 && (G & (G - 1)) == 0) hp = G;
  *Hp = hp;
  *R = BM / hp;
}

inline size_t partial_slot_bytes(int d) { return (size_t)BM * (d + 2) * sizeof(float); }

// First M-tile whose causal key range reaches past key tile `tiles` - 1
// (L(t) > tiles), by bisection over the non-decreasing L(t).
inline long long first_mtile_longer_than(const Params& p, long long tiles) {
  long long lo = 0, hi = p.mtiles;  // answer in [lo, hi]
  while (lo < hi) {
    const long long mid = (lo + hi) / 2;
    if (strided_dense_len(p, mid) > tiles) hi = mid; else lo = mid + 1;
  }
  return lo;
}

// Level order with n_lev levels of `chunk` tiles (n_lev = ceil(L_max / chunk)):
// units per head group, the cumulative counts per processing step, and the
// units of split M-tiles per group.
inline void plan_levels(Params& p, long long chunk) {
  const long long L_max = strided_dense_len(p, p.mtiles - 1);
  p.order = SPLIT_LEVELS;
  p.chunk = chunk;
  p.n_lev = (int)cdiv(L_max, chunk);
  long long cum = 0;
  for (int l = 0; l < p.n_lev; ++l) {  // step l processes level c = n_lev - 1 - l
    const int c = p.n_lev - 1 - l;
    p.lev_cum[l] = cum;
    cum += p.mtiles - first_mtile_longer_than(p, (long long)c * chunk);
  }
  for (int l = p.n_lev; l <= kMaxLevels; ++l) p.lev_cum[l] = cum;
  p.units_per_group = cum;
  // M-tiles with one level (L(t) <= chunk) are the last units of level 0
  p.split_per_group = p.n_lev > 1 ? cum - first_mtile_longer_than(p, chunk) : 0;
  const long long groups = (long long)p.B * p.groups_per_b;
  p.n_units = groups * cum;
  p.n_multi = groups * p.split_per_group;
}

// Longest-first order: the chunk is chosen so that about two units per SM
// exist; the longest M-tiles split, short ones stay whole.
inline void plan_longest_first(Params& p, int sms, long long min_chunk = kMinChunk) {
  long long total_tiles = 0;
  for (long long t = 0; t < p.mtiles; ++t) total_tiles += strided_dense_len(p, t);
  total_tiles *= (long long)p.B * p.groups_per_b;
  p.order = SPLIT_LONGEST_FIRST;
  p.n_lev = 0;
  p.chunk = std::max<long long>(min_chunk, cdiv(total_tiles, 2LL * std::max(sms, 1)));
  long long units = 0, multi = 0;
  for (long long t = 0; t < p.mtiles; ++t) {
    const long long nc = cdiv(strided_dense_len(p, t), p.chunk);
    units += nc;
    if (nc > 1) multi += nc;
  }
  p.n_units = units * p.B * p.groups_per_b;
  p.n_multi = multi * p.B * p.groups_per_b;
}

struct SplitPolicy {
  int max_levels;
  long long unit_tiles;
  long long min_chunk;
  size_t budget;  // bytes of partials the level order may use
};

inline SplitPolicy library_policy(const Params& p, int d) {
  const size_t out_bytes = (size_t)p.B * p.Hq * p.n_s * d * 2;
  return SplitPolicy{kMaxLevelsUsed, kUnitTiles, kMinChunk, std::max(kLevelPartialBytes, 3 * out_bytes)};
}

// Split-K plan of a strided-dense pass over p.n_s samples (p.R, p.groups_per_b,
// p.row0 and p.gamma set).  `d` sizes the partials.
inline void plan_split_k(Params& p, int sms, int d, const SplitPolicy& pol) {
  p.mtiles = cdiv(p.n_s, p.R);
  const long long L_max = strided_dense_len(p, p.mtiles - 1);
  long long total_tiles = 0;
  for (long long t = 0; t < p.mtiles; ++t) total_tiles += strided_dense_len(p, t);
  total_tiles *= (long long)p.B * p.groups_per_b;
  const long long balanced = cdiv(total_tiles, 2LL * std::max(sms, 1));
  long long chunk = std::max(std::max(pol.min_chunk, std::min(pol.unit_tiles, balanced)),
                             cdiv(L_max, std::max(1, std::min(pol.max_levels, kMaxLevels))));
  for (; cdiv(L_max, chunk) >= 2; chunk *= 2) {  // one level: nothing to gain over longest-first
    plan_levels(p, chunk);
    if ((size_t)p.n_multi * partial_slot_bytes(d) <= pol.budget) return;
  }
  plan_longest_first(p, sms, pol.min_chunk);
}

inline void plan_split_k(Params& p, int sms, int d) {
  p.mtiles = cdiv(p.n_s, p.R);
  plan_split_k(p, sms, d, library_policy(p, d));
}

// Bytes of the control block zeroed before a strided-dense launch: 4 item
// counters, then one merge ticket per split unit.
inline size_t ctrl_bytes(const Params& p) { return 4 * sizeof(unsigned long long) + (size_t)p.n_multi * sizeof(int); }

}  // namespace da
