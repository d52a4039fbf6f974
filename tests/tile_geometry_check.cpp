// Host-side check of the tile geometry in tiles.cuh (compiled as plain C++ by
// tests/test_tile_geometry.py): the visibility words the kernels mask scores
// with match the key sets bit by bit; for every work item of many shapes and all
// three modes, unmasked_tiles() must select exactly the tiles for which
// tile_needs_mask() is false, and tile_needs_mask() must be true wherever a
// (row, key) pair of the tile is not visible (checked pair by pair against
// the definition of the key sets), and the dense pass's split-K units, as the
// library's planner (plan.h) lays them out, cover every M-tile's causal key
// range exactly once with the partial slots and tickets the merge assumes.  For every head packing of the dense tiles (GQA 1, 2,
// 3, 4 and 16), each lane's query head reads its own KV head (floor(h / G))
// and every (batch, head, row or sample) sits in exactly one lane.  For the
// two-CTA sink + window kernel, the items the two CTAs of a cluster take
// together are two heads of one row tile with the same key tiles.
#define __host__
#define __device__
#define __forceinline__ inline
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <initializer_list>
#include <vector>
#include "plan.h"
#include "tiles.cuh"

using namespace da;

static bool visible(const Params& p, int mode, long long row, long long key) {
  if (key > row) return false;
  if (mode == MODE_STRIDED_DENSE) return true;
  return key < p.n_sink || key > row - p.window;
}

template <int MODE>
static int check(const Params& p, long long items) {
  int bad = 0;
  // every (b, query head, row or sample) is held by exactly one lane of one item
  const long long per_head = MODE == MODE_SPARSE ? p.N : p.n_s;
  std::vector<unsigned char> held(MODE == MODE_STRIDED_DENSE ? 0 : (size_t)p.B * p.Hq * per_head, 0);
  for (long long it = 0; it < items; ++it) {
    Work w = p.q_row0 > 0 ? decode_work<MODE, true>(p, it) : decode_work<MODE>(p, it);
    int j0, j1;
    unmasked_tiles<MODE>(p, w, j0, j1);
    for (int t = 0; t < BM; ++t) {  // GQA: every lane's query head reads the item's KV head
      long long row, sample;
      int head;
      if (!lane_row<MODE>(p, w, t, row, sample, head)) continue;
      const bool head_ok = head >= 0 && head < p.Hq && head / p.G == w.g && w.b >= 0 && w.b < p.B;
      if (!head_ok) {
        if (bad < 5) std::printf("mode %d item %lld lane %d: head %d, kv head %d, G %d\n", MODE, it, t, head, w.g, p.G);
        ++bad;
        continue;
      }
      if (MODE != MODE_STRIDED_DENSE) {
        const long long r = MODE == MODE_SPARSE ? row : sample;
        unsigned char& h = held[((size_t)w.b * p.Hq + head) * per_head + r];
        if (h) {
          if (bad < 5) std::printf("mode %d: (b %d, head %d, %lld) held twice\n", MODE, w.b, head, r);
          ++bad;
        }
        h = 1;
      }
    }
    {  // the visited tiles are the sink tiles and the band [kt_lo, kt_hi], each once
      std::vector<long long> seen;
      for (int j = 0; j < w.T; ++j) seen.push_back(tile_index(w, j));
      std::vector<long long> want;
      for (long long kt = 0; kt < w.n_sink_tiles; ++kt) want.push_back(kt);
      for (long long kt = w.kt_lo; kt <= w.kt_hi; ++kt) want.push_back(kt);
      std::sort(seen.begin(), seen.end());
      if (seen != want || w.n_sink_tiles > w.kt_lo) {
        if (bad < 5) std::printf("mode %d item %lld: visited tiles are not the sink tiles and the band\n", MODE, it);
        ++bad;
      }
    }
    for (int j = 0; j < w.T; ++j) {
      const bool need = tile_needs_mask<MODE>(p, w, j);
      const bool in_range = j >= j0 && j < j1;
      if (need == in_range) {
        if (bad < 5) std::printf("mode %d item %lld tile %d: needs_mask %d, in unmasked range [%d,%d)\n", MODE, it, j,
                                 need, j0, j1);
        ++bad;
      }
      if (!need) {  // the pairs at the tile's edges must be visible (the key sets are ranges)
        const long long k0 = tile_index(w, j) * BN;
        const int edge[] = {0, 1, 31, 63, 64, 126, 127};
        for (int t : edge) {
          long long row, sample;
          int head;
          if (!lane_row<MODE>(p, w, t, row, sample, head)) continue;
          for (int c : edge)
            if (!visible(p, MODE, row, k0 + c)) {
              if (bad < 5) std::printf("mode %d item %lld tile %d: pair (%lld, %lld) hidden\n", MODE, it, j, row, k0 + c);
              ++bad;
              break;
            }
        }
      }
    }
  }
  // rows (samples) from the call's first one are each held once; earlier ones never
  const long long first = MODE == MODE_SPARSE ? p.q_row0 : 0;
  for (size_t i = 0; i < held.size(); ++i)
    if ((long long)(i % per_head) >= first ? !held[i] : held[i]) {
      if (bad < 5) std::printf("mode %d: (b, head, row) %zu held %d times\n", MODE, i, (int)held[i]);
      ++bad;
    }
  return bad;
}

// The split-K units of the dense pass, for a plan made by plan_split_k():
// every M-tile's causal key range [0, L) is covered exactly once by its chunks
// (chunk c holds tiles [c chunk, min(L, (c+1) chunk))); the units of split
// M-tiles hold distinct partial slots that fill [0, n_multi), and
// partial_slot() finds every chunk's slot; each split M-tile has one merge
// ticket, distinct from every other M-tile's, in [0, n_multi); the unit's
// (b, head group) and M-tile index are those of its rows.  In the level
// order, units run group by group, level by level from the top, and by
// descending M-tile inside a level, each at most `chunk` tiles.
static int check_dense_units(const Params& p) {
  int bad = 0;
  auto fail = [&](const char* what, long long u) {
    if (bad < 5) std::printf("dense unit %lld (order %d): %s\n", u, p.order, what);
    ++bad;
  };
  const long long n_mt = (long long)p.B * p.groups_per_b * p.mtiles;
  std::vector<long long> covered((size_t)n_mt, 0), ticket_of((size_t)n_mt, -1);
  std::vector<std::vector<long long>> slot_of_chunk((size_t)n_mt);
  std::vector<char> slot_used((size_t)p.n_multi, 0), ticket_used((size_t)p.n_multi, 0);
  long long prev_gi = -1, prev_c = 0, prev_t = 0;
  for (long long u = 0; u < p.n_units; ++u) {
    const Work w = decode_strided_dense(p, u);
    const long long t = w.r0 / p.R;
    const long long gi = (long long)w.b * p.groups_per_b + w.h0 / p.Hp;
    if (w.b < 0 || w.b >= p.B || t < 0 || t >= p.mtiles || w.t != t || w.gi != gi) {
      fail("rows do not match the M-tile index", u);
      continue;
    }
    const long long idx = gi * p.mtiles + t;
    const long long L = strided_dense_len(p, t);
    const int c = w.chunk_idx;
    if (w.kt_lo != (long long)c * p.chunk || w.kt_hi != lmin(L, (long long)(c + 1) * p.chunk) - 1 ||
        w.n_chunks != cdiv(L, p.chunk) || w.T != w.kt_hi - w.kt_lo + 1 || w.T < 1)
      fail("key range of the chunk", u);
    std::vector<long long>& sl = slot_of_chunk[(size_t)idx];
    if (sl.empty()) sl.assign((size_t)w.n_chunks, -2);
    if (c < 0 || c >= (int)sl.size() || sl[(size_t)c] != -2) {
      fail("chunk held twice", u);
      continue;
    }
    sl[(size_t)c] = w.unit;
    covered[(size_t)idx] += w.T;
    if (w.n_chunks > 1) {
      if (w.unit < 0 || w.unit >= p.n_multi || slot_used[(size_t)w.unit]) fail("partial slot", u);
      else slot_used[(size_t)w.unit] = 1;
      if (partial_slot(p, w, c) != w.unit) fail("partial_slot() of its own chunk", u);
      if (w.u0 < 0 || w.u0 >= p.n_multi) fail("ticket out of range", u);
      else if (ticket_of[(size_t)idx] < 0) {
        if (ticket_used[(size_t)w.u0]) fail("ticket shared by two M-tiles", u);
        ticket_used[(size_t)w.u0] = 1;
        ticket_of[(size_t)idx] = w.u0;
      } else if (ticket_of[(size_t)idx] != w.u0) {
        fail("chunks of one M-tile with different tickets", u);
      }
    }
    if (p.order == SPLIT_LEVELS) {
      if (w.T > p.chunk) fail("unit longer than a chunk", u);
      const bool next = gi > prev_gi || (gi == prev_gi && (c < prev_c || (c == prev_c && t < prev_t)));
      if (u > 0 && !next) fail("level order", u);
      if (gi < prev_gi) fail("group order", u);
      prev_gi = gi;
      prev_c = c;
      prev_t = t;
    }
  }
  for (long long idx = 0; idx < n_mt; ++idx) {
    const long long t = idx % p.mtiles;
    const std::vector<long long>& sl = slot_of_chunk[(size_t)idx];
    bool ok = covered[(size_t)idx] == strided_dense_len(p, t) && !sl.empty();
    for (size_t c = 0; ok && c < sl.size(); ++c) ok = sl[c] != -2;
    if (ok && sl.size() > 1) {  // the merge finds every chunk's partial from any unit of the M-tile
      const Work w = decode_strided_dense(p, 0);
      Work m = w;
      m.gi = idx / p.mtiles;
      m.t = t;
      m.u0 = ticket_of[(size_t)idx];
      for (size_t c = 0; ok && c < sl.size(); ++c) ok = partial_slot(p, m, (int)c) == sl[c];
    }
    if (!ok) {
      if (bad < 5) std::printf("dense M-tile %lld (order %d) not covered exactly once\n", idx, p.order);
      ++bad;
    }
  }
  for (long long sidx = 0; sidx < p.n_multi; ++sidx)
    if (!slot_used[(size_t)sidx]) {
      if (bad < 5) std::printf("partial slot %lld (order %d) unused\n", sidx, p.order);
      ++bad;
    }
  return bad;
}

// Plans made by the library's planner for several machines and policies:
// SM counts 152, 7 and 1; the library's policy; units of a few tiles (many
// levels on small shapes); at most two levels; and a zero budget
// (longest-first whenever an M-tile splits).
struct PlanCase {
  int sms;
  SplitPolicy pol;
};
static const PlanCase kPlans[] = {{152, {kMaxLevelsUsed, kUnitTiles, kMinChunk, kLevelPartialBytes}},
                                  {7, {kMaxLevelsUsed, 2, 1, kLevelPartialBytes}},
                                  {1, {2, 1, 1, kLevelPartialBytes}},
                                  {152, {kMaxLevelsUsed, 3, 1, 0}},
                                  {1, {kMaxLevels, 1, 1, kLevelPartialBytes}}};

// The two-CTA sink + window kernel (G even, whole sequences): the CTAs 2c and
// 2c + 1 of a cluster walk items 2c + k grid and 2c + 1 + k grid.  With G and
// the grid even these are always the two heads h0, h0 + 1 of one KV group and
// one row tile, whose key-tile lists and masked-tile ranges are identical, and
// both CTAs see the same number of items: the leader's MMAs serve both.
static int check_pairs(const Params& p) {
  int bad = 0;
  const long long n = (long long)p.B * p.Hq * p.qtiles;
  if (n % 2 != 0) {
    std::printf("pairs: odd item count %lld\n", n);
    return 1;
  }
  for (long long lin = 0; lin < n; lin += 2) {
    const Work a = decode_work<MODE_SPARSE>(p, lin), b = decode_work<MODE_SPARSE>(p, lin + 1);
    bool same = a.b == b.b && a.g == b.g && b.h0 == a.h0 + 1 && a.r0 == b.r0 && a.r_last == b.r_last &&
                a.kt_lo == b.kt_lo && a.kt_hi == b.kt_hi && a.n_sink_tiles == b.n_sink_tiles && a.T == b.T;
    int a0, a1, b0, b1;
    unmasked_tiles<MODE_SPARSE>(p, a, a0, a1);
    unmasked_tiles<MODE_SPARSE>(p, b, b0, b1);
    same = same && a0 == b0 && a1 == b1;
    for (int j = 0; same && j < a.T; ++j) same = tile_index(a, j) == tile_index(b, j);
    if (!same) {
      if (bad < 5) std::printf("pairs: items %lld and %lld differ (heads %d, %d)\n", lin, lin + 1, a.h0, b.h0);
      ++bad;
    }
  }
  for (long long grid : {2LL, 148LL, 150LL, 152LL}) {
    for (long long c = 0; 2 * c < grid; ++c)
      for (long long x = 2 * c; x < n || x + 1 < n; x += grid)
        if ((x < n) != (x + 1 < n)) {
          if (bad < 5) std::printf("pairs: grid %lld cluster %lld sees unequal item counts\n", grid, c);
          ++bad;
        }
  }
  return bad;
}

// q_row0: a row-range call computing rows [q_row0, N) (0: the whole sequence).
static int check_shape(int B, int Hq, int Hkv, long long N, long long win, int ns, int gm, long long q_row0 = 0) {
  int bad = 0;
  Params p = {};
  p.B = B; p.Hq = Hq; p.Hkv = Hkv; p.G = Hq / Hkv; p.N = N; p.n_sink = ns; p.window = win; p.gamma = gm;
  p.q_row0 = q_row0; p.row0 = q_row0; p.o_rows = N - q_row0;
  p.n_s = (N - q_row0 + gm - 1) / gm;
  packing(p.G, &p.Hp, &p.R);
  p.groups_per_b = p.Hq / p.Hp;
  p.qtiles = (N - q_row0 + BM - 1) / BM;
  plan_split_k(p, 152, 128);
  bad += check<MODE_SPARSE>(p, (long long)p.B * p.Hq * p.qtiles);
  if (q_row0 == 0 && p.G % 2 == 0) bad += check_pairs(p);
  bad += check<MODE_STRIDED_SPARSE>(p, (long long)p.B * p.groups_per_b * p.mtiles);
  {  // the library's own policy for this shape
    Params q = p;
    plan_split_k(q, 152, 128);
    bad += check_dense_units(q);
  }
  for (const PlanCase& pc : kPlans) {
    Params q = p;
    plan_split_k(q, pc.sms, 128, pc.pol);
    bad += check<MODE_STRIDED_DENSE>(q, q.n_units);
    bad += check_dense_units(q);
    // the dense tail: gamma 1 from row N - tail
    for (long long tail : {1LL, 77LL, N}) {
      if (tail > N) continue;
      Params r = p;
      r.gamma = 1; r.n_s = tail; r.row0 = N - tail;
      plan_split_k(r, pc.sms, 128, pc.pol);
      bad += check<MODE_STRIDED_DENSE>(r, r.n_units);
      bad += check_dense_units(r);
    }
  }
  return bad;
}

// visible_bits() against the key-set definition, bit by bit: window and
// causal range [lo, hi] (empty when hi < lo) and sinks c < se.
static int check_visible_bits() {
  int bad = 0;
  const int ses[] = {0, 1, 3, 4, 31, 32, 33, 64, 100, 127, 128};
  for (int lo = 0; lo <= BN + 1; ++lo)
    for (int hi = -1; hi < BN; ++hi)
      for (int se : ses)
        for (int c0 = 0; c0 < BN; c0 += 32) {
          const uint32_t v = visible_bits(lo, hi, se, c0);
          for (int c = c0; c < c0 + 32; ++c) {
            const bool want = (lo <= c && c <= hi) || c < se;
            if (((v >> (c - c0)) & 1u) != (want ? 1u : 0u)) {
              if (bad < 5) std::printf("visible_bits(%d, %d, %d, %d): key %d\n", lo, hi, se, c0, c);
              ++bad;
            }
          }
        }
  return bad;
}

int main() {
  int bad = check_visible_bits(), cases = 0;
  const long long Ns[] = {1, 100, 128, 129, 1000, 4097, 20000};
  const long long windows[] = {1, 7, 64, 128, 129, 300, 2048, 100000};
  const int sinks[] = {0, 1, 4, 130, 300};
  const int gammas[] = {1, 3, 16, 64, 200};
  for (long long N : Ns)
    for (long long win : windows)
      for (int ns : sinks)
        for (int gm : gammas) {
          bad += check_shape(1, 4, 2, N, win, ns, gm);
          ++cases;
        }
  // other head packings (GQA 1, 3, 4 with B = 2, 16) on a smaller grid
  const int packs[][3] = {{1, 2, 2}, {1, 6, 2}, {2, 8, 2}, {1, 16, 1}};
  for (const auto& hk : packs)
    for (long long N : {1LL, 129LL, 1000LL, 4097LL})
      for (long long win : {1LL, 64LL, 300LL, 2048LL})
        for (int ns : {0, 4, 300})
          for (int gm : {1, 3, 16, 64}) {
            bad += check_shape(hk[0], hk[1], hk[2], N, win, ns, gm);
            ++cases;
          }
  // row ranges of a longer sequence (context parallelism): the first row a
  // multiple of 128 and of gamma
  for (long long N : {1000LL, 4097LL, 20000LL})
    for (long long win : {1LL, 300LL, 2048LL})
      for (int ns : {0, 4, 300})
        for (int gm : {1, 16, 64, 3, 48})
          for (long long q_row0 : {128LL * 3, 128LL * 48, 128LL * 96}) {
            if (q_row0 % gm != 0 || q_row0 >= N) continue;
            bad += check_shape(1, 4, 2, N, win, ns, gm, q_row0);
            ++cases;
          }
  std::printf("%d shapes, %d mismatches\n", cases, bad);
  return bad == 0 ? 0 : 1;
}
