// Host-side check of the tile geometry in tiles.cuh (compiled as plain C++ by
// tests/test_tile_geometry.py): for every work item of many shapes and all
// three modes, unmasked_tiles() must select exactly the tiles for which
// tile_needs_mask() is false, and tile_needs_mask() must be true wherever a
// (row, key) pair of the tile is not visible (checked pair by pair against
// the definition of the key sets), and the dense pass's split-K units cover
// every M-tile's causal key range exactly once in the order the partial slots
// and tickets assume.  For every head packing of the dense tiles (GQA 1, 2,
// 3, 4 and 16), each lane's query head reads its own KV head (floor(h / G))
// and every (batch, head, row or sample) sits in exactly one lane.
#define __host__
#define __device__
#define __forceinline__ inline
#include <cstdio>
#include <cstdlib>
#include <initializer_list>
#include <vector>
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
    Work w = decode_work<MODE>(p, it);
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
  for (size_t i = 0; i < held.size(); ++i)
    if (!held[i]) {
      if (bad < 5) std::printf("mode %d: (b, head, row) %zu held by no lane\n", MODE, i);
      ++bad;
    }
  return bad;
}

// The split-K units of the dense pass: every M-tile's key range [0, L) is
// covered exactly once by adjacent units u0 .. u0 + n_chunks - 1, units with
// more than one chunk are exactly [0, n_multi), and the (b, head group, t)
// of each unit is a valid M-tile.
static int check_dense_units(const Params& p) {
  int bad = 0;
  std::vector<long long> cover((size_t)p.B * p.groups_per_b * p.mtiles, -1);
  std::vector<int> seen_tiles((size_t)p.B * p.groups_per_b * p.mtiles, 0);
  for (long long u = 0; u < p.n_units; ++u) {
    const Work w = decode_strided_dense(p, u);
    const long long t = w.r0 / p.R;
    const long long idx = ((long long)w.b * p.groups_per_b + w.h0 / p.Hp) * p.mtiles + t;
    const long long L = strided_dense_len(p, t);
    bool ok = w.b >= 0 && w.b < p.B && t >= 0 && t < p.mtiles && w.kt_lo == (long long)w.chunk_idx * p.chunk &&
              w.kt_hi == lmin(L, (long long)(w.chunk_idx + 1) * p.chunk) - 1 && w.n_chunks == cdiv(L, p.chunk) &&
              w.u0 == u - w.chunk_idx && ((w.n_chunks > 1) == (u < p.n_multi));
    if (ok && w.chunk_idx == 0) {
      ok = cover[idx] < 0;
      cover[idx] = u;
    }
    if (ok) seen_tiles[idx] += w.T;
    if (!ok) {
      if (bad < 5) std::printf("dense unit %lld: bad decode (t %lld chunk %d of %d)\n", u, t, w.chunk_idx, w.n_chunks);
      ++bad;
    }
  }
  for (size_t i = 0; i < cover.size(); ++i) {
    const long long t = (long long)(i % p.mtiles);
    if (cover[i] < 0 || seen_tiles[i] != strided_dense_len(p, t)) {
      if (bad < 5) std::printf("dense M-tile %zu not covered exactly once\n", i);
      ++bad;
    }
  }
  return bad;
}

// Hp query heads of one KV group share a dense tile when G is a power of two
// up to 16 (R = 128 / Hp samples each); otherwise one head per tile.
static void set_packing(Params& p) {
  p.Hp = (p.G >= 2 && p.G <= 16 && (p.G & (p.G - 1)) == 0) ? p.G : 1;
  p.R = BM / p.Hp;
  p.groups_per_b = p.Hq / p.Hp;
}

static long long count_units(Params& p) {
  p.mtiles = (p.n_s + p.R - 1) / p.R;
  long long units = 0, multi = 0;
  for (long long t = 0; t < p.mtiles; ++t) {
    const long long nc = (strided_dense_len(p, t) + p.chunk - 1) / p.chunk;
    units += nc;
    if (nc > 1) multi += nc;
  }
  p.n_units = units * p.B * p.groups_per_b;
  p.n_multi = multi * p.B * p.groups_per_b;
  return p.n_units;
}

static int check_shape(int B, int Hq, int Hkv, long long N, long long win, int ns, int gm) {
  int bad = 0;
  Params p = {};
  p.B = B; p.Hq = Hq; p.Hkv = Hkv; p.G = Hq / Hkv; p.N = N; p.n_sink = ns; p.window = win; p.gamma = gm;
  p.n_s = (N + gm - 1) / gm;
  set_packing(p);
  p.qtiles = (N + BM - 1) / BM;
  p.chunk = 3;
  count_units(p);
  bad += check<MODE_SPARSE>(p, (long long)p.B * p.Hq * p.qtiles);
  bad += check<MODE_STRIDED_SPARSE>(p, (long long)p.B * p.groups_per_b * p.mtiles);
  bad += check<MODE_STRIDED_DENSE>(p, p.n_units);
  bad += check_dense_units(p);
  // the dense tail: gamma 1 from row N - tail
  for (long long tail : {1LL, 77LL, N}) {
    if (tail > N) continue;
    Params q = p;
    q.gamma = 1; q.n_s = tail; q.row0 = N - tail;
    count_units(q);
    bad += check<MODE_STRIDED_DENSE>(q, q.n_units);
    bad += check_dense_units(q);
  }
  return bad;
}

int main() {
  int bad = 0, cases = 0;
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
  std::printf("%d shapes, %d mismatches\n", cases, bad);
  return bad == 0 ? 0 : 1;
}
