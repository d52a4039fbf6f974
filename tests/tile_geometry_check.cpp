// Host-side check of the tile geometry in tiles.cuh (compiled as plain C++ by
// tests/test_tile_geometry.py): for every work item of many shapes and all
// three modes, unmasked_tiles() must select exactly the tiles for which
// tile_needs_mask() is false, and tile_needs_mask() must be true wherever a
// (row, key) pair of the tile is not visible (checked pair by pair against
// the definition of the key sets), and the dense pass's split-K units cover
// every M-tile's causal key range exactly once in the order the partial slots
// and tickets assume.
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
  for (long long it = 0; it < items; ++it) {
    Work w = decode_work<MODE>(p, it);
    int j0, j1;
    unmasked_tiles<MODE>(p, w, j0, j1);
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
          Params p = {};
          p.B = 1; p.Hq = 4; p.Hkv = 2; p.G = 2; p.N = N; p.n_sink = ns; p.window = win; p.gamma = gm;
          p.n_s = (N + gm - 1) / gm;
          p.Hp = 2; p.R = BM / 2; p.groups_per_b = 2;
          p.mtiles = (p.n_s + p.R - 1) / p.R;
          p.qtiles = (N + BM - 1) / BM;
          p.chunk = 3;
          long long units = 0;
          for (long long t = 0; t < p.mtiles; ++t) units += (strided_dense_len(p, t) + p.chunk - 1) / p.chunk;
          p.n_units = units * p.B * p.groups_per_b;
          bad += check<MODE_SPARSE>(p, (long long)p.B * p.Hq * p.qtiles);
          bad += check<MODE_STRIDED_SPARSE>(p, (long long)p.B * p.groups_per_b * p.mtiles);
          p.n_multi = 0;
          for (long long t = 0; t < p.mtiles; ++t) {
            const long long nc = (strided_dense_len(p, t) + p.chunk - 1) / p.chunk;
            if (nc > 1) p.n_multi += nc;
          }
          p.n_multi *= (long long)p.B * p.groups_per_b;
          bad += check<MODE_STRIDED_DENSE>(p, p.n_units);
          bad += check_dense_units(p);
          // the dense tail: gamma 1 from row N - tail
          for (long long tail : {1LL, 77LL, N}) {
            if (tail > N) continue;
            Params q = p;
            q.gamma = 1; q.n_s = tail; q.row0 = N - tail;
            q.mtiles = (q.n_s + q.R - 1) / q.R;
            long long u = 0;
            for (long long t = 0; t < q.mtiles; ++t) u += (strided_dense_len(q, t) + q.chunk - 1) / q.chunk;
            q.n_units = u * q.B * q.groups_per_b;
            q.n_multi = 0;
            for (long long t = 0; t < q.mtiles; ++t) {
              const long long nc = (strided_dense_len(q, t) + q.chunk - 1) / q.chunk;
              if (nc > 1) q.n_multi += nc;
            }
            q.n_multi *= (long long)q.B * q.groups_per_b;
            bad += check<MODE_STRIDED_DENSE>(q, q.n_units);
            bad += check_dense_units(q);
          }
          ++cases;
        }
  std::printf("%d shapes, %d mismatches\n", cases, bad);
  return bad == 0 ? 0 : 1;
}
