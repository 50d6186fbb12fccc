// Host-only checks of the tile bookkeeping: the Gram tile table (gram_fill_tiles) lists every
// 256 x 256 output tile that meets the lower triangle exactly once, its lookup table maps
// each listed tile to its index and every other tile to -1, and consecutive entries stay
// inside square supertiles; lower_tile (the persistent Cholesky update's tile walk) maps
// 0..T-1 onto the lower triangle in row-major order.  Prints "ok" or the first violation.
#include <cstdio>
#include <vector>

#include "ffh_internal.cuh"

using namespace ffh;

static int check(int64_t d) {
  const int nbm = (int)((d + kGramBM - 1) / kGramBM), nbn = (int)((d + kGramBN - 1) / kGramBN);
  std::vector<int2> tiles(nbm * nbn);
  std::vector<int> lut(nbm * nbn, -7);
  const int T = gram_fill_tiles(nbm, nbn, tiles.data(), lut.data());
  std::vector<int> seen(nbm * nbn, 0);
  int expect = 0;
  for (int ti = 0; ti < nbm; ++ti)
    for (int tj = 0; tj < nbn; ++tj) {
      const bool lower = (int64_t)tj * kGramBN <= (int64_t)ti * kGramBM + kGramBM - 1;
      expect += lower;
      const int v = lut[ti * nbn + tj];
      if (!lower && v != -1) return printf("d=%lld tile (%d,%d) above the triangle has lut %d\n", (long long)d, ti, tj, v), 1;
      if (lower && (v < 0 || v >= T)) return printf("d=%lld tile (%d,%d) lut %d out of range\n", (long long)d, ti, tj, v), 1;
    }
  if (T != expect) return printf("d=%lld: %d tiles listed, %d expected\n", (long long)d, T, expect), 1;
  for (int t = 0; t < T; ++t) {
    const int ti = tiles[t].x, tj = tiles[t].y;
    if (ti < 0 || ti >= nbm || tj < 0 || tj >= nbn) return printf("d=%lld: entry %d out of the grid\n", (long long)d, t), 1;
    if (seen[ti * nbn + tj]++) return printf("d=%lld: tile (%d,%d) listed twice\n", (long long)d, ti, tj), 1;
    if (lut[ti * nbn + tj] != t) return printf("d=%lld: lut of entry %d is %d\n", (long long)d, t, lut[ti * nbn + tj]), 1;
    if (t > 0) {
      // supertile order: the previous entry is in the same supertile or an earlier one
      const int pi = tiles[t - 1].x / kGramSuper, pj = tiles[t - 1].y / kGramSuper;
      const int ci = ti / kGramSuper, cj = tj / kGramSuper;
      if (!(ci > pi || (ci == pi && cj >= pj))) return printf("d=%lld: entry %d leaves supertile order\n", (long long)d, t), 1;
    }
  }
  return 0;
}

// lower_tile: a bijection from 0..T-1 onto the tiles (tm, tn), tn <= tm, in row-major order
static int check_lower_tile(int ntm) {
  int t = 0;
  for (int tm = 0; tm < ntm; ++tm)
    for (int tn = 0; tn <= tm; ++tn, ++t) {
      int a, b;
      lower_tile(t, a, b);
      if (a != tm || b != tn)
        return printf("lower_tile(%d) = (%d,%d), expected (%d,%d)\n", t, a, b, tm, tn), 1;
    }
  return 0;
}

int main() {
  for (int64_t d : {1, 64, 255, 256, 257, 4096, 3000, 11008, 14336, 40000})
    if (check(d)) return 1;
  // up to a 65536 x 65536 trailing matrix of 128 x 128 tiles
  if (check_lower_tile(512)) return 1;
  printf("ok\n");
  return 0;
}
