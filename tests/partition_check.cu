// Host-side check of CostPartition (csrc/common.cuh), the split of the
// verification kernel's tile sequence into shares of equal cost.  For seeded
// random batches (ragged sequences, empty ones among them), grid sizes and
// switch weights w: the shares cover the tile sequence exactly and in order,
// the share that the merge bookkeeping looks up for every tile is the share
// that holds it, and no share costs more than ceil(C / G), the cost of a share
// being its tiles plus w for every switch from one slab to the next.
// Prints "ok <cases>" and exits 0, or prints the first failures and exits 1.
#include <cstdio>
#include <random>
#include <vector>

#include "common.cuh"

namespace {

// the index among slabs with tiles of the slab holding tile g
int slab_of(const std::vector<long long>& start, const std::vector<int>& nt, const std::vector<int>& sidx,
            long long g) {
  int b = 0;
  while (b + 1 < (int)nt.size() && start[b + 1] <= g) ++b;
  return sidx[b] + (int)((g - start[b]) / nt[b]);
}

}  // namespace

int main() {
  std::mt19937 rng(20261202);
  auto pick = [&](std::initializer_list<int> v) { return *(v.begin() + rng() % v.size()); };
  int cases = 0, failures = 0;
  for (int it = 0; it < 3000 && failures < 10; ++it) {
    const int B = pick({1, 2, 3, 4, 8, 37, 64});
    const int H = pick({1, 2, 8, 32, 52});
    std::vector<int> nt(B);
    for (int b = 0; b < B; ++b) nt[b] = pick({0, 1, 2, 7, 33, 257, (int)(rng() % 301)});
    const int G = pick({1, 2, 7, 100, 152, 1000});
    const int w = pick({0, 1, 4, 5, 8});
    std::vector<long long> start(B + 1);
    std::vector<int> sidx(B + 1), len(B), plen(B);
    long long T = 0;
    int k = 0;
    for (int b = 0; b < B; ++b) {
      start[b] = T;
      sidx[b] = k;
      T += (long long)H * nt[b];
      if (nt[b] > 0) k += H;
    }
    start[B] = T;
    sidx[B] = k;
    glide::BatchTiles bt;
    bt.start = start.data();
    bt.ntiles = nt.data();
    bt.len = len.data();
    bt.plen = plen.data();
    bt.sidx = sidx.data();
    glide::CostPartition P;
    P.init(bt, B, H, G, w);
    ++cases;
    const long long cap = (P.C + G - 1) / G;  // the largest part of the cost line
    long long prev = 0;
    bool ok = true;
    for (int c = 0; c < G && ok; ++c) {
      const long long b0 = P.begin(c), e0 = P.end(c);
      if (b0 != prev || e0 < b0) {
        std::printf("case %d (B=%d H=%d G=%d w=%d): share %d is [%lld, %lld), expected to start at %lld\n", it, B, H, G,
                    w, c, b0, e0, prev);
        ok = false;
      } else if (e0 > b0) {
        const long long cost = (e0 - b0) + (long long)w * (slab_of(start, nt, sidx, e0 - 1) - slab_of(start, nt, sidx, b0));
        if (cost > cap) {
          std::printf("case %d (B=%d H=%d G=%d w=%d): share %d costs %lld > %lld\n", it, B, H, G, w, c, cost, cap);
          ok = false;
        }
      }
      prev = e0;
    }
    if (ok && prev != T) {
      std::printf("case %d (B=%d H=%d G=%d w=%d): shares end at %lld of %lld tiles\n", it, B, H, G, w, prev, T);
      ok = false;
    }
    for (long long g = 0; ok && g < T && T <= 200000; ++g) {
      const int c = P.cta_of(g);
      if (c < 0 || c >= G || g < P.begin(c) || g >= P.end(c)) {
        std::printf("case %d (B=%d H=%d G=%d w=%d): tile %lld looked up in share %d\n", it, B, H, G, w, g, c);
        ok = false;
      }
    }
    if (!ok) ++failures;
  }
  if (failures) {
    std::printf("FAIL %d of %d cases\n", failures, cases);
    return 1;
  }
  std::printf("ok %d\n", cases);
  return 0;
}
