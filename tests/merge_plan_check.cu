// Host-side check of the merge Gram's tile plan on SM pairs (Sec. 4.3, the
// nearest-kept-token assignment): for each shape given on the command line,
// every pruned row of every sample must get each partial slot written exactly
// once (by its range's tile, or as the spare slot of a group with fewer
// ranges), every range must be 1..256 columns wide, its box height one of the
// plan's, and each pair's tiles distinct, and a second request for the same
// shape (from the plan cache) must give the same plan. Prints "ok" per shape or
// the first violation. Built and run by tests/test_merge_plan.py (host code only: no
// GPU is touched).
#include "../paper_2608_25332_gb300/csrc/merge_pair_tc.cu"

#include <cstdio>
#include <cstdlib>
#include <set>
#include <vector>

namespace provip {
int make_tmap_bf16_2d(CUtensorMap*, const void*, uint64_t, uint64_t, uint64_t, uint32_t) { return -1; }
}  // namespace provip

using namespace provip;

static int check(int B, int N_v, int keep, int D, int sms) {
  const int n_pruned = N_v - keep;
  MergePairPlan p;
  if (!merge_pair_plan(B, n_pruned, keep, D, sms, &p)) {
    // no split into at most 16 ranges of at most 256 columns: the caller takes
    // the single-SM form
    printf("noplan B=%d N_v=%d keep=%d\n", B, N_v, keep);
    return 0;
  }
  // a second request (answered from the plan cache once the shape is known)
  // gives the same plan
  MergePairPlan q;
  if (!merge_pair_plan(B, n_pruned, keep, D, sms, &q) || q.n_quads != p.n_quads || q.Q != p.Q ||
      q.n_lo != p.n_lo || q.x_hi != p.x_hi || q.T != p.T || q.P != p.P || q.n_slots != p.n_slots ||
      q.n_heights != p.n_heights) {
    printf("B=%d N_v=%d keep=%d: a second request gave another plan\n", B, N_v, keep);
    return 1;
  }
  if (p.P < 1 || p.P > sms / 2 || p.n_slots < 1 || p.n_slots > kMergeMaxSplit || p.n_heights < 1 ||
      p.n_heights > kMergePairHeights) {
    printf("B=%d N_v=%d keep=%d: bad plan P=%d slots=%d heights=%d\n", B, N_v, keep, p.P, p.n_slots,
           p.n_heights);
    return 1;
  }
  std::vector<unsigned char> cover((size_t)B * n_pruned * p.n_slots, 0);
  std::set<int> seen;
  for (int pair = 0; pair < p.P; ++pair) {
    for (int r = 0, k; (k = pair_deal_tile(p, pair, r)) >= 0; ++r) {
      if (!seen.insert(k).second || k >= p.T) {
        printf("tile %d dealt twice or out of range\n", k);
        return 1;
      }
      const PairTile g = pair_tile(p, n_pruned, keep, k);
      if (g.nv < 1 || g.nv > 256 || g.N % 32 || g.N < g.nv) {
        printf("tile %d: %d columns (MMA width %d)\n", k, g.nv, g.N);
        return 1;
      }
      bool h_ok = false;
      for (int j = 0; j < p.n_heights; ++j) h_ok |= p.heights[j] == g.N / 2;
      if (!h_ok || g.c0 + g.nv > keep || g.b >= B) {
        printf("tile %d: height %d, columns %d..%d, sample %d\n", k, g.N / 2, g.c0, g.c0 + g.nv, g.b);
        return 1;
      }
      const bool spare = g.t + 1 == g.n && g.n < p.n_slots;
      for (int pos = g.m0; pos < g.m0 + 512 && pos < n_pruned; ++pos) {
        if (pos >= g.m0 + 256 && !g.has1) {
          printf("tile %d: row %d of the second half without its MMA\n", k, pos);
          return 1;
        }
        for (int sl = g.t; sl <= (spare ? g.t + 1 : g.t); ++sl) ++cover[((size_t)g.b * n_pruned + pos) * p.n_slots + sl];
      }
    }
  }
  if ((int)seen.size() != p.T) {
    printf("%zu of %d tiles dealt\n", seen.size(), p.T);
    return 1;
  }
  for (size_t i = 0; i < cover.size(); ++i)
    if (cover[i] != 1) {
      printf("B=%d N_v=%d keep=%d: row %zu slot %zu written %d times\n", B, N_v, keep, i / p.n_slots,
             i % p.n_slots, cover[i]);
      return 1;
    }
  printf("ok B=%d N_v=%d keep=%d T=%d P=%d slots=%d\n", B, N_v, keep, p.T, p.P, p.n_slots);
  return 0;
}

int main(int argc, char** argv) {
  // arguments: groups of B N_v keep D sms
  int rc = 0;
  for (int i = 1; i + 4 < argc; i += 5)
    rc |= check(atoi(argv[i]), atoi(argv[i + 1]), atoi(argv[i + 2]), atoi(argv[i + 3]), atoi(argv[i + 4]));
  return rc;
}
