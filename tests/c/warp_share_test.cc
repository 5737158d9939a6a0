// warp_share_test.cc -- checks the rule that shares one sweep launch's warps
// among the element-type/alignment classes, and the cost-weighted cut of a
// class into warp ranges (csrc/warp_share.h), on the host.
// Exits 0 and prints "warp_share ok" when every check holds.
#include <cmath>
#include <cstdio>
#include <vector>

#include "warp_share.h"

using namespace frk;

#define EXPECT(c)                                                    \
  do {                                                               \
    if (!(c)) {                                                      \
      std::fprintf(stderr, "%s:%d check failed: %s\n", __FILE__, __LINE__, #c); \
      return 1;                                                      \
    }                                                                \
  } while (0)

// One case: n classes with the given costs, n_ctas CTAs of wpc warps.
static int check(const std::vector<double>& cost, int n_ctas, int wpc) {
  const int n = static_cast<int>(cost.size());
  const uint64_t W = static_cast<uint64_t>(n_ctas) * wpc;
  std::vector<uint64_t> wc(n);
  share_warps(cost.data(), n, W, wc.data());
  double total = 0.0;
  for (double c : cost) total += c;
  uint64_t sum = 0;
  for (int q = 0; q < n; ++q) {
    EXPECT(wc[q] >= 1);
    sum += wc[q];
    // within one warp of the exact share, unless the class was lifted to one
    const double share = static_cast<double>(W) * cost[q] / total;
    EXPECT(std::fabs(static_cast<double>(wc[q]) - share) < 1.0 + 1e-9 || (wc[q] == 1 && share < 1.0) ||
           n * 1.0 > share);
  }
  EXPECT(sum == W);
  std::vector<uint32_t> slot(static_cast<size_t>(n) * W, 0xFFFFFFFFu);
  spread_warps(wc.data(), n, W, n_ctas, wpc, slot.data(), W);
  // the slots are a permutation of the launch's warps
  std::vector<int> seen(W, 0);
  std::vector<std::vector<int>> per_cta(n, std::vector<int>(n_ctas, 0));
  for (int q = 0; q < n; ++q)
    for (uint64_t j = 0; j < wc[q]; ++j) {
      const uint32_t s = slot[q * W + j];
      EXPECT(s < W);
      EXPECT(seen[s] == 0);
      seen[s] = 1;
      per_cta[q][s / wpc] += 1;
    }
  // every CTA holds floor or ceil of its share of every class
  for (int q = 0; q < n; ++q)
    for (int c = 0; c < n_ctas; ++c) {
      const uint64_t lo = wc[q] / n_ctas, hi = (wc[q] + n_ctas - 1) / n_ctas;
      EXPECT(static_cast<uint64_t>(per_cta[q][c]) >= lo && static_cast<uint64_t>(per_cta[q][c]) <= hi);
    }
  return 0;
}

// split_ranges: boundaries are monotone, span [0, n], and each is the last
// one whose cost prefix is at most its share of the total; unit costs give
// floor(n * w / Wq).
static int check_split(const std::vector<uint64_t>& seg, uint64_t Wq) {
  const uint64_t n = seg.size();
  std::vector<uint64_t> pre(n + 1, 0);
  for (uint64_t s = 0; s < n; ++s) pre[s + 1] = pre[s] + seg[s];
  std::vector<uint64_t> bnd(Wq + 1);
  split_ranges([&](uint64_t s) { return pre[s]; }, n, Wq, bnd.data());
  EXPECT(bnd[0] == 0 && bnd[Wq] == n);
  for (uint64_t w = 0; w <= Wq; ++w) {
    if (w > 0) EXPECT(bnd[w] >= bnd[w - 1]);
    const unsigned __int128 target = static_cast<unsigned __int128>(pre[n]) * w;
    EXPECT(static_cast<unsigned __int128>(pre[bnd[w]]) * Wq <= target || w == 0);
    EXPECT(bnd[w] == n || static_cast<unsigned __int128>(pre[bnd[w] + 1]) * Wq > target || w == 0);
  }
  return 0;
}

int main() {
  // split_ranges on unit costs is the equal-count split
  for (uint64_t n : {0ull, 1ull, 7ull, 1000ull, 4099ull})
    for (uint64_t Wq : {1ull, 3ull, 16ull, 2432ull}) {
      std::vector<uint64_t> pre(n + 1);
      for (uint64_t s = 0; s <= n; ++s) pre[s] = s;
      std::vector<uint64_t> bnd(Wq + 1);
      split_ranges([&](uint64_t s) { return pre[s]; }, n, Wq, bnd.data());
      for (uint64_t w = 0; w <= Wq; ++w) EXPECT(bnd[w] == n * w / Wq);
    }
  // uneven costs: chunk starts, partial segments, zero-cost runs
  {
    std::vector<uint64_t> seg;
    uint32_t x = 12345;
    for (int i = 0; i < 5000; ++i) {
      x = x * 1103515245u + 12345u;
      const uint64_t blocks = 1 + (x >> 16) % 32;
      seg.push_back(seg_cost(blocks, (x >> 8) % 5 == 0));
    }
    for (uint64_t Wq : {1ull, 2ull, 152ull, 2432ull, 6000ull})
      if (check_split(seg, Wq)) return 1;
    if (check_split({0, 0, 5, 0, 0, 7, 0}, 4)) return 1;
  }
  EXPECT(seg_cost(32, true) > seg_cost(32, false) && seg_cost(32, false) > seg_cost(1, false));

  // a Llama shard: bf16 weights (1/7 of the bytes, weighted 1.25) and fp32 state
  const double bf16 = 1.0 * block_weight(kDtBf16, kShareFingerprint);
  const double f32 = 6.0 * block_weight(kDtF32, kShareFingerprint);
  if (check({bf16, f32}, 152, 16)) return 1;
  if (check({1.0 * block_weight(kDtBf16, kSharePack), 6.0 * block_weight(kDtF32, kSharePack)}, 152, 20)) return 1;
  // one class; six classes, some tiny; a half-GPU batch; a single CTA
  if (check({5.0}, 152, 16)) return 1;
  if (check({1e-6, 3.0, 0.5, 1e-9, 40.0, 2.0}, 152, 16)) return 1;
  if (check({1.0, 1.0, 1.0}, 76, 20)) return 1;
  if (check({1.0, 2.0, 3.0, 4.0, 5.0, 6.0}, 1, 16)) return 1;
  if (check({1e-9, 1e-9, 1e-9, 1e-9, 1e-9, 1.0}, 1, 6)) return 1;
  // the weights: an fp32 block is the unit, bf16 costs more for the fingerprint only
  EXPECT(block_weight(kDtF32, kShareFingerprint) == 100.0);
  EXPECT(block_weight(kDtBf16, kShareFingerprint) > block_weight(kDtBf16, kSharePack));
  std::printf("warp_share ok\n");
  return 0;
}
