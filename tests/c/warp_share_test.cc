// warp_share_test.cc -- checks the rule that shares one sweep launch's warps
// among the element-type/alignment classes (csrc/warp_share.h), on the host.
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

int main() {
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
