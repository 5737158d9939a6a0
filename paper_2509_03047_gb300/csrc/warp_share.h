// warp_share.h -- how one sweep launch shares its warps among the (element
// type, alignment) classes of the chunks it covers.  Host code on plain
// arrays (the no-allocation fingerprint plans with it too).
//
// A warp sweeps a range of one class only.  The classes are not equally
// costly per block: a bf16 block holds twice the elements of an fp32 block,
// so the fingerprint spends about a quarter more instructions on it, while
// pack and unpack are bound by memory in every class.  The warps are shared
// in proportion to each class's blocks times its weight (percent of an fp32
// block), so that the classes' warps finish together; each class's warps are
// spread round-robin over the CTAs, so every SM runs a mix.
#pragma once

#include <cstdint>

#include "layout.h"

#ifndef FR_MIX_W_BF16
#define FR_MIX_W_BF16 125  // fingerprint: a bf16 block costs 1.25 fp32 blocks
#endif
#ifndef FR_MIX_W_BF16_PACK
#define FR_MIX_W_BF16_PACK 100  // pack and unpack: memory-bound, all blocks alike
#endif
#ifndef FR_MIX_W_BYTES
#define FR_MIX_W_BYTES 100
#endif

namespace frk {

enum : int { kShareFingerprint = 1, kSharePack = 2 };

// Weight of a block of element type `dt` for a launch of kind `kind`.
inline double block_weight(uint32_t dt, int kind) {
  if (dt == kDtF32) return 100.0;
  if (dt == kDtBf16) return kind == kShareFingerprint ? FR_MIX_W_BF16 : FR_MIX_W_BF16_PACK;
  return FR_MIX_W_BYTES;
}

// wc[q] = warps of class q (q < n <= W): W shared in proportion to cost[q] > 0,
// every class at least one, largest shortfall first for the remainder.
inline void share_warps(const double* cost, int n, uint64_t W, uint64_t* wc) {
  double total = 0.0;
  for (int q = 0; q < n; ++q) total += cost[q];
  uint64_t given = 0;
  for (int q = 0; q < n; ++q) {
    const uint64_t w = static_cast<uint64_t>(static_cast<double>(W) * cost[q] / total);
    wc[q] = w > 0 ? w : 1;
    given += wc[q];
  }
  while (given < W) {
    int best = 0;
    double gap = -1e300;
    for (int q = 0; q < n; ++q) {
      const double g = static_cast<double>(W) * cost[q] / total - static_cast<double>(wc[q]);
      if (g > gap) gap = g, best = q;
    }
    ++wc[best];
    ++given;
  }
  while (given > W) {  // only when many tiny classes each took one
    int best = 0;
    for (int q = 1; q < n; ++q)
      if (wc[q] > wc[best]) best = q;
    --wc[best];
    --given;
  }
}

// slot[q * stride + j] = launch-warp index of class q's j-th warp.  Slot i is
// warp i / n_ctas of CTA i % n_ctas (round robin over the CTAs), and each
// class takes a run of consecutive slots, so every CTA holds the floor or the
// ceiling of its share of every class.  sum(wc) == W.
inline void spread_warps(const uint64_t* wc, int n, uint64_t W, int n_ctas, int warps_per_cta, uint32_t* slot,
                         uint64_t stride) {
  uint64_t i = 0;
  for (int q = 0; q < n; ++q)
    for (uint64_t j = 0; j < wc[q] && i < W; ++j, ++i)
      slot[q * stride + j] = static_cast<uint32_t>((i % n_ctas) * warps_per_cta + i / n_ctas);
}

}  // namespace frk
