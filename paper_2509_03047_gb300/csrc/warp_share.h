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
// spread round-robin over the CTAs, so every SM runs a mix.  Within a class
// the ranges are cut by an estimated cost per segment (split_ranges).
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
// Within a class, warp ranges (whole 16 KiB sum segments) are cut by an
// estimated cost per segment, in units of one 512-byte block's sweep:
// FR_SPLIT_BLK per block it holds, FR_SPLIT_SEG for its end (the sums'
// check, fold and store), and FR_SPLIT_PIECE more if it begins a chunk (the
// warp's pipeline starts over on a new address and the CRC streams are
// folded at the end of the previous piece).  Measured on GB300: by bytes
// alone short segments are underpriced (gpt2s fingerprint -3 points against
// equal segment counts); these costs beat equal counts by up to half a point
// on the fragmented and small states.
#ifndef FR_SPLIT_BLK
#define FR_SPLIT_BLK 1
#endif
#ifndef FR_SPLIT_SEG
#define FR_SPLIT_SEG 2
#endif
#ifndef FR_SPLIT_PIECE
#define FR_SPLIT_PIECE 16
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

// Estimated cost of a segment of `blocks` blocks; `first`: it begins a chunk.
inline uint64_t seg_cost(uint64_t blocks, bool first) {
  return FR_SPLIT_BLK * blocks + FR_SPLIT_SEG + (first ? FR_SPLIT_PIECE : 0);
}

// bnd[w], w = 0..Wq: the segment where warp w's range starts, given the cost
// prefix cost(s) of segments [0, s) for s = 0..n (nondecreasing): the last
// boundary whose prefix is at most w / Wq of the total (bnd[0] = 0 even if
// the first segments cost nothing, bnd[Wq] = n).  With unit costs this is
// floor(n * w / Wq).
template <class Prefix>
inline void split_ranges(const Prefix& cost, uint64_t n, uint64_t Wq, uint64_t* bnd) {
  const unsigned __int128 total = cost(n);
  uint64_t s = 0;
  bnd[0] = 0;
  for (uint64_t w = 1; w <= Wq; ++w) {
    const unsigned __int128 target = total * w;
    while (s < n && static_cast<unsigned __int128>(cost(s + 1)) * Wq <= target) ++s;
    bnd[w] = s;
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
