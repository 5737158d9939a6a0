// finalize.cu -- per-chunk fold, tails, headers and verification; ordered
// compaction of chunk ids; fingerprint diff.
//
// The sweep kernel leaves one record per piece (the part of a chunk body one
// warp covered).  Here one warp per chunk:
//   0. issues every load the chunk needs at once, after its descriptor;
//   1. shifts each record's raw CRC to its position in the chunk's body and
//      XORs them (raw(A||B) = raw(A) * x^(8|B|) ^ raw(B)), adds the records'
//      non-finite counts, and adds the body's 16 KiB segment sums of squares
//      in an order fixed by segment index (so the result does not depend on
//      the plan);
//   2. handles the chunk's tail (len % 512 bytes, if any) as the end of a
//      512-byte window with leading zeros, window word i in lane i % 32:
//      copies it for pack/unpack (whole words when aligned), adds its squares
//      to the lanes' segment sums before one lane tree, and CRCs it with the
//      body's raw CRC folded into the tail's first word (which continues the
//      body's CRC through the tail without shifting it): each lane combines
//      its words by constant multiplies, takes its lane's shift from a
//      shared-memory table, and the lanes are XORed;
//   3. applies CRC-32C's preset and final XOR:
//      crc = raw ^ 0xFFFFFFFF * x^(8 len) ^ 0xFFFFFFFF;
//   4. fingerprint: writes the table entry; pack: writes the 64-byte header,
//      the zero padding after the payload and, for the last chunk, the zero gap
//      after the header table; unpack: checks the header against the plan, the
//      header CRC, the payload CRC and the padding, and writes a verdict.
//      Pack and unpack-fp also write the table entry when given a table.
// The verdicts become an ascending id list through an ordered compaction --
// one CTA for up to one tile of ids, a cluster of CTAs sharing their tile
// counts through distributed shared memory beyond that -- which fr_diff
// shares with a different predicate.
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "gf2.cuh"
#include "kernels.h"
#include "layout.h"

namespace frk {

namespace {

#ifndef FR_FIN_MINB
#define FR_FIN_MINB 4  // finalize CTAs per SM (caps registers at 64: more chunks in flight)
#endif
constexpr int kFinWarps = 8;
constexpr int kFinThreads = kFinWarps * 32;
constexpr unsigned kFull = 0xFFFFFFFFu;

__device__ const PowTables g_pow = make_pow_tables();
// Byte tables for multiplying by x^1024 and x^2048: a tail lane combines its
// four window words, 32 words apart, with them.
__device__ const ByteTables4 g_x1024 = make_mul_tables(gf_xpow(1024));
__device__ const ByteTables4 g_x2048 = make_mul_tables(gf_xpow(2048));

// a * m mod P, T being the byte tables of the constant m.
__device__ __forceinline__ uint32_t mul_const(const ByteTables4& T, uint32_t a) {
  return (__ldg(&T.t[0][a & 255u]) ^ __ldg(&T.t[1][(a >> 8) & 255u])) ^
         (__ldg(&T.t[2][(a >> 16) & 255u]) ^ __ldg(&T.t[3][a >> 24]));
}

// Per-lane multipliers.  In a 128-word window whose word i goes to lane
// i % 32, a word of lane l has (31 - l) + 32j words after it, j fixed by its
// slot, so lane l's partial CRC takes the shift M_l = x^(32 (32 - l)) (the
// word's own x^32 included) before the lanes are XORed together.  The
// product (n << 4k) * M_l, for nibble position k and nibble value n, sits at
// word (16k + n) * 32 + l: the 32 lanes' lookups of one nibble position fall
// in 32 different shared-memory banks.  16 KiB.
constexpr int kLaneMulWords = 8 * 16 * 32;
struct alignas(16) LaneMulTable {
  uint32_t t[kLaneMulWords];
};
__host__ __device__ constexpr LaneMulTable make_lane_mul_table() {
  LaneMulTable out{};
  for (int l = 0; l < 32; ++l) {
    const uint32_t m = gf_xpow(32ull * static_cast<uint64_t>(32 - l));
    for (int k = 0; k < 8; ++k) {
      uint32_t bit[4] = {};
      for (int j = 0; j < 4; ++j) bit[j] = gf_mulmod(1u << (4 * k + j), m);
      for (int n = 0; n < 16; ++n) {
        uint32_t v = 0;
        for (int j = 0; j < 4; ++j)
          if (n & (1 << j)) v ^= bit[j];
        out.t[(16 * k + n) * 32 + l] = v;
      }
    }
  }
  return out;
}
__device__ const LaneMulTable g_lane_mul = make_lane_mul_table();

// a * M_l mod P for the calling lane l; `LM` is the shared copy of the table
// offset by the lane.
__device__ __forceinline__ uint32_t lane_mul(const uint32_t* LM, uint32_t a) {
  uint32_t r[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) r[k] = LM[(16 * k + ((a >> (4 * k)) & 15u)) * 32];
  return (r[0] ^ r[1] ^ r[2]) ^ (r[3] ^ r[4] ^ r[5]) ^ (r[6] ^ r[7]);
}

// CRC-32C of the 60 header bytes given as 15 words: word k (followed by
// 14 - k more) sits in lane 17 + k, whose multiplier M_(17+k) = x^(32 (15 - k))
// is exactly its shift; every lane returns it.
__device__ __forceinline__ uint32_t header_crc(const uint32_t* LM, const uint32_t h[15], uint32_t lane) {
  uint32_t w = 0;
#pragma unroll
  for (int k = 0; k < 15; ++k) w = (lane == static_cast<uint32_t>(17 + k)) ? h[k] : w;
  constexpr uint32_t kHeaderXor = gf_mulmod(0xFFFFFFFFu, gf_xpow(8 * 60)) ^ 0xFFFFFFFFu;
  return __reduce_xor_sync(kFull, lane_mul(LM, w)) ^ kHeaderXor;
}

// a * b mod P, both variable.
__device__ __forceinline__ uint32_t gmul(uint32_t a, uint32_t b) {
  uint32_t r = 0;
#pragma unroll 8
  for (int k = 0; k < 32; ++k) {
    r ^= b & static_cast<uint32_t>(static_cast<int32_t>(a << k) >> 31);
    b = (b >> 1) ^ (kPoly & (0u - (b & 1u)));
  }
  return r;
}

// x^(8n) mod P for n < 2^48, from per-byte power tables.
__device__ uint32_t xpow8(uint64_t n) {
  uint32_t r = kOne;
  for (int k = 0; k < kPowBytes; ++k) {
    const uint32_t byte = static_cast<uint32_t>(n >> (8 * k)) & 255u;
    if (byte) r = gmul(r, __ldg(&g_pow.p[k][byte]));
  }
  return r;
}

__device__ __forceinline__ uint32_t shift_bytes(uint32_t raw, uint64_t n) {
  return n ? gmul(raw, xpow8(n)) : raw;
}

// (hi, lo) += (bh, bl) as unevaluated float pairs: TwoSum of the high parts,
// the low parts and the rounding error added in fp32.
__device__ __forceinline__ void two_sum_pair(float& hi, float& lo, float bh, float bl) {
  const float t = hi + bh;
  const float z = t - hi;
  const float err = (hi - (t - z)) + (bh - z);
  lo = (lo + bl) + err;
  hi = t;
}

// One tail element, given as an fp32 bit pattern `f` (a bf16 element in the
// high half): counted in nf if non-finite; its square added exactly to the
// float pair (hi, lo) -- the fp32 product and its FMA residual, by TwoSum --
// when |x| is 0 or lies in [2^-40, 2^56] (the residual is not subnormal, and
// a lane's 8 squares add at most 2^115); any other finite value sets `odd`,
// and the caller adds it in fp64 (rare).  No branch: the common case stays
// off GB300's narrow fp64 pipe and the warp does not diverge.
__device__ __forceinline__ void tail_elem(uint32_t f, uint32_t& nf, float& hi, float& lo, bool& odd) {
  const bool nonfinite = (f & 0x7F800000u) == 0x7F800000u;
  const float ax = fabsf(__uint_as_float(f));
  const bool fast = ax == 0.0f || (ax >= 0x1p-40f && ax <= 0x1p56f);  // false for NaN and Inf
  nf += nonfinite ? 1u : 0u;
  odd |= !fast && !nonfinite;
  const float x = fast ? __uint_as_float(f) : 0.0f;
  const float p2 = x * x;
  two_sum_pair(hi, lo, p2, __fmaf_rn(x, x, -p2));
}

// The fp64 share of a tail element that tail_elem left out (0 for the rest).
__device__ __forceinline__ double tail_elem_odd(uint32_t f) {
  const float ax = fabsf(__uint_as_float(f));
  const bool fast = ax == 0.0f || (ax >= 0x1p-40f && ax <= 0x1p56f);
  if (fast || (f & 0x7F800000u) == 0x7F800000u) return 0.0;
  const double d = static_cast<double>(__uint_as_float(f));
  return __dmul_rn(d, d);
}

// Adds a pair-form segment slot (see seg_value) whose sum is below 2^90 to
// the float pair (hi, lo); any other slot (tagged fp64 form, or 2^90 or more,
// both rare) sets `odd`, and the caller adds it in fp64.  A lane's float pair
// then stays below 2^119 for any chunk of fewer than 2^47 bytes, tail squares
// included, and the 32-lane tree cannot overflow.
__device__ __forceinline__ bool slot_fast(uint64_t bits) {
  return !(bits >> 63) && __uint_as_float(static_cast<uint32_t>(bits >> 32)) < 0x1p90f;
}
__device__ __forceinline__ void add_slot(uint64_t bits, float& hi, float& lo, bool& odd) {
  const bool fast = slot_fast(bits);
  odd |= !fast;
  two_sum_pair(hi, lo, fast ? __uint_as_float(static_cast<uint32_t>(bits >> 32)) : 0.0f,
               fast ? __uint_as_float(static_cast<uint32_t>(bits)) : 0.0f);
}
__device__ __forceinline__ double slot_odd(uint64_t bits) {
  if (slot_fast(bits)) return 0.0;
  if (bits >> 63) return -__longlong_as_double(static_cast<long long>(bits));
  return static_cast<double>(__uint_as_float(static_cast<uint32_t>(bits >> 32))) +
         static_cast<double>(__uint_as_float(static_cast<uint32_t>(bits)));
}

__device__ __forceinline__ void prefetch_l1(const void* q) { asm volatile("prefetch.global.L1 [%0];" ::"l"(q)); }

template <int MODE>
__global__ void __launch_bounds__(kFinThreads, FR_FIN_MINB) finalize_kernel(FinalizeParams p) {
  __shared__ LaneMulTable lm_s;
  {
    const uint4* src = reinterpret_cast<const uint4*>(g_lane_mul.t);
    uint4* dst = reinterpret_cast<uint4*>(lm_s.t);
#pragma unroll
    for (int i = 0; i < kLaneMulWords / 4 / kFinThreads; ++i) dst[threadIdx.x + i * kFinThreads] = src[threadIdx.x + i * kFinThreads];
  }
  __syncthreads();
  const uint32_t lane = threadIdx.x & 31u;
  const uint32_t* LM = lm_s.t + lane;
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * kFinWarps;
  for (uint64_t pos = p.c_begin + static_cast<uint64_t>(blockIdx.x) * kFinWarps + (threadIdx.x >> 5);
       pos < p.c_end; pos += stride) {
    const uint64_t c = p.ids ? p.ids[pos] : pos;
    // the warp's next descriptor streams into L1 while this chunk is done
    if (!p.ids && lane == 0 && pos + stride < p.c_end) prefetch_l1(p.chunks + pos + stride);
    const ChunkDesc cd = p.chunks[c];
    const uint64_t body = cd.len & ~static_cast<uint64_t>(kBlockBytes - 1);
    const uint32_t tail = static_cast<uint32_t>(cd.len - body);
    const bool values = mode_sums(MODE) && (cd.dtype != kDtBytes);
    // list mode: one record per chunk with a body, at the list position
    const uint64_t first_rec = p.ids ? pos : cd.first_rec;
    const int64_t n_recs = p.ids ? (body ? 1 : 0) : cd.n_recs;
    const uint64_t n_seg = (body / kBlockBytes + kSegBlocks - 1) / kSegBlocks;  // (read only with values)
    const bool rec_mul = p.rec_mul && !p.ids;

    // ---- 0. every load the chunk needs (records, segment sums, tail bytes,
    // preset term, header and padding) is issued here, before any is used, so
    // a chunk costs one memory latency after its descriptor
    Record rec0{0u, 0u, 0.0};
    uint32_t mul0 = 0;
    if (rec_mul && lane < n_recs) {
      rec0 = p.recs[first_rec + lane];
      mul0 = p.rec_mul[first_rec + lane];
    }
    uint64_t slot0 = 0;
    if (values && lane < n_seg) slot0 = reinterpret_cast<const uint64_t*>(p.segs + cd.seg_base)[lane];
    const uint8_t* tsrc;
    uint8_t* tdst = nullptr;
    if (mode_unpacks(MODE)) {
      tsrc = p.packed + cd.payload_off + body;
      tdst = reinterpret_cast<uint8_t*>(cd.addr) + body;
    } else {
      tsrc = reinterpret_cast<const uint8_t*>(cd.addr) + body;
      if (MODE == kModePack) tdst = p.packed + cd.payload_off + body;
    }
    // The tail is read as the end of a 512-byte window whose first z = 512 -
    // tail bytes are zeros (leading zero bytes leave a raw CRC run from zero
    // unchanged and add nothing to the sums).  Window word i (bytes 4i..4i+3,
    // little-endian) is word i / 32 of lane i % 32, so one load instruction
    // covers 32 consecutive words.  Words are loaded whole when the tail's
    // end is 4-byte aligned on both sides (a word holding the tail's first
    // byte then goes byte by byte), else every word byte by byte.
    const int32_t z = kBlockBytes - static_cast<int32_t>(tail);
    const bool wordy = ((reinterpret_cast<uintptr_t>(tsrc) + tail) & 3u) == 0 &&
                       (tdst == nullptr || ((reinterpret_cast<uintptr_t>(tdst) + tail) & 3u) == 0);
    uint32_t w[4] = {0u, 0u, 0u, 0u};
    if (tail != 0) {
      if (wordy) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int32_t t = 4 * (32 * q + static_cast<int32_t>(lane)) - z;  // the word's offset in the tail
          if (t >= 0) w[q] = __ldg(reinterpret_cast<const uint32_t*>(tsrc + t));
        }
      }
      if (!wordy || (tail & 3u) != 0) {  // byte by byte: every word, or the partial first one
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int32_t t = 4 * (32 * q + static_cast<int32_t>(lane)) - z;
          if (t > -4 && (!wordy || t < 0)) {
#pragma unroll
            for (int j = 0; j < 4; ++j)
              if (t + j >= 0) w[q] |= static_cast<uint32_t>(__ldg(tsrc + (t + j))) << (8 * j);
          }
        }
      }
    }
    const uint32_t crc_xor = p.crc_xor ? p.crc_xor[c] : 0u;
    // padding after the payload: [pad_begin, pad_end), pad_end 256-aligned,
    // covered as whole words from pad_begin rounded down to 4 bytes
    const uint64_t pad_begin = cd.payload_off + cd.len;
    const uint64_t pad_end = cd.payload_off + align_up(cd.len, kPayloadAlign);
    const uint64_t pad_w0 = pad_begin & ~static_cast<uint64_t>(3);
    uint32_t h[16];
    uint32_t pad = 0;  // OR of the padding bytes after the payload (< 256 of them)
    if (mode_unpacks(MODE)) {
      const uint4* src = reinterpret_cast<const uint4*>(p.packed + c * kHeaderBytes);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 v = src[q];
        h[4 * q] = v.x;
        h[4 * q + 1] = v.y;
        h[4 * q + 2] = v.z;
        h[4 * q + 3] = v.w;
      }
      const uint32_t* pw = reinterpret_cast<const uint32_t*>(p.packed + pad_w0);
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        const uint32_t k = lane + 32u * q;
        if (pad_w0 + 4u * k < pad_end) {
          uint32_t v = pw[k];
          if (k == 0) v &= 0xFFFFFFFFu << (8 * (pad_begin & 3u));  // payload bytes before pad_begin
          pad |= v;
        }
      }
    }
    // pack and unpack copy the tail (before the body's CRC is folded into it)
    if (tdst != nullptr && tail != 0) {
      if (wordy) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int32_t t = 4 * (32 * q + static_cast<int32_t>(lane)) - z;
          if (t >= 0) *reinterpret_cast<uint32_t*>(tdst + t) = w[q];
        }
      }
      if (!wordy || (tail & 3u) != 0) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int32_t t = 4 * (32 * q + static_cast<int32_t>(lane)) - z;
          if (t > -4 && (!wordy || t < 0)) {
#pragma unroll
            for (int j = 0; j < 4; ++j)
              if (t + j >= 0) tdst[t + j] = static_cast<uint8_t>(w[q] >> (8 * j));
          }
        }
      }
    }

    // ---- 1. records: each shifted by the bytes after it in the chunk's body
    // -- a multiplier the plan precomputed (1 for the last record, whose
    // multiply is skipped), or (list mode, no-allocation entry) found here,
    // last batch of 32 first so the byte count after each is known
    uint32_t raw = 0;      // this lane's share of the body's raw CRC
    uint32_t nf_lane = 0;  // this lane's share of the non-finite count
    uint64_t carry = 0;
    if (rec_mul) {
      raw = rec0.crc;  // zero past the chunk's records
      nf_lane = rec0.nonfinite;
      const bool shift = lane < n_recs && mul0 != kOne;
      if (__any_sync(kFull, shift)) {
        const uint32_t r = gmul(rec0.crc, mul0);
        if (shift) raw = r;
      }
      for (int64_t i = lane + 32; i < n_recs; i += 32) {
        const Record rec = p.recs[first_rec + i];
        raw ^= gmul(rec.crc, p.rec_mul[first_rec + i]);
        nf_lane += rec.nonfinite;
      }
    }
    for (int64_t hi = rec_mul ? 0 : n_recs; hi > 0;) {
      const int64_t lo = hi > 32 ? hi - 32 : 0;
      const int64_t i = lo + lane;
      const bool have = i < hi;
      Record rec{0u, 0u, 0.0};
      uint64_t len = 0;
      if (have) {
        rec = p.recs[first_rec + i];
        len = p.ids ? body : p.rec_nblk[first_rec + i] * kBlockBytes;
      }
      uint64_t suf = len;  // bytes of this record and the later ones in the batch
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const uint64_t t = __shfl_down_sync(kFull, suf, d);
        if (lane + d < 32) suf += t;
      }
      if (have) raw ^= shift_bytes(rec.crc, carry + suf - len);
      carry += __shfl_sync(kFull, suf, 0);
      nf_lane += rec.nonfinite;
      hi = lo;
    }
    // the body's raw CRC, in every lane
    raw = __reduce_xor_sync(kFull, raw);

    // ---- 2. sums of squares: each lane adds its segment slots (in an order
    // fixed by segment index, so the result does not depend on the plan),
    // then its tail elements, as a float pair (pair-form slots and tail
    // squares by TwoSum; tagged fp64 slots and out-of-range squares, both
    // rare, in fp64), and one fixed tree adds the lanes: the common case
    // stays off the narrow fp64 pipe
    double sq = 0.0;
    if (values) {
      float hi = 0.0f, lo = 0.0f;
      bool odd = false;
      const uint64_t* seg_slots = reinterpret_cast<const uint64_t*>(p.segs + cd.seg_base);
      add_slot(slot0, hi, lo, odd);  // zero past the body's segments
      for (uint64_t k = lane + 32; k < n_seg; k += 32) add_slot(seg_slots[k], hi, lo, odd);
      const bool f32 = cd.dtype == kDtF32;
      if (tail != 0) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if (f32) {
            tail_elem(w[q], nf_lane, hi, lo, odd);
          } else {
            tail_elem(w[q] << 16, nf_lane, hi, lo, odd);
            tail_elem(w[q] & 0xFFFF0000u, nf_lane, hi, lo, odd);
          }
        }
      }
      double dx = 0.0;  // the values left out of the float pairs, in fp64 (rare)
      if (__any_sync(kFull, odd)) {
        if (odd) {
          dx = slot_odd(slot0);
          for (uint64_t k = lane + 32; k < n_seg; k += 32) dx += slot_odd(seg_slots[k]);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            if (f32) {
              dx += tail_elem_odd(w[q]);
            } else {
              dx += tail_elem_odd(w[q] << 16);
              dx += tail_elem_odd(w[q] & 0xFFFF0000u);
            }
          }
        }
#pragma unroll
        for (int m = 16; m >= 1; m >>= 1) dx += __shfl_down_sync(kFull, dx, m);
      }
      // lanes at or past `active` hold zeros: tree levels that would only add
      // them are skipped (adding (0, 0) changes no bit of the pair)
      const uint64_t active = tail != 0 ? 32u : n_seg;
#pragma unroll
      for (int m = 16; m >= 1; m >>= 1) {
        if (static_cast<uint64_t>(m) < active) {
          const float oh = __shfl_down_sync(kFull, hi, m), ol = __shfl_down_sync(kFull, lo, m);
          two_sum_pair(hi, lo, oh, ol);
        }
      }
      sq = (static_cast<double>(hi) + static_cast<double>(lo)) + dx;
    }

    // ---- 3. the tail's CRC, continuing the body's: a run started from state
    // r equals one started from zero with r XORed into its first four bytes,
    // so when the tail's first byte starts a window word (tail length a
    // multiple of 4: always for fp32) the body's raw CRC is XORed into that
    // word and the window's raw CRC is raw(body || tail) with no shift of the
    // body; other tails (byte tensors, some bf16) shift the body by
    // x^(8 tail).  Lane l's words w_q (window words 32q + l) combine as
    // sum_q w_q x^(1024 (3 - q)) (two multiplies by x^1024 and one by
    // x^2048), then take the lane's shift M_l, and the lanes are XORed.
    if (tail != 0) {
      const bool fold = (tail & 3u) == 0;
      if (fold) {
        const uint32_t i0 = static_cast<uint32_t>(z) >> 2;  // the window word holding the tail's first byte
        const uint32_t fx = lane == (i0 & 31u) ? raw : 0u;
        w[0] ^= (i0 >> 5) == 0 ? fx : 0u;
        w[1] ^= (i0 >> 5) == 1 ? fx : 0u;
        w[2] ^= (i0 >> 5) == 2 ? fx : 0u;
        w[3] ^= (i0 >> 5) == 3 ? fx : 0u;
      }
      const uint32_t H = mul_const(g_x2048, mul_const(g_x1024, w[0]) ^ w[1]) ^ (mul_const(g_x1024, w[2]) ^ w[3]);
      const uint32_t joined = __reduce_xor_sync(kFull, lane_mul(LM, H));
      raw = (fold || raw == 0) ? joined : (shift_bytes(raw, tail) ^ joined);
    }

    // ---- 4. preset and final XOR
    const uint32_t crc = raw ^ (p.crc_xor ? crc_xor : (shift_bytes(0xFFFFFFFFu, cd.len) ^ 0xFFFFFFFFu));
    // lane 0 holds the fixed-order sums; every lane gets them and the count
    const double sumsq = __shfl_sync(kFull, sq, 0);
    const uint32_t nonfinite = __reduce_add_sync(kFull, nf_lane);

    const uint64_t table_end = p.n_chunks * kHeaderBytes;
    const uint64_t gap_end = align_up(table_end, kPayloadAlign);
    const bool last = (c + 1 == p.n_chunks);

    // ---- 5. outputs
    if (MODE != kModeUnpack && p.out_fp != nullptr) {  // the fingerprint table (optional for pack, unpack-fp)
      if (lane == 0) {
        FpEntry e;
        e.crc32c = crc;
        e.nonfinite = nonfinite;
        e.sumsq = sumsq;
        p.out_fp[c] = e;
      }
    }
    if (MODE == kModePack) {
      {
        uint32_t hd[15];
        const uint64_t sbits = static_cast<uint64_t>(__double_as_longlong(sumsq));
        hd[0] = kMagic;
        hd[1] = kVersion | (cd.dtype << 16);
        hd[2] = static_cast<uint32_t>(c);
        hd[3] = static_cast<uint32_t>(c >> 32);
        hd[4] = cd.tensor_idx;
        hd[5] = crc;
        hd[6] = static_cast<uint32_t>(cd.tensor_off);
        hd[7] = static_cast<uint32_t>(cd.tensor_off >> 32);
        hd[8] = static_cast<uint32_t>(cd.len);
        hd[9] = static_cast<uint32_t>(cd.len >> 32);
        hd[10] = static_cast<uint32_t>(cd.payload_off);
        hd[11] = static_cast<uint32_t>(cd.payload_off >> 32);
        hd[12] = static_cast<uint32_t>(sbits);
        hd[13] = static_cast<uint32_t>(sbits >> 32);
        hd[14] = nonfinite;
        const uint32_t hcrc = header_crc(LM, hd, lane);
        if (lane == 0) {
          uint4* dst = reinterpret_cast<uint4*>(p.packed + c * kHeaderBytes);
          for (int q = 0; q < 3; ++q) dst[q] = make_uint4(hd[4 * q], hd[4 * q + 1], hd[4 * q + 2], hd[4 * q + 3]);
          dst[3] = make_uint4(hd[12], hd[13], hd[14], hcrc);
        }
      }
      // zero padding: the bytes up to the first word boundary one by one,
      // then whole words
      const uint64_t pad_w1 = (pad_begin + 3) & ~static_cast<uint64_t>(3);
      if (pad_begin + lane < pad_w1 && pad_begin + lane < pad_end) p.packed[pad_begin + lane] = 0;
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const uint64_t j = pad_w1 + 4u * (lane + 32u * q);
        if (j < pad_end) *reinterpret_cast<uint32_t*>(p.packed + j) = 0u;
      }
      if (last)
        for (uint64_t j = table_end + lane * 16u; j < gap_end; j += 512)
          *reinterpret_cast<uint4*>(p.packed + j) = make_uint4(0, 0, 0, 0);
    } else if (mode_unpacks(MODE)) {  // unpack + verify
      // every lane read the (same) header; check it against the plan
      const uint32_t hcrc = header_crc(LM, h, lane);
      bool bad = (h[15] != hcrc) || h[0] != kMagic || (h[1] & 0xFFFFu) != kVersion || (h[1] >> 16) != cd.dtype ||
                 h[2] != static_cast<uint32_t>(c) || h[3] != static_cast<uint32_t>(c >> 32) ||
                 h[4] != cd.tensor_idx || h[6] != static_cast<uint32_t>(cd.tensor_off) ||
                 h[7] != static_cast<uint32_t>(cd.tensor_off >> 32) || h[8] != static_cast<uint32_t>(cd.len) ||
                 h[9] != static_cast<uint32_t>(cd.len >> 32) || h[10] != static_cast<uint32_t>(cd.payload_off) ||
                 h[11] != static_cast<uint32_t>(cd.payload_off >> 32) || h[5] != crc;
      if (pad != 0) bad = true;
      if (last)
        for (uint64_t j = table_end + lane; j < gap_end; j += 32)
          if (p.packed[j] != 0) bad = true;
      bad = __any_sync(kFull, bad);
      if (lane == 0) p.flags[c] = bad ? 1 : 0;
    }
  }
}

// ------------------------------------------------------------------ compaction

constexpr int kCompactThreads = 1024;
constexpr int kPerThread = 8;
constexpr int kTile = kCompactThreads * kPerThread;

// Bulk prefetch of [p, p + bytes) into L2 (bytes rounded down to 16).
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint64_t bytes) {
  const uint32_t b = static_cast<uint32_t>(bytes) & ~15u;
  if (b) asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(b) : "memory");
}

struct FlagPred {
  const uint8_t* flags;
  __device__ __forceinline__ bool operator()(uint64_t i) const { return flags[i] != 0; }
  __device__ __forceinline__ void prefetch(uint64_t first, uint64_t count) const {
    prefetch_l2_bulk(flags + first, count);
  }
};

struct DiffPred {
  const uint4* a;
  const uint4* b;
  __device__ __forceinline__ bool operator()(uint64_t i) const {
    const uint4 x = a[i], y = b[i];
    return ((x.x ^ y.x) | (x.y ^ y.y) | (x.z ^ y.z) | (x.w ^ y.w)) != 0u;
  }
  __device__ __forceinline__ void prefetch(uint64_t first, uint64_t count) const {
    prefetch_l2_bulk(a + first, count * 16);
    prefetch_l2_bulk(b + first, count * 16);
  }
};

// One CTA walks the index space in tiles of kTile.  Warp w tests the 256
// indices [tile + 256w, tile + 256w + 256) in kPerThread rounds, lane l taking
// index 32j + l in round j, so every load of a round is coalesced; the ballots
// of the rounds give each hit its rank inside the warp, a block-wide scan of
// the warp totals gives the warp's output position, and the ids are written in
// ascending order.  Deterministic: no atomics decide any position.
template <class Pred>
__global__ void __launch_bounds__(kCompactThreads) compact_kernel(Pred pred, uint64_t n, uint32_t* out,
                                                                  uint64_t cap, uint64_t* count,
                                                                  uint32_t* status) {
  __shared__ uint32_t warp_tot[kCompactThreads / 32];
  __shared__ uint64_t base_sh;
  const uint32_t tid = threadIdx.x, lane = tid & 31u, warp = tid >> 5;
  const uint32_t lt = (1u << lane) - 1u;  // lanes below this one
  uint64_t base = 0;
  if (tid == 0) pred.prefetch(0, n < kTile ? n : kTile);
  for (uint64_t t0 = 0; t0 < n; t0 += kTile) {
    // the next tile streams into L2 while this one is tested
    if (tid == 0 && t0 + kTile < n) pred.prefetch(t0 + kTile, n - (t0 + kTile) < kTile ? n - (t0 + kTile) : kTile);
    const uint64_t wbase = t0 + static_cast<uint64_t>(warp) * (32 * kPerThread);
    uint32_t mask[kPerThread];
    uint32_t total = 0;
    // branch-free, so all rounds' loads can be in flight at once (indices
    // past the end test entry 0 and are masked off)
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      const uint64_t i = wbase + 32u * j + lane;
      const bool in = i < n;
      const bool hit = pred(in ? i : 0);
      mask[j] = __ballot_sync(kFull, in && hit);
      total += __popc(mask[j]);
    }
    if (lane == 0) warp_tot[warp] = total;
    __syncthreads();
    if (warp == 0) {
      uint32_t w = warp_tot[lane];
      uint32_t winc = w;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const uint32_t v = __shfl_up_sync(kFull, winc, d);
        if (lane >= static_cast<uint32_t>(d)) winc += v;
      }
      warp_tot[lane] = winc - w;  // exclusive prefix of warp totals
      if (lane == 31) base_sh = base + winc;
    }
    __syncthreads();
    uint64_t pos = base + warp_tot[warp];
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      if ((mask[j] >> lane) & 1u) {
        const uint64_t q = pos + __popc(mask[j] & lt);
        if (q < cap) out[q] = static_cast<uint32_t>(wbase + 32u * j + lane);
      }
      pos += __popc(mask[j]);
    }
    base = base_sh;
    __syncthreads();
  }
  if (tid == 0) {
    *count = base;
    if (base > cap && status != nullptr) atomicOr(status, kStatusCapacity);
  }
}

// The same compaction over a cluster of kCompactCluster CTAs for more than
// one tile: in round r, CTA k tests tile r * kCompactCluster + k exactly as
// above, publishes its hit count in its shared memory, and after a cluster
// barrier reads the other CTAs' counts through distributed shared memory to
// place its ids after those of the lower tiles.  A second barrier per round
// keeps a count from being overwritten before every CTA has read it.  Every
// CTA runs the same number of rounds and reaches every barrier; no global
// scratch, no atomics deciding positions.
constexpr int kCompactCluster = 8;

template <class Pred>
__global__ void __cluster_dims__(kCompactCluster, 1, 1) __launch_bounds__(kCompactThreads)
    compact_cluster_kernel(Pred pred, uint64_t n, uint32_t* out, uint64_t cap, uint64_t* count, uint32_t* status) {
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  __shared__ uint32_t warp_tot[kCompactThreads / 32];
  __shared__ uint32_t tile_tot;     // this CTA's hits this round, read by the whole cluster
  __shared__ uint64_t round_first;  // this CTA's first output position this round
  __shared__ uint64_t round_hits;   // the cluster's hits this round
  const uint32_t rank = cluster.block_rank();
  const uint32_t tid = threadIdx.x, lane = tid & 31u, warp = tid >> 5;
  const uint32_t lt = (1u << lane) - 1u;
  const uint64_t n_tiles = (n + kTile - 1) / kTile;
  const uint64_t rounds = (n_tiles + kCompactCluster - 1) / kCompactCluster;
  constexpr uint64_t kStride = static_cast<uint64_t>(kCompactCluster) * kTile;
  uint64_t base = 0;
  if (tid == 0 && static_cast<uint64_t>(rank) * kTile < n) {
    const uint64_t t0 = static_cast<uint64_t>(rank) * kTile;
    pred.prefetch(t0, n - t0 < kTile ? n - t0 : kTile);
  }
  for (uint64_t r = 0; r < rounds; ++r) {
    const uint64_t t0 = r * kStride + static_cast<uint64_t>(rank) * kTile;  // may lie past n: no hits
    if (tid == 0 && t0 + kStride < n) pred.prefetch(t0 + kStride, n - (t0 + kStride) < kTile ? n - (t0 + kStride) : kTile);
    const uint64_t wbase = t0 + static_cast<uint64_t>(warp) * (32 * kPerThread);
    uint32_t mask[kPerThread];
    uint32_t total = 0;
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      const uint64_t i = wbase + 32u * j + lane;
      const bool in = i < n;
      const bool hit = pred(in ? i : 0);
      mask[j] = __ballot_sync(kFull, in && hit);
      total += __popc(mask[j]);
    }
    if (lane == 0) warp_tot[warp] = total;
    __syncthreads();
    if (warp == 0) {
      const uint32_t w = warp_tot[lane];
      uint32_t winc = w;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const uint32_t v = __shfl_up_sync(kFull, winc, d);
        if (lane >= static_cast<uint32_t>(d)) winc += v;
      }
      warp_tot[lane] = winc - w;  // exclusive prefix of warp totals
      if (lane == 31) tile_tot = winc;
    }
    cluster.sync();  // every CTA's tile_tot is written and visible
    if (tid == 0) {
      uint64_t before = 0, hits = 0;
      for (uint32_t k = 0; k < static_cast<uint32_t>(kCompactCluster); ++k) {
        const uint32_t v = *cluster.map_shared_rank(&tile_tot, k);
        if (k < rank) before += v;
        hits += v;
      }
      round_first = base + before;
      round_hits = hits;
    }
    __syncthreads();
    uint64_t pos = round_first + warp_tot[warp];
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      if ((mask[j] >> lane) & 1u) {
        const uint64_t q = pos + __popc(mask[j] & lt);
        if (q < cap) out[q] = static_cast<uint32_t>(wbase + 32u * j + lane);
      }
      pos += __popc(mask[j]);
    }
    base += round_hits;
    cluster.sync();  // every CTA has read the tile counts and round_hits
  }
  if (rank == 0 && tid == 0) {
    *count = base;
    if (base > cap && status != nullptr) atomicOr(status, kStatusCapacity);
  }
}

template <class Pred>
cudaError_t launch_compact(const Pred& pred, uint64_t n, uint32_t* out, uint64_t cap, uint64_t* count,
                           uint32_t* status, cudaStream_t s) {
  if (n > static_cast<uint64_t>(kTile))
    compact_cluster_kernel<Pred><<<kCompactCluster, kCompactThreads, 0, s>>>(pred, n, out, cap, count, status);
  else
    compact_kernel<Pred><<<1, kCompactThreads, 0, s>>>(pred, n, out, cap, count, status);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_finalize(int mode, const FinalizeParams& p, cudaStream_t s) {
  if (p.c_end <= p.c_begin) return cudaSuccess;
  // every CTA copies the 16 KiB multiplier table into shared memory, so the
  // grid is at most one full wave (FR_FIN_MINB CTAs per SM), its warps
  // looping over the chunks
  int dev = 0, n_sm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const uint64_t cap = static_cast<uint64_t>(n_sm > 0 ? n_sm : 1) * FR_FIN_MINB;
  const uint64_t want = (p.c_end - p.c_begin + kFinWarps - 1) / kFinWarps;
  const int grid = static_cast<int>(want < cap ? want : cap);
  if (mode == kModeFingerprint)
    finalize_kernel<kModeFingerprint><<<grid, kFinThreads, 0, s>>>(p);
  else if (mode == kModePack)
    finalize_kernel<kModePack><<<grid, kFinThreads, 0, s>>>(p);
  else if (mode == kModeUnpackFp)
    finalize_kernel<kModeUnpackFp><<<grid, kFinThreads, 0, s>>>(p);
  else
    finalize_kernel<kModeUnpack><<<grid, kFinThreads, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_compact_flags(const uint8_t* flags, uint64_t n, uint32_t* out, uint64_t cap,
                                 uint64_t* count, uint32_t* status, cudaStream_t s) {
  return launch_compact(FlagPred{flags}, n, out, cap, count, status, s);
}

cudaError_t launch_diff(const FpEntry* a, const FpEntry* b, uint64_t n, uint32_t* out, uint64_t cap,
                        uint64_t* count, cudaStream_t s) {
  DiffPred pred{reinterpret_cast<const uint4*>(a), reinterpret_cast<const uint4*>(b)};
  return launch_compact(pred, n, out, cap, count, nullptr, s);
}

}  // namespace frk
