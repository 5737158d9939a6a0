// sweep_impl.cuh -- the bandwidth-bound body sweep of fingerprint / pack / unpack.
//
// Restoration of a rank's state from a data-parallel replica (FlashRecovery,
// arXiv 2509.03047, Sec. III-E) is, on one GPU, a sweep over every byte of
// the param / master / Adam-m / Adam-v tensors: checksum it, and for the
// transfer copy it into (pack) or out of (unpack) a flat buffer.  This kernel
// does the whole-512-byte-block part of every chunk in one HBM pass:
//
//  * copy engine: each lane moves 16 bytes per block with a coalesced 128-bit
//    load and (pack/unpack) a coalesced 128-bit store;
//  * CRC-32C: the 128 words of a block are 128 interleaved CRC streams
//    (lane l owns streams 4l..4l+3, four independent dependency chains), each
//    advanced by s <- (s ^ w) * x^4096 with four byte lookups in tables kept in
//    shared memory.  Every lane has a private copy of each table entry in its
//    own bank, so the 32 lookups of a warp never conflict.  At the end of a
//    piece the streams are folded with GF(2) multiplications by constants and
//    warp shuffles into the raw CRC of the piece;
//  * non-finite count and sum of squares, fused on the same registers: each
//    square is added to a packed f32x2 running sum by one FMA, and the
//    addition's error -- including the square's own rounding for fp32 -- is
//    recovered to second order by a TwoSum whose low term is a second FMA
//    (two_sum_sq), then flushed into fp64.  A 16 KiB segment whose running
//    sum is not finite (NaN/Inf input, or overflow) or is tiny with non-zero
//    input is redone element by element, exactly, from a reload of its
//    16-byte units (slow_span), so the fast path never needs a per-element
//    test.
//
// No tensor cores: nothing here is a contraction.  One CTA per SM, with a warp
// count per mode (the 128 KiB of lane-replicated tables fill most of shared
// memory).  The plan sorts chunks into classes by element type and by whether
// the tensor is 16-byte aligned; each class has its own block stream, cut
// into per-warp ranges, and its own code specialization, so each warp runs a
// single loop variant.  A call launches once for all its classes
// (sweep_mixed_kernel: each warp dispatches on its range's class once);
// pack and unpack warps then claim the last few percent of the work as small
// units (see sweep_warp_claims).  sweep_{fp,pack,unpack,unpack_fp}.cu each
// instantiate one mode.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "gf2.cuh"
#include "kernels.h"
#include "layout.h"

namespace frk {

namespace {

// Warps and threads of one mode's CTA.
template <int MODE>
struct Cta {
  static constexpr int kWarps = sweep_warps(MODE);
  static constexpr int kThreads = kWarps * 32;
};
constexpr int kTableBytes = 4 * 256 * 32 * 4;  // 4 tables x 256 entries x 32 lanes x 4 B
// Pipeline geometry (compile-time), tuned on GB300 by timing the 31.8 GB
// Llama-70B shard.  The read-only fingerprint gains from bulk L2 prefetch
// exactly one span ahead (none: -9 points; two spans: -25) and from 8-block
// register stages; pack and unpack lose by the prefetch (their write stream
// evicts the prefetched lines before use, and DRAM reads grow by ~20%), so
// they rely on 4-block register stages and more warps (kernels.h).
#ifndef FR_STAGE_FP
#define FR_STAGE_FP 8
#endif
#ifndef FR_STAGE_PACK
#define FR_STAGE_PACK 4
#endif
#ifndef FR_STAGE_UNPACK
#define FR_STAGE_UNPACK 4
#endif
#ifndef FR_AHEAD_FP
#define FR_AHEAD_FP 1
#endif
#ifndef FR_AHEAD_PACK
#define FR_AHEAD_PACK 0
#endif
#ifndef FR_AHEAD_UNPACK
#define FR_AHEAD_UNPACK 0
#endif
#ifndef FR_LOADFIRST_FP
#define FR_LOADFIRST_FP 0
#endif
#ifndef FR_LOADFIRST_PACK
#define FR_LOADFIRST_PACK 0
#endif
#ifndef FR_LOADFIRST_UNPACK
#define FR_LOADFIRST_UNPACK 1
#endif
// Blocks per validity span: one sum segment (a power of two, a multiple of
// every stage).
constexpr int kSpan = static_cast<int>(kSegBlocks);

typedef unsigned long long u64;

__device__ const ByteTables4 g_braid = make_mul_tables(kBraidMul);

extern __shared__ __align__(16) uint8_t g_smem[];

// ------------------------------------------------------------------ tables

// Table k, entry i, lane l lives at byte
//   (k >> 1) * 65536 + i * 256 + (k & 1) * 128 + l * 4,
// i.e. bank l.  The address of (table k, byte k of x, this lane) is one
// byte-permute: byte 0 = l*4, byte 1 = byte k of x.
// Every thread of a kThreads-thread CTA stores its share of 16-byte units;
// the loop is unrolled so a thread's table loads all issue before the first
// store waits on one (a rolled loop made the fill a chain of ~16 L2 round
// trips, about 3 us per launch).
template <int kThreads>
__device__ __forceinline__ void fill_tables() {
  constexpr int kUnits = kTableBytes / 16;
  constexpr int kIters = (kUnits + kThreads - 1) / kThreads;
  uint32_t v[kIters];
#pragma unroll
  for (int it = 0; it < kIters; ++it) {
    const int q = static_cast<int>(threadIdx.x) + it * kThreads;
    const int k = q >> 11, i = (q & 2047) >> 3;
    v[it] = q < kUnits ? g_braid.t[k][i] : 0u;
  }
#pragma unroll
  for (int it = 0; it < kIters; ++it) {
    const int q = static_cast<int>(threadIdx.x) + it * kThreads;
    if (q < kUnits) {
      const int k = q >> 11, rem = q & 2047, i = rem >> 3, g = rem & 7;
      const uint32_t off = (k >> 1) * 65536 + i * 256 + (k & 1) * 128 + g * 16;
      *reinterpret_cast<uint4*>(g_smem + off) = make_uint4(v[it], v[it], v[it], v[it]);
    }
  }
}

__device__ __forceinline__ uint32_t tab(uint32_t off) {
  return *reinterpret_cast<const uint32_t*>(g_smem + off);
}

// (s ^ w) * x^4096 for this lane's stream, given x = s ^ w.
__device__ __forceinline__ uint32_t braid_step(uint32_t x, uint32_t lb) {
  const uint32_t t0 = tab(__byte_perm(x, lb, 0x5504));
  const uint32_t t1 = tab(__byte_perm(x, lb, 0x5514) + 128);
  const uint32_t t2 = tab(__byte_perm(x, lb, 0x5524) + 65536);
  const uint32_t t3 = tab(__byte_perm(x, lb, 0x5534) + 65536 + 128);
  return (t0 ^ t1) ^ (t2 ^ t3);
}

// The piece-end fold multiplies by seven constants: x^32 (Horner inside the
// lane), x^128 ... x^2048 (the shuffle tree) and the unbraid factor.  Each
// multiply is four byte lookups in that constant's tables (read-only, cached
// in L1) instead of a 32-step bit loop: a warp pays the fold once per piece,
// which matters for states of many small tensors.
struct FoldTables {
  ByteTables4 m[7];
};
__host__ __device__ constexpr FoldTables make_fold_tables() {
  FoldTables f{};
  f.m[0] = make_mul_tables(gf_xpow(32));
  f.m[1] = make_mul_tables(gf_xpow(128));
  f.m[2] = make_mul_tables(gf_xpow(256));
  f.m[3] = make_mul_tables(gf_xpow(512));
  f.m[4] = make_mul_tables(gf_xpow(1024));
  f.m[5] = make_mul_tables(gf_xpow(2048));
  f.m[6] = make_mul_tables(kUnbraid);
  return f;
}
__device__ const FoldTables g_fold = make_fold_tables();

// a * (constant i) mod P.
__device__ __forceinline__ uint32_t mul_fold(int i, uint32_t a) {
  const ByteTables4& T = g_fold.m[i];
  return (__ldg(&T.t[0][a & 255u]) ^ __ldg(&T.t[1][(a >> 8) & 255u])) ^
         (__ldg(&T.t[2][(a >> 16) & 255u]) ^ __ldg(&T.t[3][a >> 24]));
}

// ------------------------------------------------------------------ memory

template <int AL>
__device__ __forceinline__ uint4 ld_unit(const uint8_t* p);

template <>
__device__ __forceinline__ uint4 ld_unit<16>(const uint8_t* p) {
  uint4 v;
  asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
      : "l"(p));
  return v;
}

template <>
__device__ __forceinline__ uint4 ld_unit<4>(const uint8_t* p) {
  const uint32_t* q = reinterpret_cast<const uint32_t*>(p);
  return make_uint4(__ldg(q), __ldg(q + 1), __ldg(q + 2), __ldg(q + 3));
}

template <>
__device__ __forceinline__ uint4 ld_unit<1>(const uint8_t* p) {
  uint32_t w[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    w[j] = static_cast<uint32_t>(__ldg(p + 4 * j)) | (static_cast<uint32_t>(__ldg(p + 4 * j + 1)) << 8) |
           (static_cast<uint32_t>(__ldg(p + 4 * j + 2)) << 16) |
           (static_cast<uint32_t>(__ldg(p + 4 * j + 3)) << 24);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

template <int AL>
__device__ __forceinline__ void st_unit(uint8_t* p, uint4 v);

template <>
__device__ __forceinline__ void st_unit<16>(uint8_t* p, uint4 v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

template <>
__device__ __forceinline__ void st_unit<4>(uint8_t* p, uint4 v) {
  uint32_t* q = reinterpret_cast<uint32_t*>(p);
  __stcs(q, v.x);
  __stcs(q + 1, v.y);
  __stcs(q + 2, v.z);
  __stcs(q + 3, v.w);
}

template <>
__device__ __forceinline__ void st_unit<1>(uint8_t* p, uint4 v) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int j = 0; j < 16; ++j) p[j] = static_cast<uint8_t>(w[j >> 2] >> (8 * (j & 3)));
}

// ------------------------------------------------------------------ f32x2

__device__ __forceinline__ u64 pk(uint32_t lo, uint32_t hi) {
  u64 r;
  asm("mov.b64 %0, {%1,%2};" : "=l"(r) : "r"(lo), "r"(hi));
  return r;
}
__device__ __forceinline__ float lo_f(u64 v) { return __uint_as_float(static_cast<uint32_t>(v)); }
__device__ __forceinline__ float hi_f(u64 v) { return __uint_as_float(static_cast<uint32_t>(v >> 32)); }
__device__ __forceinline__ u64 add2(u64 a, u64 b) {
  u64 r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ u64 sub2(u64 a, u64 b) {
  u64 r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ u64 fma2(u64 a, u64 b, u64 c) {
  u64 r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}

// S + C += x*x, for each half of a packed pair (S, x >= 0 in effect: squares
// and sums of squares).  t = fl(S + x*x) by one FMA; then zn = fl(S - t),
// y = t + zn, a = S - y, b = fl(x*x + zn) by a second FMA, and C takes a + b.
//  * t <= 2S: S - t is exact (Sterbenz), so zn = S - t, y = S, a = 0 and b is
//    the addition's exact error S + x*x - t rounded once.
//  * t > 2S: zn lies in [-t, -t/2], so y = t + zn is exact and equals S + d,
//    d the rounding error of S - t; a = -d exactly, and b = (error + d)
//    rounded once, with |error + d| <= ulp(t).
// Either way a + b is the error of t to within about 3u^2 t (u = 2^-24): the
// square need not be exact in fp32, so fp32 inputs need no separate residual
// term, and for bf16 inputs (exact squares) this is Knuth's TwoSum exactly.
__device__ __forceinline__ void two_sum_sq(u64& S, u64& C, u64 x) {
  const u64 t = fma2(x, x, S);
  const u64 zn = sub2(S, t);
  const u64 y = add2(t, zn);
  const u64 a = sub2(S, y);
  const u64 b = fma2(x, x, zn);
  C = add2(C, add2(a, b));
  S = t;
}

// S + C += p, error-free (Knuth's TwoSum): S takes the rounded sum, C the
// rounding error.
__device__ __forceinline__ void two_sum_acc(u64& S, u64& C, u64 p) {
  const u64 t = add2(S, p);
  const u64 z = sub2(t, S);
  const u64 y = sub2(t, z);
  const u64 a = sub2(S, y);
  const u64 b = sub2(p, z);
  C = add2(C, add2(a, b));
  S = t;
}

struct FpAcc {
  u64 A, CA, B, CB;  // two f32x2 accumulators with their error terms
};

template <int DT>
__device__ __forceinline__ void fp_unit(const uint4& v, FpAcc& f) {
  if (DT == kDtF32) {
    two_sum_sq(f.A, f.CA, pk(v.x, v.y));
    two_sum_sq(f.B, f.CB, pk(v.z, v.w));
  } else {
    // bf16 pairs: the low element is the low half-word
    const u64 y0 = pk(v.x << 16, v.x & 0xFFFF0000u), y1 = pk(v.y << 16, v.y & 0xFFFF0000u);
    const u64 y2 = pk(v.z << 16, v.z & 0xFFFF0000u), y3 = pk(v.w << 16, v.w & 0xFFFF0000u);
    two_sum_sq(f.A, f.CA, y0);
    two_sum_sq(f.B, f.CB, y2);
    two_sum_sq(f.A, f.CA, y1);
    two_sum_sq(f.B, f.CB, y3);
  }
}

struct Exact {
  double d;
  uint32_t nonfinite;
};

// Exact per-element fallback for this lane's units of blocks [b0, b1):
// non-finite elements are counted; each finite square is added exactly --
// for |x| in [2^-40, 2^56] as its fp32 product and FMA residual into an
// unevaluated float pair by TwoSum, else (tiny or huge values, rare) in fp64,
// where the square of an fp32 value is exact.  Its error, under n^2 u^2 of
// the sum for the n elements of a lane, is far inside the sums' bound.  The
// segment was just swept (its lines are mostly in L2); the lane first
// prefetches all its units into L1, so the reloads do not wait for L2 one by
// one, and the float pair keeps the arithmetic off GB300's narrow fp64 pipe.
// (Loading the units in register batches instead makes the compiler spill in
// the hot loop that calls this.)
template <int DT, int AL>
__device__ __noinline__ Exact slow_span(const uint8_t* sp, uint64_t b0, uint64_t b1) {
  for (uint64_t b = b0; b < b1; ++b) asm volatile("prefetch.global.L1 [%0];" ::"l"(sp + b * kBlockBytes));
  float hi = 0.0f, lo = 0.0f;
  double d = 0.0;
  uint32_t nonfinite = 0;
  for (uint64_t b = b0; b < b1; ++b) {
    const uint4 v = ld_unit<AL>(sp + b * kBlockBytes);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
#pragma unroll
      for (int h = 0; h < (DT == kDtF32 ? 1 : 2); ++h) {
        const uint32_t f = DT == kDtF32 ? w[j] : (h == 0 ? w[j] << 16 : w[j] & 0xFFFF0000u);
        if ((f & 0x7F800000u) == 0x7F800000u) {
          ++nonfinite;
          continue;
        }
        const float x = __uint_as_float(f);
        const float ax = fabsf(x);
        if (ax >= 0x1p-40f && ax <= 0x1p56f) {
          const float p2 = x * x;
          const float e = __fmaf_rn(x, x, -p2);
          const float t = hi + p2;
          const float z = t - hi;
          lo += ((hi - (t - z)) + (p2 - z)) + e;
          hi = t;
        } else if (ax != 0.0f) {
          const double xd = static_cast<double>(x);
          d = __dadd_rn(d, __dmul_rn(xd, xd));
        }
      }
    }
  }
  return Exact{(static_cast<double>(hi) + static_cast<double>(lo)) + d, nonfinite};
}

// Whether this lane's units of blocks [b0, b1) hold only (signed) zeros.
template <int DT, int AL>
__device__ __noinline__ bool span_is_zero(const uint8_t* sp, uint64_t b0, uint64_t b1) {
  constexpr uint32_t kMask = (DT == kDtF32) ? 0x7FFFFFFFu : 0x7FFF7FFFu;
  uint32_t acc = 0;
  for (uint64_t b = b0; b < b1; ++b) {
    const uint4 v = ld_unit<AL>(sp + b * kBlockBytes);
    acc |= (v.x | v.y | v.z | v.w) & kMask;
  }
  return acc == 0;
}

// The span's sum as an unevaluated float pair (hi, lo): the four fp32 partial
// sums are merged error-free in fp32 (TwoSum); the error terms (about 2^-24
// of the sum) are merged with plain fp32 adds, which costs about 2^-48
// relative.  No fp64 work: GB300's fp64 pipe is narrow.
__device__ __forceinline__ void fold_to_pair(const FpAcc& f, float& hi, float& lo) {
  u64 s = f.A, c = add2(f.CA, f.CB);
  two_sum_acc(s, c, f.B);
  const float a = lo_f(s), b = hi_f(s);
  const float t = a + b;
  const float z = t - a;
  const float err = (a - (t - z)) + (b - z);
  hi = t;
  lo = (lo_f(c) + hi_f(c)) + err;
}

// ------------------------------------------------------------------ piece

// Bulk prefetch of [p, p + bytes) into L2 (TMA unit; no registers held).
__device__ __forceinline__ void prefetch_l2(const uint8_t* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// The same, issued by lane 0 only, as a predicated instruction (no branch).
__device__ __forceinline__ void prefetch_l2_lane0(const uint8_t* p, uint32_t bytes, uint32_t lane) {
  asm volatile(
      "{\n\t.reg .pred q;\n\tsetp.eq.u32 q, %2, 0;\n\t@q cp.async.bulk.prefetch.L2.global [%0], %1;\n\t}" ::"l"(p),
      "r"(bytes), "r"(lane)
      : "memory");
}

// Per-mode pipeline geometry: blocks per lane held in registers one stage
// ahead, and spans (kSpan blocks) prefetched into L2 ahead of use.
template <int MODE>
// Unpack with fingerprint values does pack's work per byte (copy, CRC, sums),
// so it takes pack's geometry.
struct Geo {
  static constexpr bool kPackLike = MODE == kModePack || MODE == kModeUnpackFp;
  static constexpr int kStage = MODE == kModeFingerprint ? FR_STAGE_FP : (kPackLike ? FR_STAGE_PACK
                                                                                    : FR_STAGE_UNPACK);
  static constexpr int kAhead = MODE == kModeFingerprint ? FR_AHEAD_FP : (kPackLike ? FR_AHEAD_PACK
                                                                                    : FR_AHEAD_UNPACK);
  // Issue a unit's reload before consuming it (more load lead, one register
  // copy) or after (no copy): latency-bound modes want the former.
  static constexpr bool kLoadFirst = MODE == kModeFingerprint ? FR_LOADFIRST_FP
                                     : (kPackLike ? FR_LOADFIRST_PACK : FR_LOADFIRST_UNPACK);
  static_assert(kSpan % kStage == 0, "a span holds whole stages");
};

// State of one lane while it sweeps a piece.
template <int MODE, int DT>
struct Lane {
  uint32_t s[4];  // CRC streams 4l..4l+3
  FpAcc f;        // fp32 sums of the current span
  uint32_t nonfinite;
};

template <int MODE, int DT, int DAL>
__device__ __forceinline__ void do_unit(Lane<MODE, DT>& L, const uint4& v, uint8_t* wp, uint32_t lb) {
  constexpr bool kFp = mode_sums(MODE) && (DT != kDtBytes);
  if (MODE != kModeFingerprint) st_unit<DAL>(wp, v);
  L.s[0] = braid_step(L.s[0] ^ v.x, lb);
  L.s[1] = braid_step(L.s[1] ^ v.y, lb);
  L.s[2] = braid_step(L.s[2] ^ v.z, lb);
  L.s[3] = braid_step(L.s[3] ^ v.w, lb);
  if (kFp) fp_unit<DT>(v, L.f);
}

// End of a span [b0, b1) (one segment): the fast sums are kept if finite and
// either large enough that fp32 underflow is negligible (below 2^-77 relative)
// or made of zeros only; otherwise the segment is summed exactly from a
// reload.  The lanes' sums are then added in a fixed tree and lane 0 stores
// the segment's sum (a float pair, see seg_value) at its index.
template <int MODE, int DT, int SAL>
__device__ __forceinline__ void span_end(Lane<MODE, DT>& L, const uint8_t* sp, uint64_t b0, uint64_t b1,
                                         double* seg, uint32_t lane) {
  const u64 ab = add2(L.f.A, L.f.B);
  const float tot = lo_f(ab) + hi_f(ab);
  bool ok = tot < __int_as_float(0x7F800000);
  if (ok && !(tot >= 0x1p-60f)) ok = span_is_zero<DT, SAL>(sp, b0, b1);
  float hi = 0.0f, lo = 0.0f;
  double d = 0.0;
  if (ok) {
    fold_to_pair(L.f, hi, lo);
  } else {
    const Exact x = slow_span<DT, SAL>(sp, b0, b1);
    d = x.d;
    L.nonfinite += x.nonfinite;
  }
  L.f.A = L.f.CA = L.f.B = L.f.CB = 0ull;
  // The lanes' sums are added in a fixed tree: as float pairs by TwoSum when
  // every lane took the fast path with a sum far from fp32 overflow (no fp64
  // work), else in fp64 (rare).  Lane 0 stores the form seg_value() reads.
  if (__all_sync(0xFFFFFFFFu, ok && tot < 0x1p120f)) {
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) {
      const float oh = __shfl_down_sync(0xFFFFFFFFu, hi, m);
      const float ol = __shfl_down_sync(0xFFFFFFFFu, lo, m);
      const float t = hi + oh;
      const float z = t - hi;
      const float err = (hi - (t - z)) + (oh - z);
      lo = (lo + ol) + err;
      hi = t;
    }
    if (lane == 0) *reinterpret_cast<float2*>(seg) = make_float2(lo, hi);
  } else {
    if (ok) d = static_cast<double>(hi) + static_cast<double>(lo);
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) d += __shfl_down_sync(0xFFFFFFFFu, d, m);
    if (lane == 0) *seg = -d;
  }
}

// One piece: `nblk` 512-byte blocks from `src` (to `dst` for pack/unpack).
// SAL / DAL: alignment class (16, 4 or 1 bytes) of the source / destination.
//
// Pipeline: lane 0 prefetches whole spans into L2 kAhead spans ahead with the
// bulk-copy unit; each lane keeps kStage 16-byte units of the next stage in
// flight in registers, which therefore mostly wait for L2.  Each span is one
// sum segment: its fp32 sums start at zero, are checked at its end, and are
// replaced by an exact sum from a reload when they fail.
template <int MODE, int DT, int SAL, int DAL>
__device__ __forceinline__ void sweep_piece(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                            uint64_t nblk, uint32_t lane, Record* rec, double* segs) {
  constexpr bool kFp = mode_sums(MODE) && (DT != kDtBytes);
  constexpr int kStage = Geo<MODE>::kStage;
  constexpr int kAhead = Geo<MODE>::kAhead;
  constexpr uint32_t kStageBytes = kStage * kBlockBytes;
  const uint32_t lb = lane << 2;
  const uint8_t* sp = src + lane * 16;
  uint8_t* wp = dst + lane * 16;

  // The first span goes to L2 now; each later one about a span before use.
  if (kAhead > 0 && SAL == 16) {
    const uint64_t n = nblk < kSpan ? nblk : kSpan;
    prefetch_l2_lane0(src, static_cast<uint32_t>(n * kBlockBytes), lane);
  }

  Lane<MODE, DT> L;
  L.s[0] = L.s[1] = L.s[2] = L.s[3] = 0;
  L.f = FpAcc{0ull, 0ull, 0ull, 0ull};
  L.nonfinite = 0;

  uint4 cur[kStage];
#pragma unroll
  for (int u = 0; u < kStage; ++u)
    if (u < nblk) cur[u] = ld_unit<SAL>(sp + static_cast<uint64_t>(u) * kBlockBytes);
  const uint8_t* lp = sp + kStageBytes;  // the next stage's loads

  // Three loops cover a piece: (1) whole spans whose following stage is
  // whole too, each span (one sum segment) a call-free loop of kSpan/kStage
  // stages with no branch, preceded by the L2 prefetch of the span kAhead
  // ahead and followed by its validity check -- the bulk of a long piece;
  // (2) the stages left whose following stage is still whole, one stage per
  // iteration, a span's check and the next prefetch when a stage ends a span;
  // (3) the last one or two stages, predicated.  Loop (2) keeps the
  // predicated drain to under 2 * kStage blocks (it used to take the last
  // span and a stage, and ran at half speed); loop (1) keeps long pieces on
  // the tighter loop (with (2) alone the bf16 fingerprint lost 12% per warp).
  uint64_t i = 0;  // first block of the current span
  for (; i + kSpan + kStage <= nblk; i += kSpan) {
    if (kAhead > 0 && SAL == 16 && lane == 0) {
      const uint64_t pf = i + kSpan * kAhead;
      if (pf < nblk) {
        const uint64_t n = (nblk - pf < kSpan) ? nblk - pf : kSpan;
        prefetch_l2(src + pf * kBlockBytes, static_cast<uint32_t>(n * kBlockBytes));
      }
    }
#pragma unroll 1
    for (int stg = 0; stg < kSpan / kStage; ++stg) {
#pragma unroll
      for (int u = 0; u < kStage; ++u) {
        if (Geo<MODE>::kLoadFirst) {
          const uint4 v = cur[u];
          cur[u] = ld_unit<SAL>(lp + u * kBlockBytes);
          do_unit<MODE, DT, DAL>(L, v, wp + u * kBlockBytes, lb);
        } else {
          do_unit<MODE, DT, DAL>(L, cur[u], wp + u * kBlockBytes, lb);
          cur[u] = ld_unit<SAL>(lp + u * kBlockBytes);
        }
      }
      lp += kStageBytes;
      wp += kStageBytes;
    }
    if (kFp) span_end<MODE, DT, SAL>(L, sp, i, i + kSpan, segs + i / kSpan, lane);
  }
  if (kAhead > 0 && SAL == 16) {  // loop (2) prefetches at span ends only
    const uint64_t pf = i + kSpan * kAhead;
    if (pf < nblk) {
      const uint64_t n = (nblk - pf < kSpan) ? nblk - pf : kSpan;
      prefetch_l2_lane0(src + pf * kBlockBytes, static_cast<uint32_t>(n * kBlockBytes), lane);
    }
  }
  // Loop (2): stage j after i is steady if i + (j + 2) * kStage <= nblk.
  uint32_t st = 0;  // stages of the current span done
  const uint64_t left = nblk - i;
  const uint32_t n_steady = left >= 2 * kStage ? static_cast<uint32_t>((left - kStage) / kStage) : 0u;
#pragma unroll 1
  for (uint32_t k = n_steady; k > 0; --k) {
#pragma unroll
    for (int u = 0; u < kStage; ++u) {
      if (Geo<MODE>::kLoadFirst) {
        const uint4 v = cur[u];
        cur[u] = ld_unit<SAL>(lp + u * kBlockBytes);
        do_unit<MODE, DT, DAL>(L, v, wp + u * kBlockBytes, lb);
      } else {
        do_unit<MODE, DT, DAL>(L, cur[u], wp + u * kBlockBytes, lb);
        cur[u] = ld_unit<SAL>(lp + u * kBlockBytes);
      }
    }
    lp += kStageBytes;
    wp += kStageBytes;
    if (++st == kSpan / kStage) {
      st = 0;
      if (kFp) span_end<MODE, DT, SAL>(L, sp, i, i + kSpan, segs + i / kSpan, lane);
      if (kAhead > 0 && SAL == 16) {
        const uint64_t pf = i + kSpan + kSpan * kAhead;
        if (pf < nblk) {
          const uint64_t n = (nblk - pf < kSpan) ? nblk - pf : kSpan;
          prefetch_l2_lane0(src + pf * kBlockBytes, static_cast<uint32_t>(n * kBlockBytes), lane);
        }
      }
      i += kSpan;
    }
  }
  i += static_cast<uint64_t>(st) * kStage;
  // Drain: the last one or two stages (fewer than 2 * kStage blocks), with
  // predicates.
  for (; i < nblk; i += kStage) {
#pragma unroll
    for (int u = 0; u < kStage; ++u) {
      if (i + u < nblk) {
        do_unit<MODE, DT, DAL>(L, cur[u], wp + u * kBlockBytes, lb);
        if (i + kStage + u < nblk) cur[u] = ld_unit<SAL>(lp + u * kBlockBytes);
      }
    }
    lp += kStageBytes;
    wp += kStageBytes;
    const uint64_t end = (i + kStage < nblk) ? i + kStage : nblk;
    if (kFp && ((end & (kSpan - 1)) == 0 || end == nblk))
      span_end<MODE, DT, SAL>(L, sp, i & ~static_cast<uint64_t>(kSpan - 1), end, segs + i / kSpan, lane);
  }

  // ---- fold the 128 streams into the raw CRC of the piece
  uint32_t v = mul_fold(0, L.s[0]) ^ L.s[1];
  v = mul_fold(0, v) ^ L.s[2];
  v = mul_fold(0, v) ^ L.s[3];
  {
    uint32_t o;
    o = __shfl_down_sync(0xFFFFFFFFu, v, 1);
    v = mul_fold(1, v) ^ o;
    o = __shfl_down_sync(0xFFFFFFFFu, v, 2);
    v = mul_fold(2, v) ^ o;
    o = __shfl_down_sync(0xFFFFFFFFu, v, 4);
    v = mul_fold(3, v) ^ o;
    o = __shfl_down_sync(0xFFFFFFFFu, v, 8);
    v = mul_fold(4, v) ^ o;
    o = __shfl_down_sync(0xFFFFFFFFu, v, 16);
    v = mul_fold(5, v) ^ o;
  }

  uint32_t nonfinite = L.nonfinite;
  if (kFp) {
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) nonfinite += __shfl_down_sync(0xFFFFFFFFu, nonfinite, m);
  }
  if (lane == 0) {
    Record r;
    r.crc = mul_fold(6, v);
    r.nonfinite = nonfinite;
    r.unused = 0.0;
    *rec = r;
  }
}

template <int MODE, int DT, int AL>
__device__ __forceinline__ void sweep_piece_al(const uint8_t* tensor, uint8_t* packed, uint64_t n,
                                               uint32_t lane, Record* rec, double* segs) {
  if (mode_unpacks(MODE))
    sweep_piece<MODE, DT, 16, AL>(packed, const_cast<uint8_t*>(tensor), n, lane, rec, segs);
  else
    sweep_piece<MODE, DT, AL, 16>(tensor, packed, n, lane, rec, segs);
}

// Claims the next unit of class c for this warp: its index within the
// class's units, or n_units[c] when none is left.
__device__ __forceinline__ uint32_t claim_unit(const SweepParams& p, uint32_t c, uint32_t lane) {
  uint32_t u = 0;
  if (lane == 0) u = atomicAdd(p.queue + c, 1u);
  return __shfl_sync(0xFFFFFFFFu, u, 0);
}

// Whether a mode's mixed launches take claimed units: pack and unpack, which
// are bound by memory latency and whose warps' rates differ from SM to SM by
// a few percent.  The issue-bound fingerprint keeps its static split: the
// claim loop around its sweep costs it more registers than the tail it
// would save.
__host__ __device__ constexpr bool mode_claims(int m) { return m != kModeFingerprint; }

// One warp's range of its class's block stream: the pieces it overlaps, in
// order.  ALIGNED: every tensor of the class is 16-byte aligned (128-bit
// loads and stores); else the tensor side uses 32-bit or byte accesses, chosen
// per piece.
template <int MODE, int DT, bool ALIGNED>
__device__ __forceinline__ void sweep_warp(const SweepParams& p, const WarpDesc& wd, const uint32_t* class_chunks,
                                           uint32_t lane) {
  uint64_t b = wd.blk_begin, left = wd.nblk;
  uint32_t k = wd.first_chunk, r = wd.rec_base;
  while (left > 0) {
    const ChunkDesc cd = p.chunks[class_chunks[k]];
    const uint64_t nb = cd.len / kBlockBytes;
    const uint64_t off = b - cd.blk_begin;
    const uint64_t n = (left < nb - off) ? left : nb - off;
    const uint8_t* tensor = reinterpret_cast<const uint8_t*>(cd.addr) + off * kBlockBytes;
    uint8_t* packed = (MODE == kModeFingerprint) ? nullptr : p.packed + cd.payload_off + off * kBlockBytes;
    double* segs = p.segs + cd.seg_base + off / kSegBlocks;
    if (ALIGNED) {
      sweep_piece_al<MODE, DT, 16>(tensor, packed, n, lane, p.recs + r, segs);
    } else if ((reinterpret_cast<uintptr_t>(tensor) & 3u) == 0) {
      sweep_piece_al<MODE, DT, 4>(tensor, packed, n, lane, p.recs + r, segs);
    } else {
      sweep_piece_al<MODE, DT, 1>(tensor, packed, n, lane, p.recs + r, segs);
    }
    ++r;
    b += n;
    left -= n;
    ++k;
  }
}

// One warp's range, then (pack and unpack launches with units, p.queue set)
// the units of sweep class `cls` it claims, one at a time, until none is
// left.  (Plain unpack runs every element type as bytes, so `cls` names the
// class's queue, not the code.)
template <int MODE, int DT, bool ALIGNED>
__device__ __forceinline__ void sweep_warp_claims(const SweepParams& p, const WarpDesc& wd, uint32_t cls,
                                                  uint32_t lane) {
  const uint32_t* class_chunks = p.class_chunks + wd.list_off;
  WarpDesc cur = wd;
  for (;;) {
    sweep_warp<MODE, DT, ALIGNED>(p, cur, class_chunks, lane);
    if (p.queue == nullptr) return;
    const uint32_t u = claim_unit(p, cls, lane);
    if (u >= p.n_units[cls]) return;
    cur = p.units[p.unit_off[cls] + u];
  }
}

// One kernel per (mode, element type, alignment class).
template <int MODE, int DT, bool ALIGNED>
__global__ void __launch_bounds__(Cta<MODE>::kThreads, 1) sweep_kernel(SweepParams p) {
  fill_tables<Cta<MODE>::kThreads>();
  __syncthreads();
  const uint32_t lane = threadIdx.x & 31u;
  const uint32_t w = blockIdx.x * Cta<MODE>::kWarps + (threadIdx.x >> 5);
  if (w >= p.n_warps) return;
  sweep_warp<MODE, DT, ALIGNED>(p, p.warps[w], p.class_chunks, lane);
}

// Class c's code for this mode: plain unpack only copies and checksums, so
// it runs every element type as bytes.
template <int MODE, uint32_t C>
__device__ __forceinline__ void sweep_class(const SweepParams& p, const WarpDesc& wd, uint32_t lane) {
  constexpr int DT = mode_sums(MODE) ? static_cast<int>(C / 2) : static_cast<int>(kDtBytes);
  sweep_warp_claims<MODE, DT, (C & 1u) != 0>(p, wd, C, lane);
}

// Help with class c's units left once a warp's own class has none.
template <int MODE, uint32_t C>
__device__ __forceinline__ void help_class(const SweepParams& p, uint32_t lane) {
  if (p.n_units[C] == 0) return;
  WarpDesc none;
  none.blk_begin = 0;
  none.nblk = 0;
  none.first_chunk = 0;
  none.rec_base = 0;
  none.cls = C;
  none.list_off = p.list_off[C];
  sweep_class<MODE, C>(p, none, lane);
}

// Every class of a batch in one launch: each warp sweeps a range of its own
// class, and the plan spreads each class's warps over all CTAs, so warps that
// wait on memory and warps that are bound by instruction issue share every
// SM.  The ranges cover most of each class's blocks; the rest is cut into
// small units that warps claim one at a time once their own range is done:
// first their own class's, then, in a fixed order, every other class's, so
// the launch ends when the work does, not when its slowest warp does.  Which
// warp sweeps a unit changes nothing in the results: a unit's records and
// segment sums have fixed slots.  (The class code is inlined once per call
// site and no loop runs over classes: a loop around the inlined sweeps makes
// the compiler keep every variant's registers live at once.)
template <int MODE>
__global__ void __launch_bounds__(Cta<MODE>::kThreads, 1) sweep_mixed_kernel(SweepParams p) {
  fill_tables<Cta<MODE>::kThreads>();
  __syncthreads();
  const uint32_t lane = threadIdx.x & 31u;
  const uint32_t w = blockIdx.x * Cta<MODE>::kWarps + (threadIdx.x >> 5);
  if constexpr (!mode_claims(MODE)) {
    // the static split: each warp its own range, one dispatch on its class
    if (w >= p.n_warps) return;
    const WarpDesc wd = p.warps[w];
    const uint32_t* list = p.class_chunks + wd.list_off;
    switch (wd.cls) {
      case kDtF32 * 2 + 1: sweep_warp<MODE, kDtF32, true>(p, wd, list, lane); break;
      case kDtBf16 * 2 + 1: sweep_warp<MODE, kDtBf16, true>(p, wd, list, lane); break;
      case kDtBytes * 2 + 1: sweep_warp<MODE, kDtBytes, true>(p, wd, list, lane); break;
      case kDtF32 * 2: sweep_warp<MODE, kDtF32, false>(p, wd, list, lane); break;
      case kDtBf16 * 2: sweep_warp<MODE, kDtBf16, false>(p, wd, list, lane); break;
      default: sweep_warp<MODE, kDtBytes, false>(p, wd, list, lane); break;
    }
  } else {
    if (w < p.n_warps) {
      const WarpDesc wd = p.warps[w];
      switch (wd.cls) {
        case kDtF32 * 2 + 1: sweep_class<MODE, kDtF32 * 2 + 1>(p, wd, lane); break;
        case kDtBf16 * 2 + 1: sweep_class<MODE, kDtBf16 * 2 + 1>(p, wd, lane); break;
        case kDtBytes * 2 + 1: sweep_class<MODE, kDtBytes * 2 + 1>(p, wd, lane); break;
        case kDtF32 * 2: sweep_class<MODE, kDtF32 * 2>(p, wd, lane); break;
        case kDtBf16 * 2: sweep_class<MODE, kDtBf16 * 2>(p, wd, lane); break;
        default: sweep_class<MODE, kDtBytes * 2>(p, wd, lane); break;
      }
    }
    if (p.queue == nullptr) return;
    help_class<MODE, kDtF32 * 2 + 1>(p, lane);
    help_class<MODE, kDtBf16 * 2 + 1>(p, lane);
    help_class<MODE, kDtBytes * 2 + 1>(p, lane);
    help_class<MODE, kDtF32 * 2>(p, lane);
    help_class<MODE, kDtBf16 * 2>(p, lane);
    help_class<MODE, kDtBytes * 2>(p, lane);
    // Every warp has made its last claim once it gets here; the last one out
    // zeroes the queue for the next launch on this plan.
    if (lane == 0) {
      __threadfence();
      if (atomicAdd(p.queue + kClassCount, 1u) == gridDim.x * Cta<MODE>::kWarps - 1) {
        for (uint32_t c = 0; c <= kClassCount; ++c) atomicExch(p.queue + c, 0u);
      }
    }
  }
}

// List mode (re-sending failed chunks): warp w sweeps the whole body of chunk
// ids[w] into recs[w].  Every variant is a separate function, so this cold
// kernel's dispatch does not burden the registers of the hot ones.
template <int MODE, int DT, bool ALIGNED>
__device__ __noinline__ void list_piece(const uint8_t* tensor, uint8_t* packed, uint64_t n, uint32_t lane,
                                        Record* rec, double* segs) {
  if (ALIGNED)
    sweep_piece_al<MODE, DT, 16>(tensor, packed, n, lane, rec, segs);
  else if ((reinterpret_cast<uintptr_t>(tensor) & 3u) == 0)
    sweep_piece_al<MODE, DT, 4>(tensor, packed, n, lane, rec, segs);
  else
    sweep_piece_al<MODE, DT, 1>(tensor, packed, n, lane, rec, segs);
}

template <int MODE>
__global__ void __launch_bounds__(Cta<MODE>::kThreads, 1) list_kernel(ListParams p) {
  fill_tables<Cta<MODE>::kThreads>();
  __syncthreads();
  const uint32_t lane = threadIdx.x & 31u;
  const uint64_t w = static_cast<uint64_t>(blockIdx.x) * Cta<MODE>::kWarps + (threadIdx.x >> 5);
  if (w >= p.n) return;
  const ChunkDesc cd = p.chunks[p.ids[w]];
  const uint64_t nb = cd.len / kBlockBytes;
  if (nb == 0) return;
  const uint8_t* tensor = reinterpret_cast<const uint8_t*>(cd.addr);
  uint8_t* packed = (MODE == kModeFingerprint) ? nullptr : p.packed + cd.payload_off;
  const bool aligned = (cd.sweep_class & 1u) != 0;
  const uint32_t dt = mode_sums(MODE) ? cd.dtype : kDtBytes;
  double* segs = p.segs + cd.seg_base;
  Record* rec = p.recs + w;
  if (dt == kDtF32) {
    if (aligned) list_piece<MODE, kDtF32, true>(tensor, packed, nb, lane, rec, segs);
    else list_piece<MODE, kDtF32, false>(tensor, packed, nb, lane, rec, segs);
  } else if (dt == kDtBf16) {
    if (aligned) list_piece<MODE, kDtBf16, true>(tensor, packed, nb, lane, rec, segs);
    else list_piece<MODE, kDtBf16, false>(tensor, packed, nb, lane, rec, segs);
  } else {
    if (aligned) list_piece<MODE, kDtBytes, true>(tensor, packed, nb, lane, rec, segs);
    else list_piece<MODE, kDtBytes, false>(tensor, packed, nb, lane, rec, segs);
  }
}

template <int MODE>
cudaError_t launch_list(const ListParams& p, cudaStream_t s) {
  if (p.n == 0) return cudaSuccess;
  const uint64_t ctas = (p.n + Cta<MODE>::kWarps - 1) / Cta<MODE>::kWarps;
  list_kernel<MODE><<<static_cast<unsigned>(ctas), Cta<MODE>::kThreads, kTableBytes, s>>>(p);
  return cudaGetLastError();
}

template <int MODE, int DT, bool ALIGNED>
cudaError_t configure_one() {
  return cudaFuncSetAttribute(sweep_kernel<MODE, DT, ALIGNED>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kTableBytes);
}

template <int MODE, int DT, bool ALIGNED>
cudaError_t launch_one(const SweepParams& p, int n_ctas, cudaStream_t s) {
  sweep_kernel<MODE, DT, ALIGNED><<<n_ctas, Cta<MODE>::kThreads, kTableBytes, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

// Configure / launch every class kernel of one mode (plain unpack ignores the
// element type: it only checksums and copies).
template <int MODE>
cudaError_t configure_mode() {
  cudaError_t e = cudaFuncSetAttribute(list_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, kTableBytes);
  if (e == cudaSuccess) e = configure_one<MODE, kDtBytes, true>();
  if (e == cudaSuccess) e = configure_one<MODE, kDtBytes, false>();
  if (mode_sums(MODE)) {
    if (e == cudaSuccess) e = configure_one<MODE, kDtBf16, true>();
    if (e == cudaSuccess) e = configure_one<MODE, kDtBf16, false>();
    if (e == cudaSuccess) e = configure_one<MODE, kDtF32, true>();
    if (e == cudaSuccess) e = configure_one<MODE, kDtF32, false>();
  }
  return e;
}

template <int MODE>
cudaError_t configure_mixed() {
  return cudaFuncSetAttribute(sweep_mixed_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, kTableBytes);
}

template <int MODE>
cudaError_t launch_mixed(const SweepParams& p, int n_ctas, cudaStream_t s) {
  sweep_mixed_kernel<MODE><<<n_ctas, Cta<MODE>::kThreads, kTableBytes, s>>>(p);
  return cudaGetLastError();
}

template <int MODE>
cudaError_t launch_mode(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s) {
  if (!mode_sums(MODE) || dtype == kDtBytes)
    return aligned ? launch_one<MODE, kDtBytes, true>(p, n_ctas, s) : launch_one<MODE, kDtBytes, false>(p, n_ctas, s);
  if (dtype == kDtBf16)
    return aligned ? launch_one<MODE, kDtBf16, true>(p, n_ctas, s) : launch_one<MODE, kDtBf16, false>(p, n_ctas, s);
  return aligned ? launch_one<MODE, kDtF32, true>(p, n_ctas, s) : launch_one<MODE, kDtF32, false>(p, n_ctas, s);
}

}  // namespace frk
