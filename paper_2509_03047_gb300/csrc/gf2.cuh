// gf2.cuh -- CRC-32C arithmetic in GF(2)[x] / P(x), evaluated at compile time.
//
// Representation: the reflected CRC register.  Bit j of a 32-bit word is the
// coefficient of x^(31-j), so 0x80000000 is the polynomial 1 and the reflected
// Castagnoli polynomial 0x82F63B78 is x^32 mod P.  Running one zero bit
// through the register multiplies it by x; running a byte b into a zero
// register gives b * x^8; running the little-endian word w into register r
// gives (r ^ w) * x^32.  Everything the kernels need follows from linearity:
//
//   raw(A || B) = raw(A) * x^(8|B|) ^ raw(B)            (raw: preset 0, no final XOR)
//   crc(M)      = raw(M) ^ 0xFFFFFFFF * x^(8|M|) ^ 0xFFFFFFFF
//
// The tables are generated here from the polynomial by constant evaluation;
// nothing is copied from elsewhere.
#pragma once

#include <cstdint>

namespace frk {

constexpr uint32_t kPoly = 0x82F63B78u;  // reflected CRC-32C polynomial
constexpr uint32_t kOne = 0x80000000u;   // the polynomial 1

// r * x mod P
__host__ __device__ constexpr uint32_t gf_mul_x(uint32_t r) {
  return (r >> 1) ^ ((r & 1u) ? kPoly : 0u);
}

// r * x^-1 mod P (P has a constant term, so x is invertible)
__host__ __device__ constexpr uint32_t gf_div_x(uint32_t r) {
  return (r & 0x80000000u) ? (((r ^ kPoly) << 1) | 1u) : (r << 1);
}

// a * b mod P
__host__ __device__ constexpr uint32_t gf_mulmod(uint32_t a, uint32_t b) {
  uint32_t r = 0;
  for (int k = 0; k < 32; ++k) {
    if (a & (kOne >> k)) r ^= b;
    b = gf_mul_x(b);
  }
  return r;
}

// x^n mod P
__host__ __device__ constexpr uint32_t gf_xpow(uint64_t n) {
  uint32_t r = kOne, base = gf_mul_x(kOne);
  while (n) {
    if (n & 1u) r = gf_mulmod(r, base);
    base = gf_mulmod(base, base);
    n >>= 1;
  }
  return r;
}

// x^-n mod P
__host__ __device__ constexpr uint32_t gf_xpow_neg(uint64_t n) {
  uint32_t r = kOne, base = gf_div_x(kOne);
  while (n) {
    if (n & 1u) r = gf_mulmod(r, base);
    base = gf_mulmod(base, base);
    n >>= 1;
  }
  return r;
}

// ---------------------------------------------------------------------------
// Interleaved ("braided") streams.  A warp reads the state in 512-byte
// blocks, lane l taking bytes [16l, 16l+16) of every block, i.e. the 32-bit
// words 4l..4l+3.  Word j of every block forms stream j (128 streams); each
// stream is a CRC over its own words with 127 zero words between them, so a
// stream step is  s <- (s ^ w) * x^(32*128).  Lane l owns streams 4l..4l+3.
constexpr int kBlockBytes = 512;
constexpr int kStreams = kBlockBytes / 4;                  // 128
constexpr uint32_t kBraidMul = gf_xpow(32ull * kStreams);  // x^4096
// After the streams are folded Horner-style (stream 0 first), the value is
// raw(piece) * x^(32*127); kUnbraid removes that factor.
constexpr uint32_t kUnbraid = gf_xpow_neg(32ull * (kStreams - 1));

struct ByteTables4 {
  uint32_t t[4][256];
};

// t[k][b] = (b << 8k) * m : the contribution of byte k of a register.
__host__ __device__ constexpr ByteTables4 make_mul_tables(uint32_t m) {
  ByteTables4 out{};
  for (int k = 0; k < 4; ++k) {
    // contribution of the single bit j of byte k, then all 256 values by XOR
    uint32_t bit[8] = {};
    for (int j = 0; j < 8; ++j) bit[j] = gf_mulmod(1u << (8 * k + j), m);
    for (int b = 0; b < 256; ++b) {
      uint32_t v = 0;
      for (int j = 0; j < 8; ++j)
        if (b & (1 << j)) v ^= bit[j];
      out.t[k][b] = v;
    }
  }
  return out;
}

// Powers for shifting a raw CRC by n bytes: x^(8n) = prod_k p[k][byte k of n].
constexpr int kPowBytes = 6;  // n < 2^48
struct PowTables {
  uint32_t p[kPowBytes][256];
};

__host__ __device__ constexpr PowTables make_pow_tables() {
  PowTables out{};
  for (int k = 0; k < kPowBytes; ++k) {
    const uint32_t step = gf_xpow(8ull << (8 * k));  // x^(8 * 256^k)
    uint32_t v = kOne;
    for (int b = 0; b < 256; ++b) {
      out.p[k][b] = v;
      v = gf_mulmod(v, step);
    }
  }
  return out;
}

// x^(8n) mod P on the host, from the per-byte power tables.
inline uint32_t host_xpow8(uint64_t n) {
  static const PowTables T = make_pow_tables();
  uint32_t r = kOne;
  for (int k = 0; k < kPowBytes; ++k) {
    const uint32_t byte = static_cast<uint32_t>(n >> (8 * k)) & 255u;
    if (byte) r = gf_mulmod(r, T.p[k][byte]);
  }
  return r;
}

// The CRC-32C preset and final XOR of an n-byte message as one term:
// crc = raw ^ crc_xor_term(n), raw being the CRC register run from zero.
inline uint32_t host_crc_xor_term(uint64_t n) { return gf_mulmod(0xFFFFFFFFu, host_xpow8(n)) ^ 0xFFFFFFFFu; }

}  // namespace frk
