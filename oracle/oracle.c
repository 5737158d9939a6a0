/*
 * oracle.c -- plain single-threaded CPU reference for the restoration sweep.
 *
 * TEST INFRASTRUCTURE ONLY (see oracle.h).  The operations follow the
 * restoration step of FlashRecovery (arXiv 2509.03047, Sec. III-E, "Model
 * states Restoration"): a restarted rank's model and optimizer state is
 * rebuilt from a data-parallel replica.  The paper does not define the
 * checksum, chunking or transfer format; the definitions below are this
 * library's, written as plainly as possible.
 */
#include "oracle.h"

#include <stdlib.h>
#include <string.h>

/* ====================================================================== */
/* CRC                                                                     */
/* ====================================================================== */

/* One bit of the reflected shift register: the low bit leaves the register
 * and, if it was set, the reflected polynomial is XORed in. */
static uint32_t crc_shift_bit(uint32_t poly_reflected, uint32_t r) {
  if (r & 1u) return (r >> 1) ^ poly_reflected;
  return r >> 1;
}

uint32_t or_crc_bitwise(uint32_t poly_reflected, uint32_t init, uint32_t xorout,
                        const uint8_t* p, uint64_t n) {
  uint32_t r = init;
  for (uint64_t i = 0; i < n; ++i) {
    r ^= (uint32_t)p[i]; /* reflected input: bit 0 of the byte enters first */
    for (int k = 0; k < 8; ++k) r = crc_shift_bit(poly_reflected, r);
  }
  return r ^ xorout;
}

/* table[b] = register after shifting the byte value b through eight bit
 * steps from a zero register. */
static void crc_make_table(uint32_t poly_reflected, uint32_t table[256]) {
  for (uint32_t b = 0; b < 256; ++b) {
    uint32_t r = b;
    for (int k = 0; k < 8; ++k) r = crc_shift_bit(poly_reflected, r);
    table[b] = r;
  }
}

static uint32_t crc_table_run(const uint32_t table[256], uint32_t r,
                              const uint8_t* p, uint64_t n) {
  for (uint64_t i = 0; i < n; ++i) r = table[(r ^ p[i]) & 0xFFu] ^ (r >> 8);
  return r;
}

uint32_t or_crc_table(uint32_t poly_reflected, uint32_t init, uint32_t xorout,
                      const uint8_t* p, uint64_t n) {
  uint32_t table[256];
  crc_make_table(poly_reflected, table);
  return crc_table_run(table, init, p, n) ^ xorout;
}

/* The CRC register is linear over GF(2) in (register, data).  Writing
 * Adv(r, n) for "run n zero bytes through register r" and F for the preset
 * (= final XOR):
 *   crc(A||B) = Adv(crc(A) ^ F, |B|) ^ Raw(B) ^ F
 *   crc(B)    = Adv(F, |B|)          ^ Raw(B) ^ F
 * so crc(A||B) = Adv(crc(A), |B|) ^ crc(B).  The zero bytes are run one at a
 * time: O(|B|), which is all a reference needs. */
uint32_t or_crc_combine(uint32_t poly_reflected, uint32_t crc_a, uint32_t crc_b,
                        uint64_t len_b) {
  uint32_t table[256];
  crc_make_table(poly_reflected, table);
  uint32_t r = crc_a;
  for (uint64_t i = 0; i < len_b; ++i) r = table[r & 0xFFu] ^ (r >> 8);
  return r ^ crc_b;
}

#define OR_CRC32C_POLY 0x82F63B78u

static uint32_t g_crc32c_table[256];
static int g_crc32c_ready = 0;

uint32_t or_crc32c(const uint8_t* p, uint64_t n) {
  if (!g_crc32c_ready) {
    crc_make_table(OR_CRC32C_POLY, g_crc32c_table);
    g_crc32c_ready = 1;
  }
  return crc_table_run(g_crc32c_table, 0xFFFFFFFFu, p, n) ^ 0xFFFFFFFFu;
}

uint32_t or_crc32c_combine(uint32_t crc_a, uint32_t crc_b, uint64_t len_b) {
  return or_crc_combine(OR_CRC32C_POLY, crc_a, crc_b, len_b);
}

/* ====================================================================== */
/* Fingerprint values                                                      */
/* ====================================================================== */

static uint32_t load_le32(const uint8_t* p) {
  return (uint32_t)p[0] | ((uint32_t)p[1] << 8) | ((uint32_t)p[2] << 16) |
         ((uint32_t)p[3] << 24);
}

static uint16_t load_le16(const uint8_t* p) {
  return (uint16_t)((uint32_t)p[0] | ((uint32_t)p[1] << 8));
}

static float float_from_bits(uint32_t bits) {
  float f;
  memcpy(&f, &bits, sizeof f);
  return f;
}

/* An element is non-finite when its exponent field is all ones (Inf, NaN). */
void or_fp_values(const uint8_t* p, uint64_t len, uint32_t dtype,
                  uint32_t* nonfinite, double* sumsq) {
  uint32_t bad = 0;
  double s = 0.0;
  if (dtype == OR_DT_F32) {
    for (uint64_t i = 0; i + 4 <= len; i += 4) {
      uint32_t bits = load_le32(p + i);
      if ((bits & 0x7F800000u) == 0x7F800000u) {
        bad += 1;
      } else {
        double x = (double)float_from_bits(bits);
        s = s + x * x; /* the product of two 24-bit significands is exact */
      }
    }
  } else if (dtype == OR_DT_BF16) {
    for (uint64_t i = 0; i + 2 <= len; i += 2) {
      uint16_t bits = load_le16(p + i);
      if ((bits & 0x7F80u) == 0x7F80u) {
        bad += 1;
      } else {
        /* bf16 is the upper half of an IEEE binary32 */
        double x = (double)float_from_bits((uint32_t)bits << 16);
        s = s + x * x;
      }
    }
  }
  *nonfinite = bad;
  *sumsq = s;
}

void or_fingerprint_chunk(const uint8_t* p, uint64_t len, uint32_t dtype, or_fp* out) {
  out->crc32c = or_crc32c(p, len);
  or_fp_values(p, len, dtype, &out->nonfinite, &out->sumsq);
}

/* ====================================================================== */
/* Plan and packed layout                                                  */
/* ====================================================================== */

static uint64_t align_up(uint64_t v, uint64_t a) { return (v + a - 1) / a * a; }

static uint64_t elem_bytes(uint32_t dtype) {
  if (dtype == OR_DT_F32) return 4;
  if (dtype == OR_DT_BF16) return 2;
  return 1;
}

/* Packed buffer:
 *   [C x 64-byte header table][zero gap up to a 256-byte boundary]
 *   then, per chunk in id order, its payload at a 256-byte-aligned offset
 *   followed by zero padding up to the next 256-byte boundary. */
uint64_t or_plan(const uint64_t* nbytes, const uint32_t* dtypes, uint64_t n_tensors,
                 uint64_t chunk_bytes, or_chunk* out, uint64_t cap,
                 uint64_t* packed_bytes) {
  if (chunk_bytes == 0 || chunk_bytes % 4 != 0) return UINT64_MAX;
  uint64_t count = 0;
  for (uint64_t t = 0; t < n_tensors; ++t) {
    if (dtypes[t] > OR_DT_F32) return UINT64_MAX;
    if (nbytes[t] % elem_bytes(dtypes[t]) != 0) return UINT64_MAX;
    count += (nbytes[t] + chunk_bytes - 1) / chunk_bytes;
  }
  uint64_t off = align_up(count * OR_HEADER_BYTES, OR_PAYLOAD_ALIGN);
  uint64_t c = 0;
  for (uint64_t t = 0; t < n_tensors; ++t) {
    for (uint64_t start = 0; start < nbytes[t]; start += chunk_bytes) {
      uint64_t len = nbytes[t] - start;
      if (len > chunk_bytes) len = chunk_bytes;
      if (out != 0 && c < cap) {
        out[c].tensor_idx = (uint32_t)t;
        out[c].dtype = dtypes[t];
        out[c].tensor_off = start;
        out[c].len = len;
        out[c].payload_off = off;
      }
      off += align_up(len, OR_PAYLOAD_ALIGN);
      c += 1;
    }
  }
  if (packed_bytes != 0) *packed_bytes = off;
  return count;
}

static void store_le16(uint8_t* p, uint32_t v) {
  p[0] = (uint8_t)v;
  p[1] = (uint8_t)(v >> 8);
}
static void store_le32(uint8_t* p, uint32_t v) {
  for (int i = 0; i < 4; ++i) p[i] = (uint8_t)(v >> (8 * i));
}
static void store_le64(uint8_t* p, uint64_t v) {
  for (int i = 0; i < 8; ++i) p[i] = (uint8_t)(v >> (8 * i));
}
static uint64_t load_le64(const uint8_t* p) {
  uint64_t v = 0;
  for (int i = 0; i < 8; ++i) v |= (uint64_t)p[i] << (8 * i);
  return v;
}

/* Header fields (little-endian):
 *    0 u32 magic          4 u16 version      6 u16 dtype
 *    8 u64 chunk_id      16 u32 tensor_idx  20 u32 payload_crc
 *   24 u64 tensor_off    32 u64 len         40 u64 payload_off
 *   48 f64 sumsq         56 u32 nonfinite   60 u32 header_crc
 * header_crc is the CRC-32C of bytes [0, 60). */
void or_header(const or_chunk* ch, uint64_t chunk_id, const or_fp* fp, uint8_t h[64]) {
  memset(h, 0, 64);
  store_le32(h + 0, OR_MAGIC);
  store_le16(h + 4, OR_VERSION);
  store_le16(h + 6, ch->dtype);
  store_le64(h + 8, chunk_id);
  store_le32(h + 16, ch->tensor_idx);
  store_le32(h + 20, fp->crc32c);
  store_le64(h + 24, ch->tensor_off);
  store_le64(h + 32, ch->len);
  store_le64(h + 40, ch->payload_off);
  uint64_t sbits;
  memcpy(&sbits, &fp->sumsq, 8);
  store_le64(h + 48, sbits);
  store_le32(h + 56, fp->nonfinite);
  store_le32(h + 60, or_crc32c(h, 60));
}

/* ====================================================================== */
/* Whole-state calls                                                       */
/* ====================================================================== */

static or_chunk* plan_alloc(const uint64_t* nbytes, const uint32_t* dtypes,
                            uint64_t n_tensors, uint64_t chunk_bytes,
                            uint64_t* count, uint64_t* packed_bytes) {
  uint64_t c = or_plan(nbytes, dtypes, n_tensors, chunk_bytes, 0, 0, packed_bytes);
  if (c == UINT64_MAX) return 0;
  or_chunk* chunks = (or_chunk*)malloc((size_t)(c ? c : 1) * sizeof(or_chunk));
  if (chunks == 0) return 0;
  or_plan(nbytes, dtypes, n_tensors, chunk_bytes, chunks, c, packed_bytes);
  *count = c;
  return chunks;
}

int or_fingerprint(const uint8_t* const* tensors, const uint64_t* nbytes,
                   const uint32_t* dtypes, uint64_t n_tensors, uint64_t chunk_bytes,
                   or_fp* out) {
  uint64_t count, packed;
  or_chunk* chunks = plan_alloc(nbytes, dtypes, n_tensors, chunk_bytes, &count, &packed);
  if (chunks == 0) return OR_ERR_INVALID_ARG;
  for (uint64_t c = 0; c < count; ++c) {
    const uint8_t* p = tensors[chunks[c].tensor_idx] + chunks[c].tensor_off;
    or_fingerprint_chunk(p, chunks[c].len, chunks[c].dtype, &out[c]);
  }
  free(chunks);
  return OR_OK;
}

int or_pack(const uint8_t* const* tensors, const uint64_t* nbytes,
            const uint32_t* dtypes, uint64_t n_tensors, uint64_t chunk_bytes,
            uint8_t* dst, uint64_t dst_bytes) {
  uint64_t count, packed;
  or_chunk* chunks = plan_alloc(nbytes, dtypes, n_tensors, chunk_bytes, &count, &packed);
  if (chunks == 0) return OR_ERR_INVALID_ARG;
  if (dst_bytes < packed) {
    free(chunks);
    return OR_ERR_BUFFER_TOO_SMALL;
  }
  memset(dst, 0, (size_t)packed); /* every unused byte is zero */
  for (uint64_t c = 0; c < count; ++c) {
    const uint8_t* p = tensors[chunks[c].tensor_idx] + chunks[c].tensor_off;
    or_fp fp;
    or_fingerprint_chunk(p, chunks[c].len, chunks[c].dtype, &fp);
    or_header(&chunks[c], c, &fp, dst + c * OR_HEADER_BYTES);
    memcpy(dst + chunks[c].payload_off, p, (size_t)chunks[c].len);
  }
  free(chunks);
  return OR_OK;
}

/* The checks of unpack_verify on one chunk: the header CRC, every addressing
 * field against the receiver's own plan, the payload CRC, the zero padding,
 * and (last chunk only) the zero gap after the header table.  Returns 1 if
 * any check fails. */
int or_verify_chunk(const or_chunk* ch, uint64_t chunk_id, const uint8_t* h,
                    const uint8_t* payload, const uint8_t* gap, uint64_t gap_len) {
  int bad = 0;
  /* 1. the header protects itself */
  if (load_le32(h + 60) != or_crc32c(h, 60)) bad = 1;
  /* 2. every addressing field must equal the receiver's own plan */
  if (load_le32(h + 0) != OR_MAGIC) bad = 1;
  if (load_le16(h + 4) != OR_VERSION) bad = 1;
  if (load_le16(h + 6) != ch->dtype) bad = 1;
  if (load_le64(h + 8) != chunk_id) bad = 1;
  if (load_le32(h + 16) != ch->tensor_idx) bad = 1;
  if (load_le64(h + 24) != ch->tensor_off) bad = 1;
  if (load_le64(h + 32) != ch->len) bad = 1;
  if (load_le64(h + 40) != ch->payload_off) bad = 1;
  /* 3. the payload must match the CRC the header carries */
  if (or_crc32c(payload, ch->len) != load_le32(h + 20)) bad = 1;
  /* 4. the padding after the payload must be zero */
  uint64_t pad_end = align_up(ch->len, OR_PAYLOAD_ALIGN);
  for (uint64_t i = ch->len; i < pad_end; ++i)
    if (payload[i] != 0) bad = 1;
  /* the gap after the header table (passed for the last chunk only) */
  for (uint64_t i = 0; i < gap_len; ++i)
    if (gap[i] != 0) bad = 1;
  return bad;
}

int or_unpack_verify(uint8_t* const* tensors, const uint64_t* nbytes,
                     const uint32_t* dtypes, uint64_t n_tensors, uint64_t chunk_bytes,
                     const uint8_t* src, uint64_t src_bytes,
                     uint32_t* mismatch, uint64_t cap, uint64_t* n_mismatch) {
  uint64_t count, packed;
  or_chunk* chunks = plan_alloc(nbytes, dtypes, n_tensors, chunk_bytes, &count, &packed);
  if (chunks == 0) return OR_ERR_INVALID_ARG;
  if (src_bytes < packed) {
    free(chunks);
    return OR_ERR_BUFFER_TOO_SMALL;
  }
  uint64_t gap_begin = count * OR_HEADER_BYTES;
  uint64_t gap_end = align_up(count * OR_HEADER_BYTES, OR_PAYLOAD_ALIGN);
  uint64_t found = 0;
  for (uint64_t c = 0; c < count; ++c) {
    const or_chunk* ch = &chunks[c];
    const uint8_t* payload = src + ch->payload_off;
    /* the gap after the header table belongs to the last chunk */
    int last = (c + 1 == count);
    int bad = or_verify_chunk(ch, c, src + c * OR_HEADER_BYTES, payload,
                              last ? src + gap_begin : 0, last ? gap_end - gap_begin : 0);

    /* the payload is copied to the plan's destination whatever the verdict */
    memcpy(tensors[ch->tensor_idx] + ch->tensor_off, payload, (size_t)ch->len);

    if (bad) {
      if (found < cap) mismatch[found] = (uint32_t)c;
      found += 1;
    }
  }
  *n_mismatch = found;
  free(chunks);
  return OR_OK;
}

uint64_t or_diff(const or_fp* a, const or_fp* b, uint64_t n, uint32_t* out, uint64_t cap) {
  uint64_t found = 0;
  for (uint64_t c = 0; c < n; ++c) {
    if (memcmp(&a[c], &b[c], sizeof(or_fp)) != 0) {
      if (found < cap) out[found] = (uint32_t)c;
      found += 1;
    }
  }
  return found;
}
