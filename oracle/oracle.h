/*
 * oracle.h -- plain, slow, single-threaded CPU reference ("the oracle").
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may include, link or
 * call this code: only tests/, __graft_entry__.smoke() and bench.py's
 * cpu_baseline leg / reference arm use it.  It shares no code, tables,
 * headers or constants generators with the CUDA library under
 * paper_2509_03047_gb300/csrc/.
 *
 * What it computes.  FlashRecovery (arXiv 2509.03047) restores a restarted
 * rank's model and optimizer state from a healthy data-parallel replica
 * instead of from a checkpoint (Sec. III-E, "Model states Restoration", and
 * the vanilla-DP panel of the restoration figure).  The paper says only that
 * the states are moved "with collective communication"; it defines no
 * checksum, chunking or transfer format.  The oracle therefore states, in the
 * plainest possible code, the four per-chunk operations of the restoration
 * sweep as this library defines them:
 *
 *   fingerprint   per chunk: CRC-32C of its bytes, count of non-finite
 *                 elements, fp64 sum of squares of the finite elements;
 *   pack          chunk headers + 256-byte-aligned payloads in one buffer;
 *   unpack_verify scatter payloads back, list chunks that fail verification;
 *   diff          list chunks whose fingerprints differ.
 *
 * CRC-32C is the Castagnoli polynomial 0x1EDC6F41 (reflected 0x82F63B78),
 * reflected input and output, register preset 0xFFFFFFFF, final XOR
 * 0xFFFFFFFF (Castagnoli, IEEE Trans. Commun. 41(6), 1993; the variant
 * catalogued as CRC-32/ISCSI).
 *
 * Every function here follows its definition step by step, in address order,
 * with no blocking, fusion or reordering.
 */
#ifndef FLASHREC_ORACLE_H
#define FLASHREC_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Element types of a tensor (same numbering as the library's, restated). */
enum { OR_DT_BYTES = 0, OR_DT_BF16 = 1, OR_DT_F32 = 2 };

/* Status codes of the oracle's whole-buffer calls. */
enum { OR_OK = 0, OR_ERR_INVALID_ARG = 1, OR_ERR_BUFFER_TOO_SMALL = 3 };

/* One fingerprint entry: 16 bytes, no padding. */
typedef struct {
  uint32_t crc32c;
  uint32_t nonfinite;
  double sumsq;
} or_fp;

/* One chunk of the plan. */
typedef struct {
  uint32_t tensor_idx;
  uint32_t dtype;
  uint64_t tensor_off;  /* byte offset of the chunk inside its tensor */
  uint64_t len;         /* chunk bytes                                  */
  uint64_t payload_off; /* byte offset of the payload in the packed buffer */
} or_chunk;

#define OR_HEADER_BYTES 64u
#define OR_PAYLOAD_ALIGN 256u
#define OR_MAGIC 0x31435246u /* the bytes 'F','R','C','1' read little-endian */
#define OR_VERSION 1u

/* ---------------- CRC ---------------- */

/* Bit-at-a-time CRC straight from the shift-register definition, for any
 * reflected polynomial, preset and final XOR. */
uint32_t or_crc_bitwise(uint32_t poly_reflected, uint32_t init, uint32_t xorout,
                        const uint8_t* p, uint64_t n);

/* Byte-at-a-time (Sarwate) CRC for any reflected polynomial; the 256-entry
 * table is generated from the polynomial on every call. */
uint32_t or_crc_table(uint32_t poly_reflected, uint32_t init, uint32_t xorout,
                      const uint8_t* p, uint64_t n);

/* CRC of A||B from crc(A), crc(B) and |B|, for a CRC whose preset equals its
 * final XOR: advance crc(A) through |B| zero bytes, then XOR crc(B). */
uint32_t or_crc_combine(uint32_t poly_reflected, uint32_t crc_a, uint32_t crc_b,
                        uint64_t len_b);

/* CRC-32C with the standard parameters (table-driven). */
uint32_t or_crc32c(const uint8_t* p, uint64_t n);
uint32_t or_crc32c_combine(uint32_t crc_a, uint32_t crc_b, uint64_t len_b);

/* ---------------- per-chunk fingerprint ---------------- */

/* Non-finite count and fp64 sum of squares of the finite elements, in
 * address order.  OR_DT_BYTES gives 0 and 0.0. */
void or_fp_values(const uint8_t* p, uint64_t len, uint32_t dtype,
                  uint32_t* nonfinite, double* sumsq);
void or_fingerprint_chunk(const uint8_t* p, uint64_t len, uint32_t dtype, or_fp* out);

/* ---------------- plan ---------------- */

/* Chunks of tensor t are [k*chunk_bytes, min((k+1)*chunk_bytes, nbytes_t)),
 * k = 0.. ; tensor order, then offset.  Writes at most `cap` chunks to `out`
 * (may be NULL) and the packed buffer size to *packed_bytes (may be NULL).
 * Returns the number of chunks, or UINT64_MAX on invalid arguments. */
uint64_t or_plan(const uint64_t* nbytes, const uint32_t* dtypes, uint64_t n_tensors,
                 uint64_t chunk_bytes, or_chunk* out, uint64_t cap,
                 uint64_t* packed_bytes);

/* The 64-byte header of chunk `chunk_id`. */
void or_header(const or_chunk* ch, uint64_t chunk_id, const or_fp* fp, uint8_t h[64]);

/* ---------------- whole-state calls ---------------- */

int or_fingerprint(const uint8_t* const* tensors, const uint64_t* nbytes,
                   const uint32_t* dtypes, uint64_t n_tensors, uint64_t chunk_bytes,
                   or_fp* out);

int or_pack(const uint8_t* const* tensors, const uint64_t* nbytes,
            const uint32_t* dtypes, uint64_t n_tensors, uint64_t chunk_bytes,
            uint8_t* dst, uint64_t dst_bytes);

/* The verdict of unpack_verify for one chunk: 1 if it fails any check.
 *   ch, chunk_id  the receiver's own plan entry for the chunk;
 *   h             the chunk's 64-byte header in the packed buffer;
 *   payload       its payload followed by its zero padding
 *                 (ch->len rounded up to OR_PAYLOAD_ALIGN bytes);
 *   gap, gap_len  the zero gap between the header table and the first
 *                 payload, which belongs to the last chunk: pass it for the
 *                 last chunk only (else NULL, 0). */
int or_verify_chunk(const or_chunk* ch, uint64_t chunk_id, const uint8_t* h,
                    const uint8_t* payload, const uint8_t* gap, uint64_t gap_len);

/* Always copies every payload to its plan destination; lists, ascending,
 * the chunks that fail any check.  *n_mismatch gets the true count; at most
 * `cap` ids are written. */
int or_unpack_verify(uint8_t* const* tensors, const uint64_t* nbytes,
                     const uint32_t* dtypes, uint64_t n_tensors, uint64_t chunk_bytes,
                     const uint8_t* src, uint64_t src_bytes,
                     uint32_t* mismatch, uint64_t cap, uint64_t* n_mismatch);

/* Chunks whose 16-byte fingerprint entries differ in any bit, ascending.
 * Returns the true count; at most `cap` ids are written. */
uint64_t or_diff(const or_fp* a, const or_fp* b, uint64_t n, uint32_t* out, uint64_t cap);

#ifdef __cplusplus
}
#endif

#endif
