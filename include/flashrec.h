/*
 * flashrec.h -- C ABI of libflashrec, the GB300 (sm_103a) restoration sweep.
 *
 * FlashRecovery (arXiv 2509.03047) restores a restarted rank's model and
 * optimizer state from a healthy data-parallel replica's memory instead of
 * from a checkpoint (Sec. III-E, "Model states Restoration"; vanilla-DP panel
 * of the restoration figure).  The paper moves the state "with collective
 * communication" and defines no checksum or transfer format.  This library is
 * the device-side sweep over one rank's state that such a restoration needs:
 *
 *   fr_fingerprint    per-chunk CRC-32C, non-finite count, fp64 sum of squares
 *   fr_pack           tensors -> one flat transfer buffer with chunk headers
 *   fr_unpack_verify  transfer buffer -> tensors, list of failing chunks
 *   fr_diff           chunks whose fingerprints differ
 *
 * All device work runs in hand-written CUDA kernels for sm_103a.  There is no
 * CPU fallback: without a usable GPU every call returns FR_ERR_CUDA.
 *
 * Conventions
 *   - Chunks are per tensor: chunk k of tensor t covers bytes
 *     [k*chunk_bytes, min((k+1)*chunk_bytes, nbytes_t)).  Chunk ids are global
 *     and ascending in tensor order, then offset.  A 0-byte tensor has no chunk.
 *   - CRC-32C: polynomial 0x1EDC6F41 (reflected 0x82F63B78), reflected in and
 *     out, preset 0xFFFFFFFF, final XOR 0xFFFFFFFF (CRC-32/ISCSI).
 *   - An element is non-finite when its exponent field is all ones.  sumsq is
 *     the sum of x*x over the finite elements, accumulated in fp64; it agrees
 *     with a sequential fp64 sum to within 1e-9 relative and is bit-for-bit
 *     reproducible from run to run on the same GPU.
 *   - Every device call is asynchronous and ordered on `stream` (a
 *     cudaStream_t passed as void*; NULL is the legacy default stream).
 *     Argument errors are returned synchronously and enqueue nothing.
 *     Conditions found on the device (list overflow) are recorded in the plan
 *     and returned by fr_sync_status().
 *   - Pointers named *_dev are device memory (or any memory the GPU can
 *     address through unified virtual addressing, such as pinned host memory).
 *     The caller owns every tensor, buffer and output; the library owns only
 *     the plan and what the plan allocates when it is created.  No call after
 *     fr_plan_create allocates memory.
 *   - Thread safety: a plan may be used by one stream at a time.  Calls on
 *     one plan whose kernels overlap on the GPU (the same plan on two streams
 *     with no ordering between them) race on the plan's scratch -- per-piece
 *     records, segment sums and the counters through which pack and unpack
 *     warps share their last work units -- and give wrong results.  (The
 *     batched calls of a batched plan have their own counters per batch.)
 */
#ifndef FLASHREC_H
#define FLASHREC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FR_OK = 0,
  FR_ERR_INVALID_ARG = 1,      /* a null pointer, bad dtype, size or chunk size  */
  FR_ERR_ALIGNMENT = 2,        /* the packed buffer is not 16-byte aligned       */
  FR_ERR_BUFFER_TOO_SMALL = 3, /* the packed buffer is shorter than the plan's   */
  FR_ERR_CAPACITY = 4,         /* more ids than the list holds (true count kept) */
  FR_ERR_PLAN_MISMATCH = 5,    /* a table length that differs from the plan's    */
  FR_ERR_DEVICE_TIMEOUT = 6,   /* a bounded device-side wait gave up             */
  FR_ERR_CUDA = 7              /* a CUDA runtime error; see fr_last_error()      */
} fr_status;

typedef enum {
  FR_DT_BYTES = 0, /* opaque bytes: CRC only, nonfinite = 0, sumsq = 0 */
  FR_DT_BF16 = 1,
  FR_DT_F32 = 2
} fr_dtype;

/* One tensor of the state: `nbytes` bytes of device memory at `ptr`
 * (any alignment; 16-byte-aligned tensors take the fast path).  nbytes must
 * be a multiple of the element size.  `flags` must be 0. */
typedef struct {
  void* ptr;
  uint64_t nbytes;
  uint32_t dtype;
  uint32_t flags;
} fr_tensor;

/* One fingerprint table entry: 16 bytes, no padding. */
typedef struct {
  uint32_t crc32c;    /* CRC-32C of the chunk's bytes                 */
  uint32_t nonfinite; /* elements whose exponent field is all ones     */
  double sumsq;       /* sum of squares of the finite elements (fp64)  */
} fr_fp;

typedef struct fr_plan_s* fr_plan;

/* ---------------------------------------------------------------- plans */

/* Build a plan over `n_tensors` tensors (host array, copied) with chunks of
 * `chunk_bytes` (a positive multiple of 4).  The plan is bound to the current
 * CUDA device and to the tensors' addresses; it allocates its device tables
 * and scratch here and nowhere else.  Host-side planning is O(tensors +
 * chunks).  Errors: FR_ERR_INVALID_ARG, FR_ERR_CUDA. */
fr_status fr_plan_create(const fr_tensor* tensors, uint64_t n_tensors, uint64_t chunk_bytes,
                         fr_plan* out);

/* Chunk count, packed buffer size and total state bytes of a plan (host). */
fr_status fr_plan_info(fr_plan plan, uint64_t* n_chunks, uint64_t* packed_bytes,
                       uint64_t* state_bytes);

/* Where chunk `chunk_id` lives (host query): its tensor, byte offset in the
 * tensor, length, and payload offset in the packed buffer. */
fr_status fr_plan_chunk(fr_plan plan, uint64_t chunk_id, uint32_t* tensor_idx,
                        uint64_t* tensor_off, uint64_t* len, uint64_t* payload_off);

/* Free the plan and its device memory (synchronizes the device first). */
void fr_plan_destroy(fr_plan plan);

/* ---------------------------------------------------------------- sweep */

/* Fingerprint every chunk of the plan's tensors into `out_dev`, an array of
 * n_chunks fr_fp entries.  Restoration step of Sec. III-E: the table a healthy
 * replica and a restored rank compare.  Reads the state once. */
fr_status fr_fingerprint(fr_plan plan, fr_fp* out_dev, void* stream);

/* Gather the plan's tensors into the transfer buffer `dst` (device memory or
 * pinned host memory; 16-byte aligned; at least packed_bytes long), the
 * replica side of the Sec. III-E restoration.  Layout (little-endian):
 *   [n_chunks x 64-byte headers][zero bytes to a 256-byte boundary]
 *   then each chunk's payload at a 256-byte-aligned offset, zero-padded to
 *   the next 256-byte boundary.
 * Header: 0 u32 magic 'FRC1' | 4 u16 version 1 | 6 u16 dtype | 8 u64 chunk_id
 *   | 16 u32 tensor_idx | 20 u32 payload_crc | 24 u64 tensor_off | 32 u64 len
 *   | 40 u64 payload_off | 48 f64 sumsq | 56 u32 nonfinite
 *   | 60 u32 header_crc = CRC-32C of bytes [0,60).
 * Every byte of [0, packed_bytes) is written.
 * Errors: FR_ERR_INVALID_ARG, FR_ERR_ALIGNMENT, FR_ERR_BUFFER_TOO_SMALL, FR_ERR_CUDA. */
fr_status fr_pack(fr_plan plan, void* dst, uint64_t dst_bytes, void* stream);

/* Scatter the transfer buffer `src` (device or pinned host; 16-byte aligned)
 * into the plan's tensors, the restarted-rank side of Sec. III-E.  Every
 * payload is copied to the address the receiver's own plan gives (a header is
 * never trusted for addressing).  A chunk is listed when its header CRC is
 * wrong, any header field differs from the plan (magic, version, dtype,
 * chunk_id, tensor_idx, tensor_off, len, payload_off), its payload CRC-32C
 * differs from the header's payload_crc, or a padding byte after its payload
 * is non-zero (the zero bytes after the header table belong to the last
 * chunk).  The ids go to `mismatch_dev` in ascending order, at most `cap` of
 * them; the true count goes to *n_mismatch_dev (device u64).  When the count
 * exceeds `cap` the plan records FR_ERR_CAPACITY for fr_sync_status().
 * Errors: FR_ERR_INVALID_ARG, FR_ERR_ALIGNMENT, FR_ERR_BUFFER_TOO_SMALL, FR_ERR_CUDA. */
fr_status fr_unpack_verify(fr_plan plan, const void* src, uint64_t src_bytes,
                           uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev,
                           void* stream);

/* Chunks whose 16-byte table entries differ in any bit (crc32c, nonfinite, or
 * the bit pattern of sumsq) between `a_dev` and `b_dev`, both n_chunks long.
 * Ascending ids, at most `cap`, to `diverged_dev`; the true count to
 * *n_out_dev (device u64).  Overflow is visible as count > cap.
 * Errors: FR_ERR_INVALID_ARG, FR_ERR_CUDA. */
fr_status fr_diff(const fr_fp* a_dev, const fr_fp* b_dev, uint64_t n_chunks,
                  uint32_t* diverged_dev, uint64_t cap, uint64_t* n_out_dev, void* stream);

/* ---------------------------------------------------------------- fused fingerprints */

/* A restoration usually wants both fingerprints -- of the replica's state
 * and of the restored state -- to confirm with fr_diff that they agree.
 * Pack already computes every fingerprint field of every chunk for its
 * headers, and unpack reads every restored byte, so these variants also
 * write the fingerprint table on the same pass, saving the two separate
 * fr_fingerprint sweeps (half the device traffic of a restore).
 *
 * fr_pack_fp: fr_pack, plus `fp_dev` (n_chunks fr_fp entries, 16-byte
 * aligned, or NULL for none) receives exactly what fr_fingerprint writes for
 * the plan's tensors.
 * fr_unpack_verify_fp: fr_unpack_verify, plus `fp_dev` (or NULL) receives the
 * fingerprint of the restored tensors -- exactly what fr_fingerprint would
 * write for them afterwards, failing chunks included (their bytes are written
 * as received).
 * fr_restore_fp: fr_restore, plus the replica's table in `fp_src_dev` and the
 * restored state's table in `fp_dst_dev` (either may be NULL); chunks sent
 * again by a retry get their entries rewritten.  `fp_src_dev` is complete once
 * `stream_src` reaches the end of the call's work, `fp_dst_dev` once
 * `stream_dst` does (the call orders the former before the latter).
 * fr_resend_fp: fr_resend, plus the re-sent chunks' entries rewritten in
 * `fp_src_dev` and `fp_dst_dev` (either may be NULL).
 * Errors: as the calls they extend. */
fr_status fr_pack_fp(fr_plan plan, void* dst, uint64_t dst_bytes, fr_fp* fp_dev, void* stream);
fr_status fr_unpack_verify_fp(fr_plan plan, const void* src, uint64_t src_bytes, uint32_t* mismatch_dev, uint64_t cap,
                              uint64_t* n_mismatch_dev, fr_fp* fp_dev, void* stream);
fr_status fr_restore_fp(fr_plan src, fr_plan dst, void* staging, uint64_t staging_bytes, uint32_t max_retries,
                        uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev, fr_fp* fp_src_dev,
                        fr_fp* fp_dst_dev, void* stream_src, void* stream_dst);
fr_status fr_resend_fp(fr_plan src, fr_plan dst, void* staging, uint64_t staging_bytes, uint64_t* n_resent,
                       fr_fp* fp_src_dev, fr_fp* fp_dst_dev, void* stream_src, void* stream_dst);

/* ---------------------------------------------------------------- streamed restore */

/* The transfer of Sec. III-E end to end: a healthy replica's state reaches a
 * restarted rank through a transfer buffer, typically pinned host memory
 * reached over NVLink-C2C.  A whole-buffer fr_pack followed by
 * fr_unpack_verify uses one direction of that link at a time; the calls below
 * split the chunks into batches so the replica packs batch b+1 while the
 * rank unpacks batch b, and re-send only the chunks that fail verification.
 *
 * fr_plan_create_batched is fr_plan_create plus a split of the chunks into
 * `n_batches` consecutive batches of about equal bytes (at most one per
 * chunk).  Batch calls run on half the SMs, so a pack on one stream and an
 * unpack on another share the GPU.  Whole-state calls on a batched plan behave
 * exactly as on a plain one.  fr_plan_batch reports the batch count and a
 * batch's chunk range. */
fr_status fr_plan_create_batched(const fr_tensor* tensors, uint64_t n_tensors, uint64_t chunk_bytes,
                                 uint32_t n_batches, fr_plan* out);
fr_status fr_plan_batch(fr_plan plan, uint32_t batch, uint32_t* n_batches, uint64_t* first_chunk,
                        uint64_t* n_chunks);

/* fr_pack / fr_unpack_verify restricted to one batch: the same bytes of the
 * same packed layout (headers, payloads and padding of the batch's chunks;
 * the table gap with the batch that holds the last chunk).  An unpacked
 * batch only records its verdicts; fr_unpack_collect then lists the failing
 * chunks of the plan's latest verdicts, exactly as fr_unpack_verify does. */
fr_status fr_pack_batch(fr_plan plan, uint32_t batch, void* dst, uint64_t dst_bytes, void* stream);
fr_status fr_unpack_verify_batch(fr_plan plan, uint32_t batch, const void* src, uint64_t src_bytes,
                                 void* stream);
fr_status fr_unpack_collect(fr_plan plan, uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev,
                            void* stream);

/* Re-send every chunk whose latest verdict in `dst` failed: re-pack it from
 * `src` into `staging` on `stream_src`, then re-unpack and re-verify it on
 * `stream_dst`.  Synchronizes `stream_dst` once to learn how many chunks fail
 * (*n_resent, may be NULL).  `src` and `dst` must describe the same layout
 * (else FR_ERR_PLAN_MISMATCH). */
fr_status fr_resend(fr_plan src, fr_plan dst, void* staging, uint64_t staging_bytes, uint64_t* n_resent,
                    void* stream_src, void* stream_dst);

/* The whole restoration: for every batch, pack it from `src` on `stream_src`
 * and, as soon as it is packed, unpack and verify it into `dst` on
 * `stream_dst`; then up to `max_retries` rounds of fr_resend (each
 * synchronizes `stream_dst` once); then list the chunks that still fail, as
 * fr_unpack_verify does.  All work is ordered before later work on
 * `stream_dst`.  With max_retries = 0 nothing synchronizes. */
fr_status fr_restore(fr_plan src, fr_plan dst, void* staging, uint64_t staging_bytes, uint32_t max_retries,
                     uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev, void* stream_src,
                     void* stream_dst);

/* Restoration from several healthy replicas at once, each sending a share of
 * the chunks (the partitioned form of the restore: with R replicas alive,
 * each packs about 1/R of the state).  Batch b of the plans is packed by
 * replica src[b % n_src] on streams_src[b % n_src] (streams_src may be NULL:
 * the legacy default stream for all) and unpacked and verified into `dst` on
 * `stream_dst` as soon as it is packed; retry round r re-sends the failing
 * chunks from replica r % n_src; then the still-failing chunks are listed as
 * fr_unpack_verify does.  `fp_dst_dev` (or NULL) receives the restored
 * state's fingerprint table.  Every source plan must describe the same layout
 * and batch count as `dst` (else FR_ERR_PLAN_MISMATCH).  Sources on distinct
 * streams pack concurrently; sharing a stream is correct, only serial.  All
 * work is ordered before later work on `stream_dst`.
 * Errors: FR_ERR_INVALID_ARG, FR_ERR_PLAN_MISMATCH, FR_ERR_ALIGNMENT,
 * FR_ERR_BUFFER_TOO_SMALL, FR_ERR_CUDA. */
fr_status fr_restore_multi(const fr_plan* src, uint32_t n_src, fr_plan dst, void* staging, uint64_t staging_bytes,
                           uint32_t max_retries, uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev,
                           fr_fp* fp_dst_dev, void* const* streams_src, void* stream_dst);

/* ---------------------------------------------------------------- sharded (ZeRO / FSDP) state */

/* With ZeRO / FSDP every data-parallel rank keeps only a shard of the
 * flattened model states (Sec. III-A; ZeRO/FSDP panel of the restoration
 * figure in Sec. III-E).  When the surviving copies are sharded another way
 * (another data-parallel degree, another ZeRO group), no single peer holds a
 * restarted rank's shard: it is assembled from pieces of several peers'
 * shards.
 *
 * Sharding rule: a flat group of `n_elems` elements of `elem_bytes` bytes
 * split `n` ways gives shard r the elements [r*q, min((r+1)*q, n_elems)),
 * q = ceil(n_elems / n); shards past the end are empty.  (ZeRO/FSDP pad the
 * group to a multiple of n; padding bytes are not model state and are not
 * moved.)
 *
 * fr_shard_pieces lists, in ascending order, where shard `rank` of the group
 * split `n_dst` ways lies among the shards of the same group split `n_src`
 * ways: for each piece the source shard, the byte offset in that source
 * shard, the byte offset in the destination shard and the byte count.  A
 * non-empty shard has between 1 and n_src pieces.  *n_pieces always receives
 * the true count; at most `cap` pieces are written, FR_ERR_CAPACITY if there
 * are more.  Host only: no device work.
 *
 * A plan over the pieces' source regions (tensors inside several peers'
 * shards) and a plan over their destination regions have the same layout, so
 * one fr_restore between them assembles the whole shard from all its
 * sources, and fr_fingerprint of both plans followed by fr_diff confirms that
 * the result matches every source.
 * Errors: FR_ERR_INVALID_ARG, FR_ERR_CAPACITY. */
typedef struct {
  uint32_t source;  /* source shard index, < n_src                */
  uint32_t reserved;
  uint64_t src_off; /* byte offset in the source shard             */
  uint64_t dst_off; /* byte offset in the destination shard        */
  uint64_t nbytes;  /* bytes in the piece (a multiple of elem_bytes) */
} fr_piece;
fr_status fr_shard_pieces(uint64_t n_elems, uint32_t elem_bytes, uint32_t n_dst, uint32_t rank, uint32_t n_src,
                          fr_piece* out, uint64_t cap, uint64_t* n_pieces);

/* ---------------------------------------------------------------- no allocation */

/* The paper has no counterpart to this call; it serves callers that cannot
 * allocate device memory.  A recovery agent living inside a training process
 * often finds every byte of the GPU reserved by the framework's allocator for
 * the model and optimizer state, and some callers may not call
 * cudaMalloc/cudaFree at all (their implicit device synchronization, or their
 * failure when memory is exhausted, would break the caller).  fr_plan_create
 * allocates, so such callers use this instead.
 *
 * fr_fingerprint_static computes exactly what fr_plan_create + fr_fingerprint
 * + fr_plan_destroy compute for the same tensors and chunk size, writing
 * n_chunks fr_fp entries to `out_dev`, but allocates nothing: its plan tables
 * and scratch live in one fixed array in the library's device memory (a few
 * MiB, held by every GPU that loads the library until the process exits), and
 * its host-side planning uses fixed static tables.
 *   - Limits: at most FR_STATIC_MAX_CHUNKS chunks, at most
 *     FR_STATIC_MAX_SEGMENTS 16 KiB segments of chunk bodies (2 GiB of state
 *     in large chunks), and GPUs of at most 160 SMs; larger inputs return
 *     FR_ERR_INVALID_ARG before any device work.
 *   - The first call on a device sets that device up (looks up the array's
 *     device address and configures the kernels), so make that first call
 *     before any stream capture.
 *   - Every call, on every stream, shares the one array and rewrites all of
 *     it that it uses; calls whose work overlaps on the GPU (calls on
 *     different streams with no ordering between them) race and give wrong
 *     results.  Host-side calls are serialized by a lock.
 *   - The table upload is a copy from pageable host memory, so the call
 *     returns only after the work already queued on `stream` has finished.
 *   - It cannot be captured into a CUDA graph (a replay would upload whatever
 *     tables the latest call left in the host buffer): on a stream under
 *     capture it returns FR_ERR_INVALID_ARG and enqueues nothing.
 * Errors: FR_ERR_INVALID_ARG (also for sizes beyond the limit, or a stream
 * under capture), FR_ERR_CUDA. */
#define FR_STATIC_MAX_CHUNKS 16384
#define FR_STATIC_MAX_SEGMENTS 131072
fr_status fr_fingerprint_static(const fr_tensor* tensors, uint64_t n_tensors, uint64_t chunk_bytes,
                                fr_fp* out_dev, void* stream);

/* ---------------------------------------------------------------- status */

/* Synchronize `stream`, then return and clear the first condition the plan's
 * kernels recorded (FR_ERR_CAPACITY or FR_ERR_DEVICE_TIMEOUT), else FR_OK. */
fr_status fr_sync_status(fr_plan plan, void* stream);

/* A static string naming a status code. */
const char* fr_status_str(fr_status status);

/* The message of the last FR_ERR_CUDA / FR_ERR_INVALID_ARG seen by the
 * calling thread ("" if none). */
const char* fr_last_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int fr_version(void);

#ifdef __cplusplus
}
#endif

#endif /* FLASHREC_H */
