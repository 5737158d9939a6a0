// kernels.h -- launchers of the device kernels (internal to libflashrec).
#pragma once

#include <cstdint>

#include <cuda_runtime.h>

#include "layout.h"
#include "../../include/flashrec.h"

namespace frk {

// Sweep modes.  kModeUnpackFp is unpack + verify that also computes the
// fingerprint values (non-finite count, sum of squares) of the restored bytes
// on the same pass, so a restore needs no separate fingerprint sweep.
enum : int { kModeFingerprint = 0, kModePack = 1, kModeUnpack = 2, kModeUnpackFp = 3 };
// Direction: the packed buffer is the source.
__host__ __device__ constexpr bool mode_unpacks(int m) { return m == kModeUnpack || m == kModeUnpackFp; }
// Whether the mode computes non-finite counts and sums of squares.
__host__ __device__ constexpr bool mode_sums(int m) { return m != kModeUnpack; }

struct SweepParams {
  const ChunkDesc* chunks;
  const WarpDesc* warps;  // this class's per-warp ranges
  const uint32_t* class_chunks;  // ids of this class's chunks with a body, in order
  Record* recs;
  double* segs;           // segment sums of squares (all modes but kModeUnpack)
  uint8_t* packed;        // pack: destination; unpack: source; fingerprint: unused
  uint32_t n_warps;       // warps with a descriptor
  // Mixed launches: per sweep class c, n_units[c] work units at
  // units + unit_off[c] (block order), claimed at run time by warps that have
  // finished their own range, and list_off[c], where the class's chunk list
  // starts.  queue[c] counts the claims on class c, queue[kClassCount] the
  // warps that have left; all are zero when a launch starts and the last warp
  // to leave puts them back to zero.  queue = null: no units.
  const WarpDesc* units;
  uint32_t* queue;
  uint32_t unit_off[kClassCount];
  uint32_t n_units[kClassCount];
  uint32_t list_off[kClassCount];
};

struct FinalizeParams {
  const ChunkDesc* chunks;
  const Record* recs;
  const double* segs;
  const uint64_t* rec_nblk;
  const uint32_t* rec_mul;  // per record: x^(8 * bytes after it in its chunk's body); null: computed here
  const uint32_t* crc_xor;  // per chunk: CRC preset/final-XOR term for its length; null: computed here
  uint64_t n_chunks;        // chunks of the whole plan
  uint64_t c_begin, c_end;  // chunks to finalize: [c_begin, c_end), or list positions if ids != null
  const uint32_t* ids;      // list mode: chunk ids; the record of list position i is recs[i]
  uint8_t* packed;  // pack: destination; unpack: source
  FpEntry* out_fp;  // fingerprint: output table; pack, unpack-fp: optional table (null: none)
  uint8_t* flags;   // unpack: per-chunk verdict
};

// Geometry of the sweep kernels: one CTA per SM, with a warp count per mode
// (measured on GB300 with the 31.8 GB shard: the issue-bound fingerprint
// wants 16 warps with deep per-warp stages -- 20 warps cost it 7 points; the
// latency-bound pack and unpack want 20 warps in flight -- 2 points more).
#ifndef FR_WARPS_FP
#define FR_WARPS_FP 16
#endif
#ifndef FR_WARPS_PACK
#define FR_WARPS_PACK 20
#endif
#ifndef FR_WARPS_UNPACK
#define FR_WARPS_UNPACK 20
#endif
#ifndef FR_WARPS_UNPACK_FP
#define FR_WARPS_UNPACK_FP 20
#endif
__host__ __device__ constexpr int sweep_warps(int mode) {
  return mode == kModeFingerprint ? FR_WARPS_FP
         : mode == kModePack      ? FR_WARPS_PACK
         : mode == kModeUnpack    ? FR_WARPS_UNPACK
                                  : FR_WARPS_UNPACK_FP;
}

// Per device, before the first launch: opt the sweep kernels in to their
// shared-memory size.
cudaError_t configure_sweep_fp();
cudaError_t configure_sweep_pack();
cudaError_t configure_sweep_unpack();
cudaError_t configure_sweep_unpack_fp();

// List mode: one warp per listed chunk sweeps its whole body into recs[i].
struct ListParams {
  const ChunkDesc* chunks;
  const uint32_t* ids;
  uint64_t n;
  Record* recs;
  double* segs;
  uint8_t* packed;
};

// One class of chunks: element type and 16-byte alignment of its tensors.
cudaError_t launch_sweep_fp(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s);
// Every class of a batch in one fingerprint launch (per-warp class in WarpDesc;
// class_chunks = the whole chunk-list table).
cudaError_t launch_sweep_fp_mixed(const SweepParams& p, int n_ctas, cudaStream_t s);
cudaError_t launch_sweep_pack_mixed(const SweepParams& p, int n_ctas, cudaStream_t s);
cudaError_t launch_sweep_unpack_mixed(const SweepParams& p, int n_ctas, cudaStream_t s);
cudaError_t launch_sweep_unpack_fp_mixed(const SweepParams& p, int n_ctas, cudaStream_t s);
cudaError_t launch_sweep_pack(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s);
cudaError_t launch_sweep_unpack(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s);
cudaError_t launch_list_pack(const ListParams& p, cudaStream_t s);
cudaError_t launch_sweep_unpack_fp(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s);
cudaError_t launch_list_unpack(const ListParams& p, cudaStream_t s);
cudaError_t launch_list_unpack_fp(const ListParams& p, cudaStream_t s);
inline cudaError_t launch_list_sweep(int mode, const ListParams& p, cudaStream_t s) {
  return mode == kModePack ? launch_list_pack(p, s)
                           : (mode == kModeUnpackFp ? launch_list_unpack_fp(p, s) : launch_list_unpack(p, s));
}

cudaError_t launch_finalize(int mode, const FinalizeParams& p, cudaStream_t s);
// Ascending ids of the set flags, first `cap` of them, and the true count.
cudaError_t launch_compact_flags(const uint8_t* flags, uint64_t n, uint32_t* out, uint64_t cap,
                                 uint64_t* count, uint32_t* status, cudaStream_t s);
// Ascending ids of the differing 16-byte entries, first `cap`, true count.
cudaError_t launch_diff(const FpEntry* a, const FpEntry* b, uint64_t n, uint32_t* out, uint64_t cap,
                        uint64_t* count, cudaStream_t s);

// Set the calling thread's fr_last_error message and return the status
// (FR_ERR_INVALID_ARG with `what`, FR_ERR_CUDA with the CUDA error's text).
fr_status report_invalid(const char* where, const char* what);
fr_status report_cuda(const char* where, cudaError_t e);

}  // namespace frk
