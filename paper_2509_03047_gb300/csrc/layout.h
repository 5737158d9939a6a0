// layout.h -- plan tables shared by the host planner and the kernels.
//
// A plan splits every tensor into chunks (per tensor, chunk_bytes each, the
// last one shorter).  Each chunk is a "body" of whole 512-byte blocks plus a
// "tail" of len % 512 bytes.  Chunks fall into sweep classes by element type
// and by whether their tensor is 16-byte aligned.  The bodies of a class's
// chunks, concatenated in chunk order, form one block stream that is cut into
// ranges of equal estimated cost (bytes, segment ends, chunk starts), one per
// warp the call's sweep launch gives that class (warp_share.h), so a class's
// warps take about equal time whatever the tensor sizes.  A warp's range
// overlaps
// one or more chunks; each overlap is a "piece" and produces one record (raw
// CRC, non-finite count).  Warp ranges start on segment boundaries.
// The records of a chunk are consecutive and in order.  The finalize kernel
// (one warp per chunk) folds a chunk's records and its tail.
#pragma once

#include <cstdint>

namespace frk {

constexpr uint64_t kHeaderBytes = 64;
// A chunk body is cut into segments of kSegBlocks 512-byte blocks (16 KiB,
// the last one shorter).  Each segment's sum of squares is computed in an
// order fixed by positions alone and stored at its own index, and a chunk's
// sum adds its segments in a fixed order: the result does not depend on how
// the plan spreads the work over warps, batches or SMs.
#ifndef FR_SEG_BLOCKS
#define FR_SEG_BLOCKS 32
#endif
constexpr uint64_t kSegBlocks = FR_SEG_BLOCKS;
static_assert((kSegBlocks & (kSegBlocks - 1)) == 0, "a power of two");
// A segment's 8-byte slot holds its sum in one of two forms, told apart by
// bit 63:
//   clear: an unevaluated float pair, lo in bytes 0-3 and hi (>= +0) in
//          bytes 4-7, whose exact sum is the segment's sum to about 2^-44
//          relative -- the common case, which keeps the sweep off the narrow
//          fp64 pipe;
//   set:   the sum as a double, negated (sums are >= 0, so -0.0 for zero) --
//          segments that needed the exact element-by-element path, or whose
//          sum is too large for the float form.
// seg_value() reads either form as a double.
#ifdef __CUDACC__
__host__ __device__
#endif
inline double seg_value(const double* slot) {
  if (*reinterpret_cast<const uint64_t*>(slot) >> 63) return -*slot;
  const float* f = reinterpret_cast<const float*>(slot);
  return static_cast<double>(f[1]) + static_cast<double>(f[0]);
}
constexpr uint64_t kPayloadAlign = 256;
constexpr uint32_t kMagic = 0x31435246u;  // bytes 'F','R','C','1'
constexpr uint32_t kVersion = 1;

enum : uint32_t { kDtBytes = 0, kDtBf16 = 1, kDtF32 = 2 };
// Sweep classes: element type * 2 + (tensor 16-byte aligned ? 1 : 0).
constexpr uint32_t kClassCount = 6;

struct ChunkDesc {       // 64 bytes
  uint64_t addr;         // device address of the chunk's first byte in its tensor
  uint64_t len;          // chunk bytes
  uint64_t tensor_off;   // offset of the chunk inside its tensor
  uint64_t payload_off;  // offset of the payload in the packed buffer
  uint64_t blk_begin;    // first body block in its class's block stream
  uint32_t tensor_idx;
  uint32_t dtype;
  uint32_t first_rec;    // records of this chunk: [first_rec, first_rec + n_recs)
  uint32_t n_recs;
  uint32_t sweep_class;  // dtype * 2 + (tensor 16-byte aligned ? 1 : 0)
  uint32_t seg_base;     // index of the body's first segment sum
};
static_assert(sizeof(ChunkDesc) == 64, "ChunkDesc layout");

struct WarpDesc {        // 32 bytes
  uint64_t blk_begin;    // first block of this warp's range
  uint64_t nblk;         // blocks in the range (0: idle warp)
  uint32_t first_chunk;  // position, in the class's chunk list, of the chunk holding blk_begin
  uint32_t rec_base;     // record index of the first piece
  uint32_t cls;          // mixed launches: the sweep class of the warp's chunks
  uint32_t list_off;     // mixed launches: where that class's chunk list starts
};
static_assert(sizeof(WarpDesc) == 32, "WarpDesc layout");

struct Record {          // one piece's partial result
  uint32_t crc;          // raw CRC (preset 0, no final XOR) of the piece's bytes
  uint32_t nonfinite;
  double unused;         // sums of squares go to the segment array
};
static_assert(sizeof(Record) == 16, "Record layout");

struct FpEntry {         // = fr_fp
  uint32_t crc32c;
  uint32_t nonfinite;
  double sumsq;
};
static_assert(sizeof(FpEntry) == 16, "FpEntry layout");

// Device-side status bits (plan scratch).
enum : uint32_t { kStatusCapacity = 1u, kStatusTimeout = 2u };

constexpr uint64_t align_up(uint64_t v, uint64_t a) { return (v + a - 1) / a * a; }

}  // namespace frk
