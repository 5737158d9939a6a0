// static_fingerprint.cu -- fr_fingerprint_static: the fingerprint call for
// callers that cannot allocate device memory.
//
// Who needs it: a recovery agent that runs inside a training process whose
// framework allocator has already reserved all of the GPU's memory for the
// model and optimizer state, or any code that is not allowed to call
// cudaMalloc/cudaFree (their implicit device synchronization or their
// failure when memory is exhausted would break the caller).  fr_plan_create
// allocates the plan's tables and scratch, so such callers cannot use it.
//
// This entry point plans on the host into fixed-size static host tables and
// runs the same sweep and finalize kernels as fr_fingerprint, with every
// device table and the per-piece scratch in one file-scope __device__ array
// below.  Every GPU that loads the library holds that array (a few MiB) until
// the process exits.  Nothing here calls cudaMalloc, cudaFree or any other
// allocating routine.
//
// Sharing: all calls, on every stream, use the same array, and each call
// rewrites every table it uses before its kernels run, so nothing carries
// over from the previous call.  Calls whose kernels overlap on the GPU (calls
// on different streams without ordering between them) race on the array and
// give wrong results.  Host-side planning is serialized by a mutex.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "../../include/flashrec.h"
#include "gf2.cuh"
#include "kernels.h"
#include "layout.h"
#include "warp_share.h"

using namespace frk;

namespace {

// Limits of the static variant.
constexpr uint64_t kMaxChunks = FR_STATIC_MAX_CHUNKS;
constexpr uint64_t kMaxWarps = 160 * sweep_warps(kModeFingerprint);  // up to 160 SMs, shared by the classes
constexpr uint64_t kClasses = 6;
constexpr uint64_t kMaxRecs = kMaxWarps + kMaxChunks;
constexpr uint64_t kMaxSegs = FR_STATIC_MAX_SEGMENTS;  // 16 KiB sum segments

// Byte offsets of the tables inside the static array (256-byte aligned).
constexpr uint64_t kOffChunks = 0;
constexpr uint64_t kOffLists = align_up(kOffChunks + kMaxChunks * sizeof(ChunkDesc), 256);
constexpr uint64_t kOffWarps = align_up(kOffLists + kMaxChunks * sizeof(uint32_t), 256);
constexpr uint64_t kOffRecNblk = align_up(kOffWarps + kMaxWarps * sizeof(WarpDesc), 256);
constexpr uint64_t kOffRecs = align_up(kOffRecNblk + kMaxRecs * sizeof(uint64_t), 256);
constexpr uint64_t kOffSegs = align_up(kOffRecs + kMaxRecs * sizeof(Record), 256);
constexpr uint64_t kScratchBytes = align_up(kOffSegs + kMaxSegs * sizeof(double), 256);
static_assert(kScratchBytes < (8ull << 20), "the static scratch must stay modest");

// The device-side scratch.  In host code this name is only a stand-in for the
// symbol, never a device address: kernels get the address that
// cudaGetSymbolAddress returns for the current device.
static __device__ __align__(256) uint8_t g_static_scratch[kScratchBytes];

// Host copies of the tables, staged here and copied into the scratch.
struct HostTables {
  ChunkDesc chunks[kMaxChunks];
  uint32_t lists[kMaxChunks];
  WarpDesc warps[kMaxWarps];
  uint64_t rec_nblk[kMaxRecs];
  uint64_t seg_start[kMaxSegs + 1];  // per class: block where each segment starts
  uint64_t seg_cost[kMaxSegs + 1];   // per class: estimated cost of its segments before each
  uint64_t bnd[kMaxWarps + 1];       // per class: the segment where each warp's range starts
  uint32_t slot[kClasses * kMaxWarps];  // per class: launch-warp index of its j-th warp
};
HostTables g_host;
std::mutex g_mu;

// Per-device set-up: the scratch address and the sweep kernels' shared-memory
// opt-in, done on the first call with that device current.
constexpr int kMaxDevices = 64;
uint8_t* g_dev_ptr[kMaxDevices] = {};

uint64_t elem_bytes(uint32_t dt) { return dt == kDtF32 ? 4 : (dt == kDtBf16 ? 2 : 1); }

// Records the reason for fr_last_error and returns the status.
constexpr const char* kWhere = "fr_fingerprint_static";
fr_status fail(const char* what) { return report_invalid(kWhere, what); }
fr_status fail(cudaError_t e) { return report_cuda(kWhere, e); }

fr_status setup_device(int dev, uint8_t** out) {
  if (dev < 0 || dev >= kMaxDevices) return fail("device index out of range");
  if (g_dev_ptr[dev] == nullptr) {
    void* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_static_scratch);
    if (e != cudaSuccess) return fail(e);
    if (ptr == nullptr) return fail("the scratch array has no device address");
    e = configure_sweep_fp();
    if (e != cudaSuccess) return fail(e);
    g_dev_ptr[dev] = static_cast<uint8_t*>(ptr);
  }
  *out = g_dev_ptr[dev];
  return FR_OK;
}

}  // namespace

extern "C" fr_status fr_fingerprint_static(const fr_tensor* tensors, uint64_t n_tensors, uint64_t chunk_bytes,
                                           fr_fp* out_dev, void* stream) {
  if (n_tensors > 0 && tensors == nullptr) return fail("tensors is null");
  if (n_tensors >= (1ull << 32)) return fail("more than 2^32 - 1 tensors");
  if (chunk_bytes == 0 || chunk_bytes % 4 != 0) return fail("chunk_bytes must be a positive multiple of 4");
  uint64_t n_chunks = 0;
  for (uint64_t t = 0; t < n_tensors; ++t) {
    const fr_tensor& x = tensors[t];
    if (x.dtype > FR_DT_F32 || x.flags != 0) return fail("bad dtype or flags");
    if (x.nbytes % elem_bytes(x.dtype) != 0) return fail("nbytes is not a multiple of the element size");
    if (x.nbytes > 0 && x.ptr == nullptr) return fail("tensor pointer is null");
    if (x.nbytes >= (1ull << 47)) return fail("tensor too large");
    n_chunks += (x.nbytes + chunk_bytes - 1) / chunk_bytes;
    if (n_chunks > kMaxChunks) return fail("more chunks than FR_STATIC_MAX_CHUNKS");
  }
  uint64_t n_segs = 0;
  for (uint64_t t = 0; t < n_tensors; ++t)
    for (uint64_t off = 0; off < tensors[t].nbytes; off += chunk_bytes) {
      const uint64_t len = std::min<uint64_t>(chunk_bytes, tensors[t].nbytes - off);
      n_segs += (len / kBlockBytes + kSegBlocks - 1) / kSegBlocks;
    }
  if (n_segs > kMaxSegs) return fail("more sum segments than FR_STATIC_MAX_SEGMENTS");
  if (n_chunks == 0) return FR_OK;
  if (out_dev == nullptr) return fail("out_dev is null");

  // The table upload reads g_host, which every call rewrites: captured into
  // a graph, a replay would read whatever plan the last call left there.
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaStreamCaptureStatus capturing = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(s, &capturing);
  if (e != cudaSuccess) return fail(e);
  if (capturing != cudaStreamCaptureStatusNone) return fail("the stream is being captured; this call cannot be");

  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(e);
  int n_sm = 0;
  e = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return fail(e);
  const uint64_t W = static_cast<uint64_t>(n_sm) * sweep_warps(kModeFingerprint);
  if (W > kMaxWarps) return fail("GPU has more SMs than the static tables hold");

  std::lock_guard<std::mutex> lk(g_mu);
  uint8_t* scratch = nullptr;
  fr_status st = setup_device(dev, &scratch);
  if (st != FR_OK) return st;

  // ---- plan into the static host tables (same rules as fr_plan_create)
  HostTables& h = g_host;
  uint64_t payload = align_up(n_chunks * kHeaderBytes, kPayloadAlign);
  uint64_t class_blocks[kClasses] = {0, 0, 0, 0, 0, 0};
  uint64_t c = 0, seg = 0;
  for (uint64_t t = 0; t < n_tensors; ++t) {
    const bool aligned = (reinterpret_cast<uintptr_t>(tensors[t].ptr) % 16 == 0) && (chunk_bytes % 16 == 0);
    const uint32_t cls = tensors[t].dtype * 2 + (aligned ? 1 : 0);
    for (uint64_t off = 0; off < tensors[t].nbytes; off += chunk_bytes) {
      ChunkDesc& d = h.chunks[c++];
      std::memset(&d, 0, sizeof d);
      d.len = std::min<uint64_t>(chunk_bytes, tensors[t].nbytes - off);
      d.addr = reinterpret_cast<uint64_t>(tensors[t].ptr) + off;
      d.tensor_off = off;
      d.payload_off = payload;
      d.blk_begin = class_blocks[cls];
      d.tensor_idx = static_cast<uint32_t>(t);
      d.dtype = tensors[t].dtype;
      d.sweep_class = cls;
      d.seg_base = static_cast<uint32_t>(seg);
      seg += (d.len / kBlockBytes + kSegBlocks - 1) / kSegBlocks;
      payload += align_up(d.len, kPayloadAlign);
      class_blocks[cls] += d.len / kBlockBytes;
    }
  }
  // one launch for every class: the W warps shared by weighted blocks, each
  // class's warps spread over the CTAs (warp_share.h)
  uint32_t cls_of[kClasses];
  double cost[kClasses];
  uint64_t wc[kClasses];
  int n_cls = 0;
  for (uint32_t cls = 0; cls < kClasses; ++cls) {
    if (class_blocks[cls] == 0) continue;
    cls_of[n_cls] = cls;
    cost[n_cls] = static_cast<double>(class_blocks[cls]) * block_weight(cls / 2, kShareFingerprint);
    ++n_cls;
  }
  if (n_cls > 0) {
    share_warps(cost, n_cls, W, wc);
    spread_warps(wc, n_cls, W, n_sm, sweep_warps(kModeFingerprint), h.slot, kMaxWarps);
  }
  uint64_t n_lists = 0, n_recs = 0;
  for (int q = 0; q < n_cls; ++q) {
    const uint32_t cls = cls_of[q];
    const uint64_t blk = class_blocks[cls], Wq = wc[q];
    const uint64_t list_off = n_lists;
    for (uint64_t i = 0; i < n_chunks; ++i)
      if (h.chunks[i].sweep_class == cls && h.chunks[i].len >= static_cast<uint64_t>(kBlockBytes))
        h.lists[n_lists++] = static_cast<uint32_t>(i);
    const uint32_t* list = h.lists + list_off;
    // warp ranges start on 16 KiB segment boundaries (see layout.h)
    uint64_t n_class_segs = 0;
    h.seg_cost[0] = 0;
    for (uint64_t i = list_off; i < n_lists; ++i) {
      const ChunkDesc& d = h.chunks[h.lists[i]];
      const uint64_t nb = d.len / kBlockBytes;
      for (uint64_t j = 0; j < nb; j += kSegBlocks) {
        h.seg_start[n_class_segs] = d.blk_begin + j;
        h.seg_cost[n_class_segs + 1] = h.seg_cost[n_class_segs] + seg_cost(std::min<uint64_t>(kSegBlocks, nb - j), j == 0);
        ++n_class_segs;
      }
    }
    h.seg_start[n_class_segs] = blk;
    split_ranges([&](uint64_t s) { return h.seg_cost[s]; }, n_class_segs, Wq, h.bnd);
    uint64_t k = 0;
    for (uint64_t w = 0; w < Wq; ++w) {
      const uint64_t b0 = h.seg_start[h.bnd[w]], b1 = h.seg_start[h.bnd[w + 1]];
      WarpDesc& wd = h.warps[h.slot[q * kMaxWarps + w]];
      std::memset(&wd, 0, sizeof wd);
      wd.blk_begin = b0;
      wd.nblk = b1 - b0;
      wd.rec_base = static_cast<uint32_t>(n_recs);
      wd.cls = cls;
      wd.list_off = static_cast<uint32_t>(list_off);
      if (b1 == b0) continue;
      while (b0 >= h.chunks[list[k]].blk_begin + h.chunks[list[k]].len / kBlockBytes) ++k;
      wd.first_chunk = static_cast<uint32_t>(k);
      uint64_t b = b0, j = k;
      while (b < b1) {
        ChunkDesc& d = h.chunks[list[j]];
        const uint64_t end = d.blk_begin + d.len / kBlockBytes;
        const uint64_t n = std::min(b1, end) - b;
        if (d.n_recs == 0) d.first_rec = static_cast<uint32_t>(n_recs);
        d.n_recs += 1;
        h.rec_nblk[n_recs++] = n;  // n_recs <= W + chunks <= kMaxRecs
        b += n;
        if (b == end) ++j;
      }
    }
  }
  const uint64_t n_warps = n_cls > 0 ? W : 0;

  // ---- tables into the scratch, ordered on the caller's stream
  e = cudaMemcpyAsync(scratch + kOffChunks, h.chunks, n_chunks * sizeof(ChunkDesc), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess && n_lists)
    e = cudaMemcpyAsync(scratch + kOffLists, h.lists, n_lists * sizeof(uint32_t), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess && n_warps)
    e = cudaMemcpyAsync(scratch + kOffWarps, h.warps, n_warps * sizeof(WarpDesc), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess && n_recs)
    e = cudaMemcpyAsync(scratch + kOffRecNblk, h.rec_nblk, n_recs * sizeof(uint64_t), cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return fail(e);

  const ChunkDesc* d_chunks = reinterpret_cast<const ChunkDesc*>(scratch + kOffChunks);
  Record* d_recs = reinterpret_cast<Record*>(scratch + kOffRecs);
  if (n_cls > 0) {
    SweepParams sp;
    sp.chunks = d_chunks;
    sp.warps = reinterpret_cast<const WarpDesc*>(scratch + kOffWarps);
    sp.class_chunks = reinterpret_cast<const uint32_t*>(scratch + kOffLists);
    sp.recs = d_recs;
    sp.segs = reinterpret_cast<double*>(scratch + kOffSegs);
    sp.packed = nullptr;
    sp.n_warps = static_cast<uint32_t>(W);
    sp.units = nullptr;  // the warps' ranges cover every block: no claimed units
    sp.queue = nullptr;
    for (uint32_t c = 0; c < kClassCount; ++c) sp.unit_off[c] = sp.n_units[c] = sp.list_off[c] = 0;
    e = launch_sweep_fp_mixed(sp, n_sm, s);
    if (e != cudaSuccess) return fail(e);
  }
  FinalizeParams fp;
  fp.chunks = d_chunks;
  fp.recs = d_recs;
  fp.segs = reinterpret_cast<const double*>(scratch + kOffSegs);
  fp.rec_nblk = reinterpret_cast<const uint64_t*>(scratch + kOffRecNblk);
  fp.rec_mul = nullptr;  // shifts and CRC terms are computed in the finalize kernel
  fp.crc_xor = nullptr;
  fp.n_chunks = n_chunks;
  fp.c_begin = 0;
  fp.c_end = n_chunks;
  fp.ids = nullptr;
  fp.packed = nullptr;
  fp.out_fp = reinterpret_cast<FpEntry*>(out_dev);
  fp.flags = nullptr;
  e = launch_finalize(kModeFingerprint, fp, s);
  if (e != cudaSuccess) return fail(e);
  return FR_OK;
}
