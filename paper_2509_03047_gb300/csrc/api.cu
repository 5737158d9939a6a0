// api.cu -- the C ABI of libflashrec (declared in include/flashrec.h) and the
// host-side planner.
//
// The planner turns a tensor list into the device tables of layout.h:
// per-tensor chunks, the packed layout, the equal per-warp block ranges of the
// sweep and the record slots of every piece.  All device memory a plan needs is
// allocated here, at creation; the four sweep calls only launch kernels.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "../../include/flashrec.h"
#include "gf2.cuh"
#include "kernels.h"
#include "layout.h"

using namespace frk;

// One sweep class: chunks of one element type whose tensors are (or are not)
// 16-byte aligned, with its own block stream and per-warp ranges.
struct SweepClass {
  uint32_t dtype = 0;
  bool aligned = false;
  uint64_t n_blocks = 0;
  uint64_t warp_off = 0;  // into d_warps
  uint64_t list_off = 0;  // into d_class_chunks
};

struct fr_plan_s {
  int device = 0;
  int n_sm = 0;
  uint64_t chunk_bytes = 0, n_chunks = 0, packed_bytes = 0, state_bytes = 0;
  uint64_t n_recs = 0;
  uint32_t n_warps = 0;  // warps per class launch (n_sm * kSweepWarps)
  std::vector<ChunkDesc> chunks;
  std::vector<SweepClass> classes;  // non-empty classes, in class-id order
  ChunkDesc* d_chunks = nullptr;
  WarpDesc* d_warps = nullptr;
  uint32_t* d_class_chunks = nullptr;
  uint64_t* d_rec_nblk = nullptr;
  Record* d_recs = nullptr;
  uint8_t* d_flags = nullptr;
  uint32_t* d_status = nullptr;
};

namespace {

thread_local char g_err[512] = "";

void set_err(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof g_err, fmt, ap);
  va_end(ap);
}

fr_status invalid(const char* what) {
  set_err("invalid argument: %s", what);
  return FR_ERR_INVALID_ARG;
}

fr_status cuda_fail(cudaError_t e, const char* where) {
  set_err("%s: %s", where, cudaGetErrorString(e));
  return FR_ERR_CUDA;
}

uint64_t elem_bytes(uint32_t dt) { return dt == kDtF32 ? 4 : (dt == kDtBf16 ? 2 : 1); }

// Kernels are configured once per device.
std::mutex g_cfg_mu;
uint64_t g_cfg_done = 0;  // bit d: device d configured

fr_status configure_device(int dev) {
  std::lock_guard<std::mutex> lk(g_cfg_mu);
  if (dev >= 0 && dev < 64 && (g_cfg_done >> dev) & 1u) return FR_OK;
  cudaError_t e = configure_sweep_fp();
  if (e == cudaSuccess) e = configure_sweep_pack();
  if (e == cudaSuccess) e = configure_sweep_unpack();
  if (e != cudaSuccess) return cuda_fail(e, "configure sweep kernels");
  if (dev >= 0 && dev < 64) g_cfg_done |= (1ull << dev);
  return FR_OK;
}

// Runs the calls on the plan's device and puts the caller's device back.
struct DeviceGuard {
  int prev = -1;
  bool ok = true;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) {
      ok = false;
      return;
    }
    if (prev != dev && cudaSetDevice(dev) != cudaSuccess) ok = false;
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

template <class T>
cudaError_t upload(T** dst, const std::vector<T>& src) {
  *dst = nullptr;
  if (src.empty()) return cudaSuccess;
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(dst), src.size() * sizeof(T));
  if (e != cudaSuccess) return e;
  return cudaMemcpy(*dst, src.data(), src.size() * sizeof(T), cudaMemcpyHostToDevice);
}

void free_device(fr_plan p) {
  cudaFree(p->d_chunks);
  cudaFree(p->d_warps);
  cudaFree(p->d_class_chunks);
  cudaFree(p->d_rec_nblk);
  cudaFree(p->d_recs);
  cudaFree(p->d_flags);
  cudaFree(p->d_status);
}

}  // namespace

extern "C" {

const char* fr_status_str(fr_status s) {
  switch (s) {
    case FR_OK: return "FR_OK";
    case FR_ERR_INVALID_ARG: return "FR_ERR_INVALID_ARG";
    case FR_ERR_ALIGNMENT: return "FR_ERR_ALIGNMENT";
    case FR_ERR_BUFFER_TOO_SMALL: return "FR_ERR_BUFFER_TOO_SMALL";
    case FR_ERR_CAPACITY: return "FR_ERR_CAPACITY";
    case FR_ERR_PLAN_MISMATCH: return "FR_ERR_PLAN_MISMATCH";
    case FR_ERR_DEVICE_TIMEOUT: return "FR_ERR_DEVICE_TIMEOUT";
    case FR_ERR_CUDA: return "FR_ERR_CUDA";
  }
  return "FR_ERR_UNKNOWN";
}

const char* fr_last_error(void) { return g_err; }

int fr_version(void) { return 10000; }

fr_status fr_plan_create(const fr_tensor* tensors, uint64_t n_tensors, uint64_t chunk_bytes, fr_plan* out) {
  if (out == nullptr) return invalid("out is null");
  *out = nullptr;
  if (n_tensors > 0 && tensors == nullptr) return invalid("tensors is null");
  if (chunk_bytes == 0 || chunk_bytes % 4 != 0) return invalid("chunk_bytes must be a positive multiple of 4");
  if (n_tensors >= (1ull << 32)) return invalid("too many tensors");
  uint64_t n_chunks = 0, state = 0;
  for (uint64_t t = 0; t < n_tensors; ++t) {
    const fr_tensor& x = tensors[t];
    if (x.dtype > FR_DT_F32) return invalid("unknown dtype");
    if (x.flags != 0) return invalid("tensor flags must be 0");
    if (x.nbytes % elem_bytes(x.dtype) != 0) return invalid("nbytes is not a multiple of the element size");
    if (x.nbytes > 0 && x.ptr == nullptr) return invalid("tensor pointer is null");
    if (x.nbytes >= (1ull << 47)) return invalid("tensor too large");
    n_chunks += (x.nbytes + chunk_bytes - 1) / chunk_bytes;
    state += x.nbytes;
  }
  if (n_chunks >= (1ull << 32) - 1) return invalid("too many chunks");

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  int n_sm = 0;
  e = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
  fr_status st = configure_device(dev);
  if (st != FR_OK) return st;

  fr_plan p = new (std::nothrow) fr_plan_s;
  if (p == nullptr) return invalid("out of host memory");
  p->device = dev;
  p->n_sm = n_sm;
  p->chunk_bytes = chunk_bytes;
  p->n_chunks = n_chunks;
  p->state_bytes = state;

  // ---- chunks and packed layout
  p->chunks.resize(n_chunks);
  uint64_t payload = align_up(n_chunks * kHeaderBytes, kPayloadAlign);
  uint64_t c = 0;
  uint64_t class_blocks[6] = {0, 0, 0, 0, 0, 0};
  for (uint64_t t = 0; t < n_tensors; ++t) {
    const bool aligned = (reinterpret_cast<uintptr_t>(tensors[t].ptr) % 16 == 0) && (chunk_bytes % 16 == 0);
    const uint32_t cls = tensors[t].dtype * 2 + (aligned ? 1 : 0);
    for (uint64_t off = 0; off < tensors[t].nbytes; off += chunk_bytes) {
      ChunkDesc& d = p->chunks[c++];
      std::memset(&d, 0, sizeof d);
      d.len = std::min<uint64_t>(chunk_bytes, tensors[t].nbytes - off);
      d.addr = reinterpret_cast<uint64_t>(tensors[t].ptr) + off;
      d.tensor_off = off;
      d.payload_off = payload;
      d.blk_begin = class_blocks[cls];
      d.tensor_idx = static_cast<uint32_t>(t);
      d.dtype = tensors[t].dtype;
      d.sweep_class = cls;
      payload += align_up(d.len, kPayloadAlign);
      class_blocks[cls] += d.len / kBlockBytes;
    }
  }
  p->packed_bytes = payload;

  // ---- per class: equal block ranges per warp, one record per (warp, chunk)
  // overlap.  Records are numbered class by class, so each chunk's records
  // are consecutive.
  std::vector<WarpDesc> warps;
  std::vector<uint32_t> lists;
  std::vector<uint64_t> rec_nblk;
  const uint64_t W = static_cast<uint64_t>(n_sm) * kSweepWarps;
  p->n_warps = static_cast<uint32_t>(W);
  for (uint32_t cls = 0; cls < 6; ++cls) {
    const uint64_t blk = class_blocks[cls];
    if (blk == 0) continue;
    SweepClass sc;
    sc.dtype = cls / 2;
    sc.aligned = (cls & 1u) != 0;
    sc.n_blocks = blk;
    sc.warp_off = warps.size();
    sc.list_off = lists.size();
    for (uint64_t i = 0; i < n_chunks; ++i)
      if (p->chunks[i].sweep_class == cls && p->chunks[i].len >= static_cast<uint64_t>(kBlockBytes))
        lists.push_back(static_cast<uint32_t>(i));
    const uint32_t* list = lists.data() + sc.list_off;
    uint64_t k = 0;  // walks the class list monotonically
    for (uint64_t w = 0; w < W; ++w) {
      const uint64_t b0 = blk * w / W, b1 = blk * (w + 1) / W;
      WarpDesc wd;
      std::memset(&wd, 0, sizeof wd);
      wd.blk_begin = b0;
      wd.nblk = b1 - b0;
      wd.rec_base = static_cast<uint32_t>(rec_nblk.size());
      if (b1 > b0) {
        while (b0 >= p->chunks[list[k]].blk_begin + p->chunks[list[k]].len / kBlockBytes) ++k;
        wd.first_chunk = static_cast<uint32_t>(k);
        uint64_t b = b0, j = k;
        while (b < b1) {
          ChunkDesc& d = p->chunks[list[j]];
          const uint64_t end = d.blk_begin + d.len / kBlockBytes;
          const uint64_t n = std::min(b1, end) - b;
          if (d.n_recs == 0) d.first_rec = static_cast<uint32_t>(rec_nblk.size());
          d.n_recs += 1;
          rec_nblk.push_back(n);
          b += n;
          if (b == end) ++j;
        }
      }
      warps.push_back(wd);
    }
    p->classes.push_back(sc);
  }
  p->n_recs = rec_nblk.size();

  // ---- device tables
  e = upload(&p->d_chunks, p->chunks);
  if (e == cudaSuccess) e = upload(&p->d_warps, warps);
  if (e == cudaSuccess) e = upload(&p->d_class_chunks, lists);
  if (e == cudaSuccess) e = upload(&p->d_rec_nblk, rec_nblk);
  if (e == cudaSuccess && p->n_recs) e = cudaMalloc(&p->d_recs, p->n_recs * sizeof(Record));
  if (e == cudaSuccess && n_chunks) e = cudaMalloc(&p->d_flags, n_chunks);
  if (e == cudaSuccess) e = cudaMalloc(&p->d_status, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMemset(p->d_status, 0, sizeof(uint32_t));
  if (e != cudaSuccess) {
    free_device(p);
    delete p;
    return cuda_fail(e, "plan device tables");
  }
  *out = p;
  return FR_OK;
}

fr_status fr_plan_info(fr_plan p, uint64_t* n_chunks, uint64_t* packed_bytes, uint64_t* state_bytes) {
  if (p == nullptr) return invalid("plan is null");
  if (n_chunks) *n_chunks = p->n_chunks;
  if (packed_bytes) *packed_bytes = p->packed_bytes;
  if (state_bytes) *state_bytes = p->state_bytes;
  return FR_OK;
}

fr_status fr_plan_chunk(fr_plan p, uint64_t chunk_id, uint32_t* tensor_idx, uint64_t* tensor_off, uint64_t* len,
                        uint64_t* payload_off) {
  if (p == nullptr) return invalid("plan is null");
  if (chunk_id >= p->n_chunks) return invalid("chunk_id out of range");
  const ChunkDesc& d = p->chunks[chunk_id];
  if (tensor_idx) *tensor_idx = d.tensor_idx;
  if (tensor_off) *tensor_off = d.tensor_off;
  if (len) *len = d.len;
  if (payload_off) *payload_off = d.payload_off;
  return FR_OK;
}

void fr_plan_destroy(fr_plan p) {
  if (p == nullptr) return;
  DeviceGuard g(p->device);
  cudaDeviceSynchronize();
  free_device(p);
  delete p;
}

static fr_status run_sweep(fr_plan p, int mode, uint8_t* packed, FpEntry* out_fp, cudaStream_t s) {
  for (const SweepClass& sc : p->classes) {
    SweepParams sp;
    sp.chunks = p->d_chunks;
    sp.warps = p->d_warps + sc.warp_off;
    sp.class_chunks = p->d_class_chunks + sc.list_off;
    sp.recs = p->d_recs;
    sp.packed = packed;
    sp.n_warps = p->n_warps;
    cudaError_t e;
    if (mode == kModeFingerprint)
      e = launch_sweep_fp(sc.dtype, sc.aligned, sp, p->n_sm, s);
    else if (mode == kModePack)
      e = launch_sweep_pack(sc.dtype, sc.aligned, sp, p->n_sm, s);
    else
      e = launch_sweep_unpack(sc.dtype, sc.aligned, sp, p->n_sm, s);
    if (e != cudaSuccess) return cuda_fail(e, "sweep kernel launch");
  }
  FinalizeParams fp;
  fp.chunks = p->d_chunks;
  fp.recs = p->d_recs;
  fp.rec_nblk = p->d_rec_nblk;
  fp.n_chunks = p->n_chunks;
  fp.packed = packed;
  fp.out_fp = out_fp;
  fp.flags = p->d_flags;
  cudaError_t e = launch_finalize(mode, fp, s);
  if (e != cudaSuccess) return cuda_fail(e, "finalize kernel launch");
  return FR_OK;
}

fr_status fr_fingerprint(fr_plan p, fr_fp* out_dev, void* stream) {
  if (p == nullptr) return invalid("plan is null");
  if (p->n_chunks == 0) return FR_OK;
  if (out_dev == nullptr) return invalid("out_dev is null");
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  return run_sweep(p, kModeFingerprint, nullptr, reinterpret_cast<FpEntry*>(out_dev),
                   static_cast<cudaStream_t>(stream));
}

fr_status fr_pack(fr_plan p, void* dst, uint64_t dst_bytes, void* stream) {
  if (p == nullptr) return invalid("plan is null");
  if (p->n_chunks == 0) return FR_OK;
  if (dst == nullptr) return invalid("dst is null");
  if (reinterpret_cast<uintptr_t>(dst) % 16 != 0) {
    set_err("packed buffer must be 16-byte aligned");
    return FR_ERR_ALIGNMENT;
  }
  if (dst_bytes < p->packed_bytes) {
    set_err("packed buffer holds %llu bytes, plan needs %llu", (unsigned long long)dst_bytes,
            (unsigned long long)p->packed_bytes);
    return FR_ERR_BUFFER_TOO_SMALL;
  }
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  return run_sweep(p, kModePack, static_cast<uint8_t*>(dst), nullptr, static_cast<cudaStream_t>(stream));
}

fr_status fr_unpack_verify(fr_plan p, const void* src, uint64_t src_bytes, uint32_t* mismatch_dev, uint64_t cap,
                           uint64_t* n_mismatch_dev, void* stream) {
  if (p == nullptr) return invalid("plan is null");
  if (n_mismatch_dev == nullptr) return invalid("n_mismatch_dev is null");
  if (cap > 0 && mismatch_dev == nullptr) return invalid("mismatch_dev is null");
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (p->n_chunks == 0) {
    cudaError_t e = cudaMemsetAsync(n_mismatch_dev, 0, sizeof(uint64_t), s);
    return e == cudaSuccess ? FR_OK : cuda_fail(e, "cudaMemsetAsync");
  }
  if (src == nullptr) return invalid("src is null");
  if (reinterpret_cast<uintptr_t>(src) % 16 != 0) {
    set_err("packed buffer must be 16-byte aligned");
    return FR_ERR_ALIGNMENT;
  }
  if (src_bytes < p->packed_bytes) {
    set_err("packed buffer holds %llu bytes, plan needs %llu", (unsigned long long)src_bytes,
            (unsigned long long)p->packed_bytes);
    return FR_ERR_BUFFER_TOO_SMALL;
  }
  fr_status st = run_sweep(p, kModeUnpack, const_cast<uint8_t*>(static_cast<const uint8_t*>(src)), nullptr, s);
  if (st != FR_OK) return st;
  cudaError_t e = launch_compact_flags(p->d_flags, p->n_chunks, mismatch_dev, cap, n_mismatch_dev, p->d_status, s);
  return e == cudaSuccess ? FR_OK : cuda_fail(e, "compaction kernel launch");
}

fr_status fr_diff(const fr_fp* a_dev, const fr_fp* b_dev, uint64_t n_chunks, uint32_t* diverged_dev, uint64_t cap,
                  uint64_t* n_out_dev, void* stream) {
  if (n_out_dev == nullptr) return invalid("n_out_dev is null");
  if (cap > 0 && diverged_dev == nullptr) return invalid("diverged_dev is null");
  if (n_chunks >= (1ull << 32)) return invalid("too many chunks");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (n_chunks == 0) {
    cudaError_t e = cudaMemsetAsync(n_out_dev, 0, sizeof(uint64_t), s);
    return e == cudaSuccess ? FR_OK : cuda_fail(e, "cudaMemsetAsync");
  }
  if (a_dev == nullptr || b_dev == nullptr) return invalid("table is null");
  if (reinterpret_cast<uintptr_t>(a_dev) % 16 != 0 || reinterpret_cast<uintptr_t>(b_dev) % 16 != 0)
    return invalid("fingerprint tables must be 16-byte aligned");
  cudaError_t e = launch_diff(reinterpret_cast<const FpEntry*>(a_dev), reinterpret_cast<const FpEntry*>(b_dev),
                              n_chunks, diverged_dev, cap, n_out_dev, s);
  return e == cudaSuccess ? FR_OK : cuda_fail(e, "diff kernel launch");
}

fr_status fr_sync_status(fr_plan p, void* stream) {
  if (p == nullptr) return invalid("plan is null");
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  uint32_t bits = 0;
  e = cudaMemcpy(&bits, p->d_status, sizeof bits, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "read plan status");
  if (bits == 0) return FR_OK;
  e = cudaMemset(p->d_status, 0, sizeof bits);
  if (e != cudaSuccess) return cuda_fail(e, "clear plan status");
  if (bits & kStatusTimeout) return FR_ERR_DEVICE_TIMEOUT;
  return FR_ERR_CAPACITY;
}

}  // extern "C"
