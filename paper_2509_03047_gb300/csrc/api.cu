// api.cu -- the C ABI of libflashrec (declared in include/flashrec.h) and the
// host-side planner.
//
// The planner turns a tensor list into the device tables of layout.h:
// per-tensor chunks, the packed layout, and one or two "decompositions" of the
// chunk bodies into per-warp work.  The whole-state decomposition cuts each
// (element type, alignment) class's block stream into ranges of equal
// estimated cost for the warps of every SM; a batched plan also cuts the
// chunks into consecutive
// batches of about equal bytes, each decomposed over half the SMs, so that a
// replica's pack of batch b+1 and a restarted rank's unpack of batch b can run
// side by side (a sweep CTA holds most of an SM's shared memory, so two
// kernels only overlap on disjoint SMs).  All device memory and events a plan
// needs are created here, at creation; the sweep calls only launch kernels.
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

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
#include "warp_share.h"

using namespace frk;

// Each call launches one sweep kernel for every class of a batch, its warps
// shared among the classes by weighted blocks (warp_share.h); the weight
// matters for the fingerprint (a bf16 weight of 100 or 150 instead of 125
// leaves one class's warps finishing last).  Off: one launch per class.
#ifndef FR_MIX_FP
#define FR_MIX_FP 1
#endif
#ifndef FR_MIX_PACK
#define FR_MIX_PACK 1
#endif
// Pack and unpack launches keep this percentage of each class's segments out
// of the warps' own ranges and cut it into units of FR_UNIT_SEGS_PACK
// segments, which warps claim at run time once their range is done (0: none;
// the fingerprint keeps a static split).
#ifndef FR_DYN_PCT_PACK
#define FR_DYN_PCT_PACK 8
#endif
#ifndef FR_UNIT_SEGS_PACK
#define FR_UNIT_SEGS_PACK 4
#endif


namespace {

// One sweep class of one batch: its kernel specialization and its slices of
// the decomposition's warp and chunk-list tables (a mixed decomposition has
// one entry per batch covering all its classes).
struct SweepClass {
  uint32_t dtype = 0;
  bool aligned = false;
  uint64_t warp_off = 0;
  uint64_t list_off = 0;
  // mixed: per sweep class, its claimable units and where its chunk list starts
  uint32_t unit_off[kClassCount] = {0, 0, 0, 0, 0, 0};
  uint32_t n_units[kClassCount] = {0, 0, 0, 0, 0, 0};
  uint32_t class_list[kClassCount] = {0, 0, 0, 0, 0, 0};
};

struct BatchInfo {
  uint64_t c_begin = 0, c_end = 0;
  std::vector<SweepClass> classes;
};

// Per-warp work of every batch, with the chunk table that carries this
// decomposition's block offsets and record ranges.
struct Decomp {
  bool mixed = false;  // one launch per batch for all its classes
  int n_ctas = 0;
  uint32_t n_warps = 0;  // per class launch: n_ctas * warps per CTA
  std::vector<BatchInfo> batches;
  uint64_t n_recs = 0;
  ChunkDesc* d_chunks = nullptr;
  WarpDesc* d_warps = nullptr;
  uint32_t* d_lists = nullptr;
  uint64_t* d_rec_nblk = nullptr;
  uint32_t* d_rec_mul = nullptr;  // per record: x^(8 * bytes after it in its chunk's body)
  Record* d_recs = nullptr;
  WarpDesc* d_units = nullptr;  // mixed: claimable units of every batch
  uint32_t* d_queue = nullptr;  // mixed: kQueueWords counters per batch (SweepParams::queue)
};

// Counters of one mixed launch: a claim count per class and a count of the
// warps that have left (kernels.h, SweepParams::queue), padded to 32 bytes.
constexpr size_t kQueueWords = 8;
static_assert(kQueueWords >= kClassCount + 1, "queue words");

}  // namespace

struct fr_plan_s {
  int device = 0;
  int n_sm = 0;
  uint64_t chunk_bytes = 0, n_chunks = 0, packed_bytes = 0, state_bytes = 0;
  uint32_t n_batches = 1;
  std::vector<ChunkDesc> chunks;  // layout fields (host copy)
  // Decompositions, one per distinct warps-per-CTA count of the sweep modes
  // (geo[mode] indexes them): whole = one batch over all SMs; batched (when
  // n_batches > 1) = batches over half the SMs.  whole[0] also holds n_chunks
  // record slots for list-mode calls.
  std::vector<Decomp> whole, batched;
  int geo[4] = {0, 0, 0, 0};
  uint64_t n_segs = 0;            // 16 KiB sum segments of all chunk bodies
  double* d_segs = nullptr;       // their sums of squares
  uint32_t* d_crc_xor = nullptr;  // per chunk: the CRC preset/final-XOR term of its length
  uint8_t* d_flags = nullptr;     // unpack verdict per chunk
  uint32_t* d_status = nullptr;
  uint32_t* d_ids = nullptr;      // restore: ids of failing chunks (capacity n_chunks)
  uint64_t* d_count = nullptr;
  std::vector<cudaEvent_t> events;  // restore: one per batch, plus one
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

// A named NVTX range around each public call, so a profiler's timeline shows
// which call issued which kernels.  NVTX is header-only: with no profiler
// attached, push and pop return at once.
struct CallRange {
  explicit CallRange(const char* name) { nvtxRangePushA(name); }
  ~CallRange() { nvtxRangePop(); }
  CallRange(const CallRange&) = delete;
  CallRange& operator=(const CallRange&) = delete;
};

fr_status cuda_fail(cudaError_t e, const char* where) {
  set_err("%s: %s", where, cudaGetErrorString(e));
  return FR_ERR_CUDA;
}

}  // namespace

// The other translation units' entry points report through the same
// thread-local message.
fr_status frk::report_invalid(const char* where, const char* what) {
  set_err("%s: invalid argument: %s", where, what);
  return FR_ERR_INVALID_ARG;
}

fr_status frk::report_cuda(const char* where, cudaError_t e) {
  set_err("%s: %s", where, cudaGetErrorString(e));
  return FR_ERR_CUDA;
}

namespace {

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
  if (e == cudaSuccess) e = configure_sweep_unpack_fp();
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

void free_decomp(Decomp& D) {
  cudaFree(D.d_chunks);
  cudaFree(D.d_warps);
  cudaFree(D.d_lists);
  cudaFree(D.d_rec_nblk);
  cudaFree(D.d_rec_mul);
  cudaFree(D.d_recs);
  cudaFree(D.d_units);
  cudaFree(D.d_queue);
  D = Decomp();
}

void free_device(fr_plan p) {
  for (Decomp& d : p->whole) free_decomp(d);
  for (Decomp& d : p->batched) free_decomp(d);
  cudaFree(p->d_segs);
  cudaFree(p->d_crc_xor);
  cudaFree(p->d_flags);
  cudaFree(p->d_status);
  cudaFree(p->d_ids);
  cudaFree(p->d_count);
  for (cudaEvent_t ev : p->events) cudaEventDestroy(ev);
  p->events.clear();
}

// Cut the chunks [bounds[b], bounds[b+1]) of every batch b into sweep work for
// `n_ctas` CTAs: per batch and class, the class's 16 KiB segments in chunk
// order are split into runs of equal estimated cost (split_ranges), one per
// warp, and every (warp, chunk) overlap gets one record.  Records are numbered batch by batch, class
// by class, so each chunk's records are consecutive.  `min_recs`: record slots
// to allocate at least (list-mode calls use one slot per listed chunk).
// Plain: every class gets all n_ctas * warps_per_cta warps (one launch per
// class).  Mixed: the classes of a batch share them in proportion to their
// weighted blocks, each class's warps spread round-robin over the CTAs.  For
// pack and unpack (mix 2) the warps' ranges cover the first
// (100 - FR_DYN_PCT_PACK)% of each class's segments and the rest becomes units
// claimed at run time (their records follow the class's range records, in
// block order).
cudaError_t build_decomp(const std::vector<ChunkDesc>& base, const std::vector<uint64_t>& bounds, int n_ctas,
                         int warps_per_cta, int mix, uint64_t min_recs, Decomp& D) {
  const bool mixed = mix != 0;  // 1: fingerprint weights, 2: pack / unpack weights
  const uint64_t W = static_cast<uint64_t>(n_ctas) * warps_per_cta;
  D.mixed = mixed;
  D.n_ctas = n_ctas;
  D.n_warps = static_cast<uint32_t>(W);
  std::vector<ChunkDesc> chunks = base;
  std::vector<WarpDesc> warps;
  std::vector<uint32_t> lists;
  std::vector<uint64_t> rec_nblk;
  std::vector<uint32_t> rec_mul;
  std::vector<WarpDesc> units;
  const uint64_t unit_segs = FR_UNIT_SEGS_PACK;
  const uint64_t dyn_pct = mix == kSharePack ? FR_DYN_PCT_PACK : 0;
  const bool claims = mixed && dyn_pct > 0;
  for (ChunkDesc& d : chunks) {
    d.blk_begin = 0;
    d.first_rec = 0;
    d.n_recs = 0;
  }
  for (size_t b = 0; b + 1 < bounds.size(); ++b) {
    BatchInfo bi;
    bi.c_begin = bounds[b];
    bi.c_end = bounds[b + 1];
    uint64_t class_blocks[6] = {0, 0, 0, 0, 0, 0};
    for (uint64_t c = bi.c_begin; c < bi.c_end; ++c) {
      ChunkDesc& d = chunks[c];
      d.blk_begin = class_blocks[d.sweep_class];
      class_blocks[d.sweep_class] += d.len / kBlockBytes;
    }
    // the batch's classes: chunk lists and, per class, the class-stream block
    // where each segment starts (warp ranges start on segment boundaries)
    struct Cls {
      uint32_t cls;
      uint64_t list_off;
      std::vector<uint64_t> seg_start;
      std::vector<uint64_t> cost;  // cost[s]: estimated cost of segments [0, s)
    };
    std::vector<Cls> cl;
    for (uint32_t cls = 0; cls < 6; ++cls) {
      if (class_blocks[cls] == 0) continue;
      Cls q;
      q.cls = cls;
      q.list_off = lists.size();
      for (uint64_t c = bi.c_begin; c < bi.c_end; ++c)
        if (chunks[c].sweep_class == cls && chunks[c].len >= static_cast<uint64_t>(kBlockBytes))
          lists.push_back(static_cast<uint32_t>(c));
      q.cost.push_back(0);
      for (size_t i = q.list_off; i < lists.size(); ++i) {
        const ChunkDesc& d = chunks[lists[i]];
        const uint64_t nb = d.len / kBlockBytes;
        for (uint64_t j = 0; j < nb; j += kSegBlocks) {
          q.seg_start.push_back(d.blk_begin + j);
          const uint64_t blocks = std::min<uint64_t>(kSegBlocks, nb - j);
          q.cost.push_back(q.cost.back() + seg_cost(blocks, j == 0));
        }
      }
      q.seg_start.push_back(class_blocks[cls]);
      cl.push_back(std::move(q));
    }
    if (cl.empty()) {
      D.batches.push_back(bi);
      continue;
    }
    // warps per class, and (mixed) slot[q * W + j] = the batch-warp index of
    // class q's j-th warp
    std::vector<uint64_t> wc(cl.size(), W);
    std::vector<uint32_t> slot;
    const uint64_t warp_base = warps.size();
    if (mixed) {
      double cost[6];
      for (size_t q = 0; q < cl.size(); ++q)
        cost[q] = static_cast<double>(class_blocks[cl[q].cls]) * block_weight(cl[q].cls / 2, mix);
      share_warps(cost, static_cast<int>(cl.size()), W, wc.data());
      slot.resize(cl.size() * W);
      spread_warps(wc.data(), static_cast<int>(cl.size()), W, n_ctas, warps_per_cta, slot.data(), W);
      warps.resize(warp_base + W);
      SweepClass sc;
      sc.warp_off = warp_base;
      sc.list_off = 0;
      bi.classes.push_back(sc);
    }
    for (size_t q = 0; q < cl.size(); ++q) {
      const uint32_t cls = cl[q].cls;
      const size_t lbase = cl[q].list_off;
      const std::vector<uint64_t>& seg_start = cl[q].seg_start;
      const uint64_t n_seg = seg_start.size() - 1, Wq = wc[q];
      const uint64_t n_fix = claims ? n_seg - n_seg * dyn_pct / 100 : n_seg;  // segments in the warps' ranges
      SweepClass sc;
      sc.dtype = cls / 2;
      sc.aligned = (cls & 1u) != 0;
      sc.warp_off = warps.size();
      sc.list_off = lbase;
      uint64_t k = 0;  // walks the class list monotonically
      // the descriptor of class blocks [b0, b1), with one record per chunk it overlaps
      auto range = [&](uint64_t b0, uint64_t b1) {
        WarpDesc wd;
        std::memset(&wd, 0, sizeof wd);
        wd.blk_begin = b0;
        wd.nblk = b1 - b0;
        wd.rec_base = static_cast<uint32_t>(rec_nblk.size());
        wd.cls = cls;
        wd.list_off = static_cast<uint32_t>(lbase);
        if (b1 > b0) {
          while (b0 >= chunks[lists[lbase + k]].blk_begin + chunks[lists[lbase + k]].len / kBlockBytes) ++k;
          wd.first_chunk = static_cast<uint32_t>(k);
          uint64_t bb = b0, j = k;
          while (bb < b1) {
            ChunkDesc& d = chunks[lists[lbase + j]];
            const uint64_t end = d.blk_begin + d.len / kBlockBytes;
            const uint64_t n = std::min(b1, end) - bb;
            if (d.n_recs == 0) d.first_rec = static_cast<uint32_t>(rec_nblk.size());
            d.n_recs += 1;
            rec_nblk.push_back(n);
            rec_mul.push_back(host_xpow8((end - bb - n) * kBlockBytes));
            bb += n;
            if (bb == end) ++j;
          }
        }
        return wd;
      };
      // the warps' ranges: the first n_fix segments cut by estimated cost
      std::vector<uint64_t> bnd(Wq + 1);
      const std::vector<uint64_t>& cost = cl[q].cost;
      split_ranges([&](uint64_t i) { return cost[i]; }, n_fix, Wq, bnd.data());
      for (uint64_t w = 0; w < Wq; ++w) {
        const WarpDesc wd = range(seg_start[bnd[w]], seg_start[bnd[w + 1]]);
        if (mixed)
          warps[warp_base + slot[q * W + w]] = wd;
        else
          warps.push_back(wd);
      }
      if (mixed) {
        SweepClass& ms = bi.classes.back();
        ms.unit_off[cls] = static_cast<uint32_t>(units.size());
        ms.class_list[cls] = static_cast<uint32_t>(lbase);
        for (uint64_t u = n_fix; u < n_seg; u += unit_segs)
          units.push_back(range(seg_start[u], seg_start[std::min(u + unit_segs, n_seg)]));
        ms.n_units[cls] = static_cast<uint32_t>(units.size() - ms.unit_off[cls]);
      } else {
        bi.classes.push_back(sc);
      }
    }
    D.batches.push_back(bi);
  }
  D.n_recs = rec_nblk.size();
  cudaError_t e = upload(&D.d_chunks, chunks);
  if (e == cudaSuccess) e = upload(&D.d_warps, warps);
  if (e == cudaSuccess) e = upload(&D.d_lists, lists);
  if (e == cudaSuccess) e = upload(&D.d_rec_nblk, rec_nblk);
  if (e == cudaSuccess) e = upload(&D.d_rec_mul, rec_mul);
  if (e == cudaSuccess) e = upload(&D.d_units, units);
  if (e == cudaSuccess && claims) {
    const size_t qbytes = kQueueWords * sizeof(uint32_t) * std::max<size_t>(D.batches.size(), 1);
    e = cudaMalloc(&D.d_queue, qbytes);
    if (e == cudaSuccess) e = cudaMemset(D.d_queue, 0, qbytes);
  }
  const uint64_t slots = std::max<uint64_t>(D.n_recs, min_recs);
  if (e == cudaSuccess && slots) e = cudaMalloc(&D.d_recs, slots * sizeof(Record));
  return e;
}

// Sweep + finalize of batches [b0, b1) of decomposition D.
fr_status run_batches(fr_plan p, const Decomp& D, int mode, uint8_t* packed, FpEntry* out_fp, size_t b0, size_t b1,
                      cudaStream_t s) {
  for (size_t b = b0; b < b1; ++b) {
    for (const SweepClass& sc : D.batches[b].classes) {
      SweepParams sp;
      sp.chunks = D.d_chunks;
      sp.warps = D.d_warps + sc.warp_off;
      sp.class_chunks = D.d_lists;  // (WarpDesc::list_off is absolute)
      sp.recs = D.d_recs;
      sp.segs = p->d_segs;
      sp.packed = packed;
      sp.n_warps = D.n_warps;
      sp.units = D.d_units;
      sp.queue = D.d_queue ? D.d_queue + kQueueWords * b : nullptr;
      for (uint32_t c = 0; c < kClassCount; ++c) {
        sp.unit_off[c] = sc.unit_off[c];
        sp.n_units[c] = sc.n_units[c];
        sp.list_off[c] = sc.class_list[c];
      }
      cudaError_t e;
      if (D.mixed)
        e = mode == kModeFingerprint ? launch_sweep_fp_mixed(sp, D.n_ctas, s)
            : mode == kModePack      ? launch_sweep_pack_mixed(sp, D.n_ctas, s)
            : mode == kModeUnpackFp  ? launch_sweep_unpack_fp_mixed(sp, D.n_ctas, s)
                                     : launch_sweep_unpack_mixed(sp, D.n_ctas, s);
      else if (mode == kModeFingerprint)
        e = launch_sweep_fp(sc.dtype, sc.aligned, sp, D.n_ctas, s);
      else if (mode == kModePack)
        e = launch_sweep_pack(sc.dtype, sc.aligned, sp, D.n_ctas, s);
      else if (mode == kModeUnpackFp)
        e = launch_sweep_unpack_fp(sc.dtype, sc.aligned, sp, D.n_ctas, s);
      else
        e = launch_sweep_unpack(sc.dtype, sc.aligned, sp, D.n_ctas, s);
      if (e != cudaSuccess) return cuda_fail(e, "sweep kernel launch");
    }
  }
  FinalizeParams fp;
  fp.chunks = D.d_chunks;
  fp.recs = D.d_recs;
  fp.segs = p->d_segs;
  fp.rec_nblk = D.d_rec_nblk;
  fp.rec_mul = D.d_rec_mul;
  fp.crc_xor = p->d_crc_xor;
  fp.n_chunks = p->n_chunks;
  fp.c_begin = D.batches[b0].c_begin;
  fp.c_end = D.batches[b1 - 1].c_end;
  fp.ids = nullptr;
  fp.packed = packed;
  fp.out_fp = out_fp;
  fp.flags = p->d_flags;
  cudaError_t e = launch_finalize(mode, fp, s);
  if (e != cudaSuccess) return cuda_fail(e, "finalize kernel launch");
  return FR_OK;
}

// Sweep + finalize of the `n` chunks listed in `ids` (device), each by one
// warp: used to re-send chunks that failed verification.  `out_fp` (may be
// null) receives the listed chunks' table entries.
fr_status run_list(fr_plan p, int mode, const uint32_t* ids, uint64_t n, uint8_t* packed, FpEntry* out_fp,
                   cudaStream_t s) {
  if (n == 0) return FR_OK;
  ListParams lp;
  lp.chunks = p->whole[0].d_chunks;
  lp.ids = ids;
  lp.n = n;
  lp.recs = p->whole[0].d_recs;
  lp.segs = p->d_segs;
  lp.packed = packed;
  cudaError_t e = launch_list_sweep(mode, lp, s);
  if (e != cudaSuccess) return cuda_fail(e, "list sweep kernel launch");
  FinalizeParams fp;
  fp.chunks = p->whole[0].d_chunks;
  fp.recs = p->whole[0].d_recs;
  fp.segs = p->d_segs;
  fp.rec_nblk = nullptr;
  fp.rec_mul = nullptr;
  fp.crc_xor = p->d_crc_xor;
  fp.n_chunks = p->n_chunks;
  fp.c_begin = 0;
  fp.c_end = n;
  fp.ids = ids;
  fp.packed = packed;
  fp.out_fp = out_fp;
  fp.flags = p->d_flags;
  e = launch_finalize(mode, fp, s);
  if (e != cudaSuccess) return cuda_fail(e, "finalize kernel launch");
  return FR_OK;
}

fr_status check_packed_buffer(fr_plan p, const void* buf, uint64_t bytes) {
  if (buf == nullptr) return invalid("packed buffer is null");
  if (reinterpret_cast<uintptr_t>(buf) % 16 != 0) {
    set_err("packed buffer must be 16-byte aligned");
    return FR_ERR_ALIGNMENT;
  }
  if (bytes < p->packed_bytes) {
    set_err("packed buffer holds %llu bytes, plan needs %llu", (unsigned long long)bytes,
            (unsigned long long)p->packed_bytes);
    return FR_ERR_BUFFER_TOO_SMALL;
  }
  return FR_OK;
}

// The decomposition a mode's whole-state / batch calls run on.
const Decomp& whole_for(fr_plan p, int mode) { return p->whole[p->geo[mode]]; }
const Decomp& batch_for(fr_plan p, int mode) {
  return p->n_batches > 1 ? p->batched[p->geo[mode]] : p->whole[p->geo[mode]];
}

fr_status check_same_layout(fr_plan src, fr_plan dst) {
  if (src->device != dst->device || src->n_chunks != dst->n_chunks || src->packed_bytes != dst->packed_bytes ||
      src->n_batches != dst->n_batches) {
    set_err("the two plans do not describe the same layout");
    return FR_ERR_PLAN_MISMATCH;
  }
  for (uint64_t c = 0; c < src->n_chunks; ++c) {
    const ChunkDesc &a = src->chunks[c], &b = dst->chunks[c];
    if (a.len != b.len || a.dtype != b.dtype || a.tensor_idx != b.tensor_idx || a.tensor_off != b.tensor_off) {
      set_err("the two plans differ at chunk %llu", (unsigned long long)c);
      return FR_ERR_PLAN_MISMATCH;
    }
  }
  return FR_OK;
}

// One re-send: list the chunks whose last verdict in `dst` failed (a host
// sync learns how many), re-pack them from `src` on `ss`, and re-unpack them
// on `sd` after that.  *failing gets the number re-sent.  Non-null fp_src /
// fp_dst get the re-sent chunks' table entries on either side.
fr_status resend_failed(fr_plan src, fr_plan dst, uint8_t* buf, cudaStream_t ss, cudaStream_t sd,
                        uint64_t* failing, FpEntry* fp_src = nullptr, FpEntry* fp_dst = nullptr) {
  *failing = 0;
  cudaError_t e =
      launch_compact_flags(dst->d_flags, dst->n_chunks, dst->d_ids, dst->n_chunks, dst->d_count, nullptr, sd);
  if (e != cudaSuccess) return cuda_fail(e, "compaction kernel launch");
  uint64_t n = 0;
  if ((e = cudaMemcpyAsync(&n, dst->d_count, sizeof n, cudaMemcpyDeviceToHost, sd)) != cudaSuccess ||
      (e = cudaStreamSynchronize(sd)) != cudaSuccess)
    return cuda_fail(e, "read failing-chunk count");
  if (n == 0) return FR_OK;
  cudaEvent_t ev_ids = dst->events[dst->n_batches], ev_packed = src->events[src->n_batches];
  if ((e = cudaEventRecord(ev_ids, sd)) != cudaSuccess || (e = cudaStreamWaitEvent(ss, ev_ids, 0)) != cudaSuccess)
    return cuda_fail(e, "order the re-send");
  fr_status st = run_list(src, kModePack, dst->d_ids, n, buf, fp_src, ss);
  if (st != FR_OK) return st;
  if ((e = cudaEventRecord(ev_packed, ss)) != cudaSuccess || (e = cudaStreamWaitEvent(sd, ev_packed, 0)) != cudaSuccess)
    return cuda_fail(e, "order the re-send");
  st = run_list(dst, fp_dst ? kModeUnpackFp : kModeUnpack, dst->d_ids, n, buf, fp_dst, sd);
  if (st != FR_OK) return st;
  *failing = n;
  return FR_OK;
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

int fr_version(void) { return 10100; }

fr_status fr_plan_create_batched(const fr_tensor* tensors, uint64_t n_tensors, uint64_t chunk_bytes,
                                 uint32_t n_batches, fr_plan* out) {
  CallRange nvtx("fr_plan_create_batched");
  if (out == nullptr) return invalid("out is null");
  *out = nullptr;
  if (n_tensors > 0 && tensors == nullptr) return invalid("tensors is null");
  if (chunk_bytes == 0 || chunk_bytes % 4 != 0) return invalid("chunk_bytes must be a positive multiple of 4");
  if (n_tensors >= (1ull << 32)) return invalid("too many tensors");
  if (n_batches == 0) return invalid("n_batches must be at least 1");
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
  p->n_batches = static_cast<uint32_t>(std::max<uint64_t>(1, std::min<uint64_t>(n_batches, n_chunks)));

  // ---- chunks and packed layout
  p->chunks.resize(n_chunks);
  uint64_t payload = align_up(n_chunks * kHeaderBytes, kPayloadAlign);
  uint64_t c = 0;
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
      d.tensor_idx = static_cast<uint32_t>(t);
      d.dtype = tensors[t].dtype;
      d.sweep_class = cls;
      d.seg_base = static_cast<uint32_t>(p->n_segs);
      p->n_segs += (d.len / kBlockBytes + kSegBlocks - 1) / kSegBlocks;
      payload += align_up(d.len, kPayloadAlign);
    }
  }
  p->packed_bytes = payload;
  if (p->n_segs >= (1ull << 32)) {
    delete p;
    return invalid("state too large");
  }

  // ---- decompositions
  e = cudaSuccess;
  if (n_chunks > 0) {
    // distinct decompositions of the modes: warps per CTA and mixing (none,
    // with the fingerprint's weights, with pack's); the fingerprint's is geo 0
    std::vector<int> counts;  // 3 * warps + mix
    for (int m = 0; m < 4; ++m) {
      const int mix = m == kModeFingerprint ? (FR_MIX_FP ? 1 : 0) : (FR_MIX_PACK ? 2 : 0);
      const int w = 3 * sweep_warps(m) + mix;
      int g = 0;
      while (g < static_cast<int>(counts.size()) && counts[g] != w) ++g;
      if (g == static_cast<int>(counts.size())) counts.push_back(w);
      p->geo[m] = g;
    }
    p->whole.resize(counts.size());
    p->batched.resize(counts.size());
    for (size_t g = 0; e == cudaSuccess && g < counts.size(); ++g)
      e = build_decomp(p->chunks, {0, n_chunks}, n_sm, counts[g] / 3, counts[g] % 3, g == 0 ? n_chunks : 0, p->whole[g]);
    if (e == cudaSuccess && p->n_batches > 1) {
      // batch starts at about equal state bytes, every batch non-empty
      std::vector<uint64_t> bounds(1, 0);
      uint64_t acc = 0, cc = 0;
      for (uint32_t b = 1; b < p->n_batches; ++b) {
        const uint64_t target = state / p->n_batches * b;
        while (cc < n_chunks && (acc < target || cc <= bounds.back())) acc += p->chunks[cc++].len;
        const uint64_t room = n_chunks - (p->n_batches - b);  // leave one chunk per later batch
        bounds.push_back(std::min(cc, room));
      }
      bounds.push_back(n_chunks);
      for (size_t i = 1; i < bounds.size(); ++i)
        if (bounds[i] <= bounds[i - 1]) bounds[i] = bounds[i - 1] + 1;
      for (size_t g = 0; e == cudaSuccess && g < counts.size(); ++g)
        e = build_decomp(p->chunks, bounds, std::max(1, n_sm / 2), counts[g] / 3, counts[g] % 3, 0, p->batched[g]);
    }
  }
  if (e == cudaSuccess && p->n_segs) e = cudaMalloc(&p->d_segs, p->n_segs * sizeof(double));
  if (e == cudaSuccess && n_chunks) {
    std::vector<uint32_t> crc_xor(n_chunks);
    for (uint64_t c = 0; c < n_chunks; ++c) crc_xor[c] = host_crc_xor_term(p->chunks[c].len);
    e = upload(&p->d_crc_xor, crc_xor);
  }
  if (e == cudaSuccess && n_chunks) e = cudaMalloc(&p->d_flags, n_chunks);
  if (e == cudaSuccess && n_chunks) e = cudaMalloc(&p->d_ids, n_chunks * sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMalloc(&p->d_count, sizeof(uint64_t));
  if (e == cudaSuccess) e = cudaMalloc(&p->d_status, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaMemset(p->d_status, 0, sizeof(uint32_t));
  for (uint32_t i = 0; e == cudaSuccess && i < p->n_batches + 1; ++i) {
    cudaEvent_t ev;
    e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
    if (e == cudaSuccess) p->events.push_back(ev);
  }
  if (e != cudaSuccess) {
    free_device(p);
    delete p;
    return cuda_fail(e, "plan device tables");
  }
  *out = p;
  return FR_OK;
}

fr_status fr_plan_create(const fr_tensor* tensors, uint64_t n_tensors, uint64_t chunk_bytes, fr_plan* out) {
  return fr_plan_create_batched(tensors, n_tensors, chunk_bytes, 1, out);
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

fr_status fr_plan_batch(fr_plan p, uint32_t batch, uint32_t* n_batches, uint64_t* first_chunk, uint64_t* n_chunks) {
  if (p == nullptr) return invalid("plan is null");
  if (n_batches) *n_batches = p->n_chunks ? p->n_batches : 0;
  if (p->n_chunks == 0) {
    if (first_chunk) *first_chunk = 0;
    if (n_chunks) *n_chunks = 0;
    return FR_OK;
  }
  if (batch >= p->n_batches) return invalid("batch out of range");
  const BatchInfo& b = batch_for(p, kModePack).batches[batch];
  if (first_chunk) *first_chunk = b.c_begin;
  if (n_chunks) *n_chunks = b.c_end - b.c_begin;
  return FR_OK;
}

void fr_plan_destroy(fr_plan p) {
  CallRange nvtx("fr_plan_destroy");
  if (p == nullptr) return;
  DeviceGuard g(p->device);
  cudaDeviceSynchronize();
  free_device(p);
  delete p;
}

fr_status fr_fingerprint(fr_plan p, fr_fp* out_dev, void* stream) {
  CallRange nvtx("fr_fingerprint");
  if (p == nullptr) return invalid("plan is null");
  if (p->n_chunks == 0) return FR_OK;
  if (out_dev == nullptr) return invalid("out_dev is null");
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  return run_batches(p, whole_for(p, kModeFingerprint), kModeFingerprint, nullptr, reinterpret_cast<FpEntry*>(out_dev), 0, 1,
                     static_cast<cudaStream_t>(stream));
}

fr_status fr_pack(fr_plan p, void* dst, uint64_t dst_bytes, void* stream) {
  CallRange nvtx("fr_pack");
  return fr_pack_fp(p, dst, dst_bytes, nullptr, stream);
}

fr_status fr_pack_fp(fr_plan p, void* dst, uint64_t dst_bytes, fr_fp* fp_dev, void* stream) {
  CallRange nvtx("fr_pack_fp");
  if (p == nullptr) return invalid("plan is null");
  if (p->n_chunks == 0) return FR_OK;
  fr_status st = check_packed_buffer(p, dst, dst_bytes);
  if (st != FR_OK) return st;
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  return run_batches(p, whole_for(p, kModePack), kModePack, static_cast<uint8_t*>(dst), reinterpret_cast<FpEntry*>(fp_dev), 0, 1,
                     static_cast<cudaStream_t>(stream));
}

fr_status fr_unpack_verify(fr_plan p, const void* src, uint64_t src_bytes, uint32_t* mismatch_dev, uint64_t cap,
                           uint64_t* n_mismatch_dev, void* stream) {
  CallRange nvtx("fr_unpack_verify");
  return fr_unpack_verify_fp(p, src, src_bytes, mismatch_dev, cap, n_mismatch_dev, nullptr, stream);
}

fr_status fr_unpack_verify_fp(fr_plan p, const void* src, uint64_t src_bytes, uint32_t* mismatch_dev, uint64_t cap,
                              uint64_t* n_mismatch_dev, fr_fp* fp_dev, void* stream) {
  CallRange nvtx("fr_unpack_verify_fp");
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
  fr_status st = check_packed_buffer(p, src, src_bytes);
  if (st != FR_OK) return st;
  const int mode = fp_dev ? kModeUnpackFp : kModeUnpack;
  st = run_batches(p, whole_for(p, mode), mode,
                   const_cast<uint8_t*>(static_cast<const uint8_t*>(src)), reinterpret_cast<FpEntry*>(fp_dev), 0, 1, s);
  if (st != FR_OK) return st;
  cudaError_t e = launch_compact_flags(p->d_flags, p->n_chunks, mismatch_dev, cap, n_mismatch_dev, p->d_status, s);
  return e == cudaSuccess ? FR_OK : cuda_fail(e, "compaction kernel launch");
}

fr_status fr_pack_batch(fr_plan p, uint32_t batch, void* dst, uint64_t dst_bytes, void* stream) {
  CallRange nvtx("fr_pack_batch");
  if (p == nullptr) return invalid("plan is null");
  if (p->n_chunks == 0) return FR_OK;
  if (batch >= p->n_batches) return invalid("batch out of range");
  fr_status st = check_packed_buffer(p, dst, dst_bytes);
  if (st != FR_OK) return st;
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  return run_batches(p, batch_for(p, kModePack), kModePack, static_cast<uint8_t*>(dst), nullptr, batch, batch + 1,
                     static_cast<cudaStream_t>(stream));
}

fr_status fr_unpack_verify_batch(fr_plan p, uint32_t batch, const void* src, uint64_t src_bytes, void* stream) {
  CallRange nvtx("fr_unpack_verify_batch");
  if (p == nullptr) return invalid("plan is null");
  if (p->n_chunks == 0) return FR_OK;
  if (batch >= p->n_batches) return invalid("batch out of range");
  fr_status st = check_packed_buffer(p, src, src_bytes);
  if (st != FR_OK) return st;
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  return run_batches(p, batch_for(p, kModeUnpack), kModeUnpack, const_cast<uint8_t*>(static_cast<const uint8_t*>(src)),
                     nullptr, batch, batch + 1, static_cast<cudaStream_t>(stream));
}

fr_status fr_unpack_collect(fr_plan p, uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev,
                            void* stream) {
  CallRange nvtx("fr_unpack_collect");
  if (p == nullptr) return invalid("plan is null");
  if (n_mismatch_dev == nullptr) return invalid("n_mismatch_dev is null");
  if (cap > 0 && mismatch_dev == nullptr) return invalid("mismatch_dev is null");
  DeviceGuard g(p->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (p->n_chunks == 0)
    e = cudaMemsetAsync(n_mismatch_dev, 0, sizeof(uint64_t), s);
  else
    e = launch_compact_flags(p->d_flags, p->n_chunks, mismatch_dev, cap, n_mismatch_dev, p->d_status, s);
  return e == cudaSuccess ? FR_OK : cuda_fail(e, "compaction kernel launch");
}

fr_status fr_restore(fr_plan src, fr_plan dst, void* staging, uint64_t staging_bytes, uint32_t max_retries,
                     uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev, void* stream_src,
                     void* stream_dst) {
  CallRange nvtx("fr_restore");
  return fr_restore_fp(src, dst, staging, staging_bytes, max_retries, mismatch_dev, cap, n_mismatch_dev, nullptr,
                       nullptr, stream_src, stream_dst);
}

fr_status fr_restore_fp(fr_plan src, fr_plan dst, void* staging, uint64_t staging_bytes, uint32_t max_retries,
                        uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev, fr_fp* fp_src_dev,
                        fr_fp* fp_dst_dev, void* stream_src, void* stream_dst) {
  CallRange nvtx("fr_restore_fp");
  if (src == nullptr || dst == nullptr) return invalid("plan is null");
  if (n_mismatch_dev == nullptr) return invalid("n_mismatch_dev is null");
  if (cap > 0 && mismatch_dev == nullptr) return invalid("mismatch_dev is null");
  fr_status st = check_same_layout(src, dst);
  if (st != FR_OK) return st;
  DeviceGuard g(dst->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  cudaStream_t ss = static_cast<cudaStream_t>(stream_src), sd = static_cast<cudaStream_t>(stream_dst);
  if (src->n_chunks == 0) {
    cudaError_t e = cudaMemsetAsync(n_mismatch_dev, 0, sizeof(uint64_t), sd);
    return e == cudaSuccess ? FR_OK : cuda_fail(e, "cudaMemsetAsync");
  }
  st = check_packed_buffer(src, staging, staging_bytes);
  if (st != FR_OK) return st;
  uint8_t* buf = static_cast<uint8_t*>(staging);
  FpEntry* fs = reinterpret_cast<FpEntry*>(fp_src_dev);
  FpEntry* fd = reinterpret_cast<FpEntry*>(fp_dst_dev);
  const Decomp& DS = batch_for(src, kModePack);
  const Decomp& DD = batch_for(dst, fd ? kModeUnpackFp : kModeUnpack);
  cudaError_t e;
  // Pipeline: batch b is unpacked on the receiver's stream as soon as the
  // replica's stream has packed it, while the replica packs batch b+1.
  for (uint32_t b = 0; b < src->n_batches; ++b) {
    st = run_batches(src, DS, kModePack, buf, fs, b, b + 1, ss);
    if (st != FR_OK) return st;
    if ((e = cudaEventRecord(src->events[b], ss)) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    if ((e = cudaStreamWaitEvent(sd, src->events[b], 0)) != cudaSuccess) return cuda_fail(e, "cudaStreamWaitEvent");
    st = run_batches(dst, DD, fd ? kModeUnpackFp : kModeUnpack, buf, fd, b, b + 1, sd);
    if (st != FR_OK) return st;
  }
  // Retries: re-send only the chunks that failed, straight from the replica.
  for (uint32_t r = 0; r < max_retries; ++r) {
    uint64_t failing = 0;
    st = resend_failed(src, dst, buf, ss, sd, &failing, fs, fd);
    if (st != FR_OK) return st;
    if (failing == 0) break;
  }
  // Everything queued on the replica's stream is ordered before what follows
  // on the receiver's stream.
  cudaEvent_t ev_end = src->events[src->n_batches];
  if ((e = cudaEventRecord(ev_end, ss)) != cudaSuccess || (e = cudaStreamWaitEvent(sd, ev_end, 0)) != cudaSuccess)
    return cuda_fail(e, "order the end of the restore");
  e = launch_compact_flags(dst->d_flags, dst->n_chunks, mismatch_dev, cap, n_mismatch_dev, dst->d_status, sd);
  return e == cudaSuccess ? FR_OK : cuda_fail(e, "compaction kernel launch");
}

fr_status fr_restore_multi(const fr_plan* src, uint32_t n_src, fr_plan dst, void* staging, uint64_t staging_bytes,
                           uint32_t max_retries, uint32_t* mismatch_dev, uint64_t cap, uint64_t* n_mismatch_dev,
                           fr_fp* fp_dst_dev, void* const* streams_src, void* stream_dst) {
  CallRange nvtx("fr_restore_multi");
  if (src == nullptr || n_src == 0) return invalid("no source plans");
  if (dst == nullptr) return invalid("plan is null");
  if (n_mismatch_dev == nullptr) return invalid("n_mismatch_dev is null");
  if (cap > 0 && mismatch_dev == nullptr) return invalid("mismatch_dev is null");
  for (uint32_t i = 0; i < n_src; ++i) {
    if (src[i] == nullptr) return invalid("a source plan is null");
    fr_status st = check_same_layout(src[i], dst);
    if (st != FR_OK) return st;
  }
  DeviceGuard g(dst->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  cudaStream_t sd = static_cast<cudaStream_t>(stream_dst);
  auto ss = [&](uint32_t i) { return static_cast<cudaStream_t>(streams_src ? streams_src[i] : nullptr); };
  if (dst->n_chunks == 0) {
    cudaError_t e = cudaMemsetAsync(n_mismatch_dev, 0, sizeof(uint64_t), sd);
    return e == cudaSuccess ? FR_OK : cuda_fail(e, "cudaMemsetAsync");
  }
  fr_status st = check_packed_buffer(dst, staging, staging_bytes);
  if (st != FR_OK) return st;
  uint8_t* buf = static_cast<uint8_t*>(staging);
  FpEntry* fd = reinterpret_cast<FpEntry*>(fp_dst_dev);
  const int umode = fd ? kModeUnpackFp : kModeUnpack;
  const Decomp& DD = batch_for(dst, umode);
  cudaError_t e;
  // Batch b is packed by replica b mod n_src on its own stream and unpacked
  // on the receiver's stream as soon as it is packed.
  for (uint32_t b = 0; b < dst->n_batches; ++b) {
    const uint32_t i = b % n_src;
    st = run_batches(src[i], batch_for(src[i], kModePack), kModePack, buf, nullptr, b, b + 1, ss(i));
    if (st != FR_OK) return st;
    if ((e = cudaEventRecord(src[i]->events[b], ss(i))) != cudaSuccess) return cuda_fail(e, "cudaEventRecord");
    if ((e = cudaStreamWaitEvent(sd, src[i]->events[b], 0)) != cudaSuccess)
      return cuda_fail(e, "cudaStreamWaitEvent");
    st = run_batches(dst, DD, umode, buf, fd, b, b + 1, sd);
    if (st != FR_OK) return st;
  }
  // Retries: round r re-sends the failing chunks from replica r mod n_src.
  for (uint32_t r = 0; r < max_retries; ++r) {
    uint64_t failing = 0;
    const uint32_t i = r % n_src;
    st = resend_failed(src[i], dst, buf, ss(i), sd, &failing, nullptr, fd);
    if (st != FR_OK) return st;
    if (failing == 0) break;
  }
  // Everything queued on every replica's stream is ordered before what
  // follows on the receiver's stream.
  for (uint32_t i = 0; i < n_src; ++i) {
    cudaEvent_t ev_end = src[i]->events[src[i]->n_batches];
    if ((e = cudaEventRecord(ev_end, ss(i))) != cudaSuccess || (e = cudaStreamWaitEvent(sd, ev_end, 0)) != cudaSuccess)
      return cuda_fail(e, "order the end of the restore");
  }
  e = launch_compact_flags(dst->d_flags, dst->n_chunks, mismatch_dev, cap, n_mismatch_dev, dst->d_status, sd);
  return e == cudaSuccess ? FR_OK : cuda_fail(e, "compaction kernel launch");
}

fr_status fr_resend(fr_plan src, fr_plan dst, void* staging, uint64_t staging_bytes, uint64_t* n_resent,
                    void* stream_src, void* stream_dst) {
  CallRange nvtx("fr_resend");
  return fr_resend_fp(src, dst, staging, staging_bytes, n_resent, nullptr, nullptr, stream_src, stream_dst);
}

fr_status fr_resend_fp(fr_plan src, fr_plan dst, void* staging, uint64_t staging_bytes, uint64_t* n_resent,
                       fr_fp* fp_src_dev, fr_fp* fp_dst_dev, void* stream_src, void* stream_dst) {
  CallRange nvtx("fr_resend_fp");
  if (src == nullptr || dst == nullptr) return invalid("plan is null");
  fr_status st = check_same_layout(src, dst);
  if (st != FR_OK) return st;
  if (n_resent) *n_resent = 0;
  if (src->n_chunks == 0) return FR_OK;
  st = check_packed_buffer(src, staging, staging_bytes);
  if (st != FR_OK) return st;
  DeviceGuard g(dst->device);
  if (!g.ok) return cuda_fail(cudaGetLastError(), "select plan device");
  uint64_t n = 0;
  st = resend_failed(src, dst, static_cast<uint8_t*>(staging), static_cast<cudaStream_t>(stream_src),
                     static_cast<cudaStream_t>(stream_dst), &n, reinterpret_cast<FpEntry*>(fp_src_dev),
                     reinterpret_cast<FpEntry*>(fp_dst_dev));
  if (n_resent) *n_resent = n;
  return st;
}

fr_status fr_diff(const fr_fp* a_dev, const fr_fp* b_dev, uint64_t n_chunks, uint32_t* diverged_dev, uint64_t cap,
                  uint64_t* n_out_dev, void* stream) {
  CallRange nvtx("fr_diff");
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
  CallRange nvtx("fr_sync_status");
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

fr_status fr_shard_pieces(uint64_t n_elems, uint32_t elem_bytes, uint32_t n_dst, uint32_t rank, uint32_t n_src,
                          fr_piece* out, uint64_t cap, uint64_t* n_pieces) {
  if (n_pieces == nullptr) return invalid("n_pieces is null");
  if (elem_bytes == 0 || n_dst == 0 || n_src == 0) return invalid("elem_bytes, n_dst and n_src must be positive");
  if (rank >= n_dst) return invalid("rank must be below n_dst");
  if (cap > 0 && out == nullptr) return invalid("out is null");
  if (n_elems > UINT64_MAX / elem_bytes) return invalid("the flat group exceeds 2^64 bytes");
  // Every shard holds ceil(n / shards) elements, the last non-empty one the rest.
  const uint64_t per_dst = n_elems / n_dst + (n_elems % n_dst != 0);
  const uint64_t per_src = n_elems / n_src + (n_elems % n_src != 0);
  const uint64_t a = std::min<uint64_t>(static_cast<uint64_t>(rank) * per_dst, n_elems);
  const uint64_t b = std::min<uint64_t>(a + per_dst, n_elems);
  uint64_t n = 0;
  if (a < b) {
    for (uint64_t j = a / per_src; j * per_src < b; ++j) {
      const uint64_t lo = std::max(a, j * per_src), hi = std::min(b, (j + 1) * per_src);
      if (n < cap) {
        fr_piece& pc = out[n];
        pc.source = static_cast<uint32_t>(j);
        pc.reserved = 0;
        pc.src_off = (lo - j * per_src) * elem_bytes;
        pc.dst_off = (lo - a) * elem_bytes;
        pc.nbytes = (hi - lo) * elem_bytes;
      }
      ++n;
    }
  }
  *n_pieces = n;
  if (n > cap) {
    set_err("%llu pieces, the list holds %llu", (unsigned long long)n, (unsigned long long)cap);
    return FR_ERR_CAPACITY;
  }
  return FR_OK;
}

}  // extern "C"
