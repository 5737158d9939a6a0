"""Thin ctypes binding of libflashrec (include/flashrec.h), same names as the C ABI.

Argument marshalling only: every step of the sweep runs in the library's CUDA
kernels.  PyTorch supplies device memory and streams.  If the compiled library
is missing or cannot be loaded, importing this module raises -- there is no
fallback of any kind.
"""
from __future__ import annotations

import ctypes
import os
from typing import List, Optional, Sequence

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libflashrec.so")

FR_OK = 0
FR_ERR_INVALID_ARG = 1
FR_ERR_ALIGNMENT = 2
FR_ERR_BUFFER_TOO_SMALL = 3
FR_ERR_CAPACITY = 4
FR_ERR_PLAN_MISMATCH = 5
FR_ERR_DEVICE_TIMEOUT = 6
FR_ERR_CUDA = 7

FR_DT_BYTES, FR_DT_BF16, FR_DT_F32 = 0, 1, 2
FP_ENTRY_BYTES = 16

_TORCH_TO_FR = {torch.bfloat16: FR_DT_BF16, torch.float32: FR_DT_F32, torch.uint8: FR_DT_BYTES,
                torch.int8: FR_DT_BYTES}


class fr_tensor(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("nbytes", ctypes.c_uint64), ("dtype", ctypes.c_uint32),
                ("flags", ctypes.c_uint32)]


class fr_piece(ctypes.Structure):
    _fields_ = [("source", ctypes.c_uint32), ("reserved", ctypes.c_uint32), ("src_off", ctypes.c_uint64),
                ("dst_off", ctypes.c_uint64), ("nbytes", ctypes.c_uint64)]


class FlashrecError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__("%s: %s (%s)" % (where, fr_status_str(status), fr_last_error()))


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError("libflashrec.so is not built (%s); run __graft_entry__.build()" % LIB_PATH)
    L = ctypes.CDLL(LIB_PATH)
    vp, u64, u32 = ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint32
    u64p = ctypes.POINTER(ctypes.c_uint64)
    L.fr_plan_create.argtypes = [ctypes.POINTER(fr_tensor), u64, u64, ctypes.POINTER(vp)]
    L.fr_plan_info.argtypes = [vp, u64p, u64p, u64p]
    L.fr_plan_chunk.argtypes = [vp, u64, ctypes.POINTER(u32), u64p, u64p, u64p]
    L.fr_plan_destroy.argtypes = [vp]
    L.fr_plan_destroy.restype = None
    L.fr_fingerprint.argtypes = [vp, vp, vp]
    L.fr_pack.argtypes = [vp, vp, u64, vp]
    L.fr_unpack_verify.argtypes = [vp, vp, u64, vp, u64, vp, vp]
    L.fr_diff.argtypes = [vp, vp, u64, vp, u64, vp, vp]
    L.fr_sync_status.argtypes = [vp, vp]
    L.fr_fingerprint_static.argtypes = [ctypes.POINTER(fr_tensor), u64, u64, vp, vp]
    L.fr_plan_create_batched.argtypes = [ctypes.POINTER(fr_tensor), u64, u64, u32, ctypes.POINTER(vp)]
    L.fr_plan_batch.argtypes = [vp, u32, ctypes.POINTER(u32), u64p, u64p]
    L.fr_pack_batch.argtypes = [vp, u32, vp, u64, vp]
    L.fr_unpack_verify_batch.argtypes = [vp, u32, vp, u64, vp]
    L.fr_unpack_collect.argtypes = [vp, vp, u64, vp, vp]
    L.fr_resend.argtypes = [vp, vp, vp, u64, u64p, vp, vp]
    L.fr_restore.argtypes = [vp, vp, vp, u64, u32, vp, u64, vp, vp, vp]
    L.fr_shard_pieces.argtypes = [u64, u32, u32, u32, u32, ctypes.POINTER(fr_piece), u64, u64p]
    L.fr_pack_fp.argtypes = [vp, vp, u64, vp, vp]
    L.fr_unpack_verify_fp.argtypes = [vp, vp, u64, vp, u64, vp, vp, vp]
    L.fr_restore_fp.argtypes = [vp, vp, vp, u64, u32, vp, u64, vp, vp, vp, vp, vp]
    L.fr_resend_fp.argtypes = [vp, vp, vp, u64, u64p, vp, vp, vp, vp]
    L.fr_restore_multi.argtypes = [ctypes.POINTER(vp), u32, vp, vp, u64, u32, vp, u64, vp, vp,
                                   ctypes.POINTER(vp), vp]
    L.fr_status_str.argtypes = [ctypes.c_int]
    L.fr_status_str.restype = ctypes.c_char_p
    L.fr_last_error.argtypes = []
    L.fr_last_error.restype = ctypes.c_char_p
    L.fr_version.argtypes = []
    for name in ["fr_plan_create", "fr_plan_info", "fr_plan_chunk", "fr_fingerprint", "fr_pack",
                 "fr_unpack_verify", "fr_diff", "fr_sync_status", "fr_version", "fr_fingerprint_static",
                 "fr_plan_create_batched", "fr_plan_batch", "fr_pack_batch", "fr_unpack_verify_batch",
                 "fr_unpack_collect", "fr_resend", "fr_restore", "fr_shard_pieces", "fr_pack_fp", "fr_unpack_verify_fp",
                 "fr_restore_fp", "fr_resend_fp", "fr_restore_multi"]:
        getattr(L, name).restype = ctypes.c_int
    return L


lib = _load()


def fr_status_str(status: int) -> str:
    return lib.fr_status_str(status).decode()


def fr_last_error() -> str:
    return lib.fr_last_error().decode()


def fr_version() -> int:
    return lib.fr_version()


def _check(status: int, where: str) -> None:
    if status != FR_OK:
        raise FlashrecError(status, where)


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def fr_dtype_of(t: torch.Tensor) -> int:
    try:
        return _TORCH_TO_FR[t.dtype]
    except KeyError:
        raise ValueError("unsupported dtype %s (bf16, fp32 or bytes)" % t.dtype)


# ---------------------------------------------------------------- C names

def _tensor_array(tensors, dtypes=None):
    arr = (fr_tensor * max(1, len(tensors)))()
    for i, t in enumerate(tensors):
        if t.numel() and not t.is_cuda:
            raise ValueError("tensor %d is not on a CUDA device" % i)
        if not t.is_contiguous():
            raise ValueError("tensor %d is not contiguous" % i)
        arr[i].ptr = t.data_ptr() if t.numel() else 0
        arr[i].nbytes = t.numel() * t.element_size()
        arr[i].dtype = dtypes[i] if dtypes is not None else fr_dtype_of(t)
        arr[i].flags = 0
    return arr


def fr_plan_create(tensors: Sequence[torch.Tensor], chunk_bytes: int, dtypes: Optional[Sequence[int]] = None):
    """Plan over contiguous CUDA tensors.  Returns the opaque handle (int)."""
    h = ctypes.c_void_p()
    _check(lib.fr_plan_create(_tensor_array(tensors, dtypes), len(tensors), chunk_bytes, ctypes.byref(h)),
           "fr_plan_create")
    return h.value


def fr_plan_create_batched(tensors: Sequence[torch.Tensor], chunk_bytes: int, n_batches: int,
                           dtypes: Optional[Sequence[int]] = None):
    h = ctypes.c_void_p()
    _check(lib.fr_plan_create_batched(_tensor_array(tensors, dtypes), len(tensors), chunk_bytes, n_batches,
                                      ctypes.byref(h)), "fr_plan_create_batched")
    return h.value


def fr_plan_batch(plan, batch: int):
    nb, first, n = ctypes.c_uint32(), ctypes.c_uint64(), ctypes.c_uint64()
    _check(lib.fr_plan_batch(plan, batch, ctypes.byref(nb), ctypes.byref(first), ctypes.byref(n)), "fr_plan_batch")
    return nb.value, first.value, n.value


def fr_pack_batch(plan, batch: int, dst: torch.Tensor, stream=None) -> None:
    _check(lib.fr_pack_batch(plan, batch, dst.data_ptr() if dst.numel() else None, dst.numel(), _stream(stream)),
           "fr_pack_batch")


def fr_unpack_verify_batch(plan, batch: int, src: torch.Tensor, stream=None) -> None:
    _check(lib.fr_unpack_verify_batch(plan, batch, src.data_ptr() if src.numel() else None, src.numel(),
                                      _stream(stream)), "fr_unpack_verify_batch")


def fr_unpack_collect(plan, mismatch: Optional[torch.Tensor], count: torch.Tensor, stream=None) -> None:
    cap = 0 if mismatch is None else mismatch.numel()
    _check(lib.fr_unpack_collect(plan, mismatch.data_ptr() if cap else None, cap, count.data_ptr(), _stream(stream)),
           "fr_unpack_collect")


def fr_resend(src_plan, dst_plan, staging: torch.Tensor, stream_src=None, stream_dst=None) -> int:
    n = ctypes.c_uint64()
    _check(lib.fr_resend(src_plan, dst_plan, staging.data_ptr() if staging.numel() else None, staging.numel(),
                         ctypes.byref(n), _stream(stream_src), _stream(stream_dst)), "fr_resend")
    return n.value


def fr_restore(src_plan, dst_plan, staging: torch.Tensor, max_retries: int, mismatch: Optional[torch.Tensor],
               count: torch.Tensor, stream_src=None, stream_dst=None) -> None:
    cap = 0 if mismatch is None else mismatch.numel()
    _check(lib.fr_restore(src_plan, dst_plan, staging.data_ptr() if staging.numel() else None, staging.numel(),
                          max_retries, mismatch.data_ptr() if cap else None, cap, count.data_ptr(),
                          _stream(stream_src), _stream(stream_dst)), "fr_restore")


def _table_ptr(t: Optional[torch.Tensor]):
    return None if t is None else t.data_ptr()


def fr_pack_fp(plan, dst: torch.Tensor, fp: Optional[torch.Tensor], stream=None) -> None:
    """fr_pack that also writes the fingerprint table `fp` (uint8, 16 B per chunk)."""
    _check(lib.fr_pack_fp(plan, dst.data_ptr() if dst.numel() else None, dst.numel() * dst.element_size(),
                          _table_ptr(fp), _stream(stream)), "fr_pack_fp")


def fr_unpack_verify_fp(plan, src: torch.Tensor, mismatch: Optional[torch.Tensor], count: torch.Tensor,
                        fp: Optional[torch.Tensor], stream=None) -> None:
    """fr_unpack_verify that also writes the restored tensors' fingerprint table."""
    cap = 0 if mismatch is None else mismatch.numel()
    _check(lib.fr_unpack_verify_fp(plan, src.data_ptr() if src.numel() else None, src.numel() * src.element_size(),
                                   mismatch.data_ptr() if cap else None, cap, count.data_ptr(), _table_ptr(fp),
                                   _stream(stream)), "fr_unpack_verify_fp")


def fr_restore_fp(src_plan, dst_plan, staging: torch.Tensor, max_retries: int, mismatch: Optional[torch.Tensor],
                  count: torch.Tensor, fp_src: Optional[torch.Tensor], fp_dst: Optional[torch.Tensor],
                  stream_src=None, stream_dst=None) -> None:
    """fr_restore that also writes both fingerprint tables."""
    cap = 0 if mismatch is None else mismatch.numel()
    _check(lib.fr_restore_fp(src_plan, dst_plan, staging.data_ptr() if staging.numel() else None, staging.numel(),
                             max_retries, mismatch.data_ptr() if cap else None, cap, count.data_ptr(),
                             _table_ptr(fp_src), _table_ptr(fp_dst), _stream(stream_src), _stream(stream_dst)),
           "fr_restore_fp")


def fr_resend_fp(src_plan, dst_plan, staging: torch.Tensor, fp_src: Optional[torch.Tensor],
                 fp_dst: Optional[torch.Tensor], stream_src=None, stream_dst=None) -> int:
    """fr_resend that also rewrites the re-sent chunks' fingerprint entries."""
    n = ctypes.c_uint64()
    _check(lib.fr_resend_fp(src_plan, dst_plan, staging.data_ptr() if staging.numel() else None, staging.numel(),
                            ctypes.byref(n), _table_ptr(fp_src), _table_ptr(fp_dst), _stream(stream_src),
                            _stream(stream_dst)), "fr_resend_fp")
    return n.value


def fr_restore_multi(src_plans, dst_plan, staging: torch.Tensor, max_retries: int, mismatch: Optional[torch.Tensor],
                     count: torch.Tensor, fp_dst: Optional[torch.Tensor] = None, streams_src=None,
                     stream_dst=None) -> None:
    """Restore `dst_plan` from several replicas, batch b packed by replica b % len(src_plans)."""
    n = len(src_plans)
    plans = (ctypes.c_void_p * n)(*[p for p in src_plans])
    streams = None
    if streams_src is not None:
        streams = (ctypes.c_void_p * n)(*[_stream(x) for x in streams_src])
    cap = 0 if mismatch is None else mismatch.numel()
    _check(lib.fr_restore_multi(plans, n, dst_plan, staging.data_ptr() if staging.numel() else None, staging.numel(),
                                max_retries, mismatch.data_ptr() if cap else None, cap, count.data_ptr(),
                                _table_ptr(fp_dst), streams, _stream(stream_dst)), "fr_restore_multi")


def fr_plan_info(plan):
    n, packed, state = ctypes.c_uint64(), ctypes.c_uint64(), ctypes.c_uint64()
    _check(lib.fr_plan_info(plan, ctypes.byref(n), ctypes.byref(packed), ctypes.byref(state)), "fr_plan_info")
    return n.value, packed.value, state.value


def fr_plan_chunk(plan, chunk_id: int):
    t, off, ln, poff = ctypes.c_uint32(), ctypes.c_uint64(), ctypes.c_uint64(), ctypes.c_uint64()
    _check(lib.fr_plan_chunk(plan, chunk_id, ctypes.byref(t), ctypes.byref(off), ctypes.byref(ln),
                             ctypes.byref(poff)), "fr_plan_chunk")
    return t.value, off.value, ln.value, poff.value


def fr_plan_destroy(plan) -> None:
    if plan:
        lib.fr_plan_destroy(plan)


def fr_fingerprint(plan, out: torch.Tensor, stream=None) -> None:
    """`out`: CUDA uint8 tensor of n_chunks * 16 bytes (fr_fp entries)."""
    _check(lib.fr_fingerprint(plan, out.data_ptr() if out.numel() else None, _stream(stream)), "fr_fingerprint")


def fr_pack(plan, dst: torch.Tensor, stream=None) -> None:
    """`dst`: uint8 tensor (CUDA, or pinned CPU memory) of >= packed_bytes."""
    _check(lib.fr_pack(plan, dst.data_ptr() if dst.numel() else None, dst.numel() * dst.element_size(),
                       _stream(stream)), "fr_pack")


def fr_unpack_verify(plan, src: torch.Tensor, mismatch: Optional[torch.Tensor], count: torch.Tensor,
                     stream=None, src_bytes: Optional[int] = None) -> None:
    """`mismatch`: CUDA int32/uint32 tensor (capacity = numel); `count`: CUDA int64 tensor of 1."""
    cap = 0 if mismatch is None else mismatch.numel()
    nbytes = src.numel() * src.element_size() if src_bytes is None else src_bytes
    _check(lib.fr_unpack_verify(plan, src.data_ptr() if src.numel() else None, nbytes,
                                mismatch.data_ptr() if cap else None, cap, count.data_ptr(), _stream(stream)),
           "fr_unpack_verify")


def fr_diff(a: torch.Tensor, b: torch.Tensor, n_chunks: int, diverged: Optional[torch.Tensor],
            count: torch.Tensor, stream=None) -> None:
    cap = 0 if diverged is None else diverged.numel()
    _check(lib.fr_diff(a.data_ptr() if n_chunks else None, b.data_ptr() if n_chunks else None, n_chunks,
                       diverged.data_ptr() if cap else None, cap, count.data_ptr(), _stream(stream)), "fr_diff")


def fr_sync_status(plan, stream=None) -> int:
    return lib.fr_sync_status(plan, _stream(stream))


FR_STATIC_MAX_CHUNKS = 16384


def fr_fingerprint_static(tensors: Sequence[torch.Tensor], chunk_bytes: int, out: torch.Tensor,
                          stream=None) -> None:
    """The fingerprint without a plan and without any device allocation, for
    callers that cannot allocate (see include/flashrec.h); `out` holds
    n_chunks * 16 bytes."""
    arr = (fr_tensor * max(1, len(tensors)))()
    for i, t in enumerate(tensors):
        if not t.is_contiguous():
            raise ValueError("tensor %d is not contiguous" % i)
        arr[i].ptr = t.data_ptr() if t.numel() else 0
        arr[i].nbytes = t.numel() * t.element_size()
        arr[i].dtype = fr_dtype_of(t)
        arr[i].flags = 0
    _check(lib.fr_fingerprint_static(arr, len(tensors), chunk_bytes, out.data_ptr() if out.numel() else None,
                                     _stream(stream)), "fr_fingerprint_static")


# ---------------------------------------------------------------- convenience

def fr_shard_pieces(n_elems: int, elem_bytes: int, n_dst: int, rank: int, n_src: int):
    """Pieces of shard `rank` (of `n_dst`) among `n_src` shards of one flat
    group: a list of (source, src_off, dst_off, nbytes), ascending.  Host only."""
    n = ctypes.c_uint64(0)
    cap = max(int(n_src), 1)
    arr = (fr_piece * cap)()
    _check(lib.fr_shard_pieces(n_elems, elem_bytes, n_dst, rank, n_src, arr, cap, ctypes.byref(n)),
           "fr_shard_pieces")
    return [(arr[i].source, arr[i].src_off, arr[i].dst_off, arr[i].nbytes) for i in range(n.value)]


def fp_view(table: torch.Tensor):
    """(crc32c as int64, nonfinite as int64, sumsq as float64) views of a
    fingerprint table held as uint8 [n * 16]."""
    t = table.view(-1, FP_ENTRY_BYTES)
    w = t.view(torch.int32)
    crc = w[:, 0].to(torch.int64) & 0xFFFFFFFF
    nf = w[:, 1].to(torch.int64) & 0xFFFFFFFF
    sumsq = t[:, 8:16].contiguous().view(torch.float64).view(-1)
    return crc, nf, sumsq


class Plan:
    """A plan over a list of CUDA tensors, with allocation helpers."""

    def __init__(self, tensors: Sequence[torch.Tensor], chunk_bytes: int, n_batches: int = 1):
        self.tensors: List[torch.Tensor] = list(tensors)
        self.chunk_bytes = chunk_bytes
        self.device = self.tensors[0].device if self.tensors else torch.device("cuda", torch.cuda.current_device())
        if n_batches > 1:
            self.handle = fr_plan_create_batched(self.tensors, chunk_bytes, n_batches)
        else:
            self.handle = fr_plan_create(self.tensors, chunk_bytes)
        self.n_batches = fr_plan_batch(self.handle, 0)[0] if n_batches > 1 else 1
        self.n_chunks, self.packed_bytes, self.state_bytes = fr_plan_info(self.handle)

    def close(self) -> None:
        if self.handle:
            fr_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def new_table(self) -> torch.Tensor:
        return torch.empty(self.n_chunks * FP_ENTRY_BYTES, dtype=torch.uint8, device=self.device)

    def new_packed(self, pinned: bool = False) -> torch.Tensor:
        if pinned:
            return torch.empty(self.packed_bytes, dtype=torch.uint8, pin_memory=True)
        return torch.empty(self.packed_bytes, dtype=torch.uint8, device=self.device)

    def fingerprint(self, out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        out = self.new_table() if out is None else out
        fr_fingerprint(self.handle, out, stream)
        return out

    def pack(self, dst: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        dst = self.new_packed() if dst is None else dst
        fr_pack(self.handle, dst, stream)
        return dst

    def unpack_verify(self, src: torch.Tensor, cap: Optional[int] = None, stream=None,
                      mismatch: Optional[torch.Tensor] = None, count: Optional[torch.Tensor] = None):
        """Returns (mismatch id tensor (first min(cap, count)), count) after a sync."""
        if mismatch is None:
            cap = self.n_chunks if cap is None else cap
            mismatch = torch.empty(max(cap, 1), dtype=torch.int32, device=self.device)[:cap]
        if count is None:
            count = torch.empty(1, dtype=torch.int64, device=self.device)
        fr_unpack_verify(self.handle, src, mismatch, count, stream)
        n = int(count.item())
        return mismatch[: min(n, mismatch.numel())], n

    def pack_fp(self, dst: Optional[torch.Tensor] = None, table: Optional[torch.Tensor] = None, stream=None):
        """fr_pack_fp: returns (packed buffer, this state's fingerprint table)."""
        dst = self.new_packed() if dst is None else dst
        table = self.new_table() if table is None else table
        fr_pack_fp(self.handle, dst, table, stream)
        return dst, table

    def unpack_verify_fp(self, src: torch.Tensor, table: Optional[torch.Tensor] = None, cap: Optional[int] = None,
                         stream=None):
        """fr_unpack_verify_fp: returns (mismatch ids, count, the restored state's
        fingerprint table) after a sync."""
        cap = self.n_chunks if cap is None else cap
        mismatch = torch.empty(max(cap, 1), dtype=torch.int32, device=self.device)[:cap]
        count = torch.empty(1, dtype=torch.int64, device=self.device)
        table = self.new_table() if table is None else table
        fr_unpack_verify_fp(self.handle, src, mismatch, count, table, stream)
        n = int(count.item())
        return mismatch[: min(n, mismatch.numel())], n, table

    def sync_status(self, stream=None) -> int:
        return fr_sync_status(self.handle, stream)


def diff(a: torch.Tensor, b: torch.Tensor, cap: Optional[int] = None, stream=None):
    n = a.numel() // FP_ENTRY_BYTES
    cap = n if cap is None else cap
    out = torch.empty(max(cap, 1), dtype=torch.int32, device=a.device)[:cap]
    count = torch.empty(1, dtype=torch.int64, device=a.device)
    fr_diff(a, b, n, out, count, stream)
    k = int(count.item())
    return out[: min(k, cap)], k
