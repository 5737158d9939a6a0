"""ctypes wrapper of the plain C CPU reference ("the oracle").

TEST INFRASTRUCTURE ONLY.  Only tests/, ``__graft_entry__.smoke()`` and
``bench.py`` (its cpu_baseline leg and its reference arm) may import this
package.  The product library under ``paper_2509_03047_gb300`` never loads it
and shares no code with it.

The C source (``oracle.c``) states the restoration sweep of FlashRecovery
(arXiv 2509.03047, Sec. III-E, "Model states Restoration"): per-chunk CRC-32C,
non-finite count and fp64 sum of squares; a packed transfer buffer with
checksummed headers; scatter-back with verification; and a fingerprint diff.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_SO = os.path.join(_HERE, "liboracle.so")
_LOCK = threading.Lock()
_LIB = None

DT_BYTES, DT_BF16, DT_F32 = 0, 1, 2
OK, ERR_INVALID_ARG, ERR_BUFFER_TOO_SMALL = 0, 1, 3
HEADER_BYTES = 64
PAYLOAD_ALIGN = 256
CRC32C_POLY = 0x82F63B78

FP_DTYPE = np.dtype([("crc32c", "<u4"), ("nonfinite", "<u4"), ("sumsq", "<f8")])
CHUNK_DTYPE = np.dtype(
    [
        ("tensor_idx", "<u4"),
        ("dtype", "<u4"),
        ("tensor_off", "<u8"),
        ("len", "<u8"),
        ("payload_off", "<u8"),
    ]
)


class _OrFp(ctypes.Structure):
    _fields_ = [("crc32c", ctypes.c_uint32), ("nonfinite", ctypes.c_uint32), ("sumsq", ctypes.c_double)]


class _OrChunk(ctypes.Structure):
    _fields_ = [
        ("tensor_idx", ctypes.c_uint32),
        ("dtype", ctypes.c_uint32),
        ("tensor_off", ctypes.c_uint64),
        ("len", ctypes.c_uint64),
        ("payload_off", ctypes.c_uint64),
    ]


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (plain C11, no FMA contraction)."""
    with _LOCK:
        if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < max(
            os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "oracle.h"))
        ):
            tmp = _SO + ".tmp%d" % os.getpid()
            subprocess.check_call(
                ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-Wall",
                 "-fPIC", "-shared", _SRC, "-o", tmp]
            )
            os.replace(tmp, _SO)
    return _SO


def use_library(path=None) -> None:
    """Load the oracle from another compiled copy (None: the default build).
    Tests use this to run the pins against deliberately broken copies."""
    global _LIB
    _LIB = None
    if path is not None:
        _LIB = _bind(ctypes.CDLL(path))


def lib() -> ctypes.CDLL:
    global _LIB
    if _LIB is None:
        build()
        _LIB = _bind(ctypes.CDLL(_SO))
    return _LIB


def _bind(L: ctypes.CDLL) -> ctypes.CDLL:
    u32p, u64p = ctypes.POINTER(ctypes.c_uint32), ctypes.POINTER(ctypes.c_uint64)
    c_u32, c_u64 = ctypes.c_uint32, ctypes.c_uint64
    L.or_crc_bitwise.argtypes = [c_u32, c_u32, c_u32, ctypes.c_void_p, c_u64]
    L.or_crc_bitwise.restype = c_u32
    L.or_crc_table.argtypes = [c_u32, c_u32, c_u32, ctypes.c_void_p, c_u64]
    L.or_crc_table.restype = c_u32
    L.or_crc_combine.argtypes = [c_u32, c_u32, c_u32, c_u64]
    L.or_crc_combine.restype = c_u32
    L.or_crc32c.argtypes = [ctypes.c_void_p, c_u64]
    L.or_crc32c.restype = c_u32
    L.or_crc32c_combine.argtypes = [c_u32, c_u32, c_u64]
    L.or_crc32c_combine.restype = c_u32
    L.or_fp_values.argtypes = [ctypes.c_void_p, c_u64, c_u32, u32p, ctypes.POINTER(ctypes.c_double)]
    L.or_fp_values.restype = None
    L.or_fingerprint_chunk.argtypes = [ctypes.c_void_p, c_u64, c_u32, ctypes.POINTER(_OrFp)]
    L.or_fingerprint_chunk.restype = None
    L.or_plan.argtypes = [u64p, u32p, c_u64, c_u64, ctypes.c_void_p, c_u64, u64p]
    L.or_plan.restype = c_u64
    L.or_header.argtypes = [ctypes.POINTER(_OrChunk), c_u64, ctypes.POINTER(_OrFp), ctypes.c_void_p]
    L.or_header.restype = None
    L.or_fingerprint.argtypes = [ctypes.POINTER(ctypes.c_void_p), u64p, u32p, c_u64, c_u64, ctypes.c_void_p]
    L.or_fingerprint.restype = ctypes.c_int
    L.or_pack.argtypes = [ctypes.POINTER(ctypes.c_void_p), u64p, u32p, c_u64, c_u64, ctypes.c_void_p, c_u64]
    L.or_pack.restype = ctypes.c_int
    L.or_unpack_verify.argtypes = [ctypes.POINTER(ctypes.c_void_p), u64p, u32p, c_u64, c_u64,
                                   ctypes.c_void_p, c_u64, u32p, c_u64, u64p]
    L.or_unpack_verify.restype = ctypes.c_int
    L.or_verify_chunk.argtypes = [ctypes.POINTER(_OrChunk), c_u64, ctypes.c_void_p, ctypes.c_void_p,
                                  ctypes.c_void_p, c_u64]
    L.or_verify_chunk.restype = ctypes.c_int
    L.or_diff.argtypes = [ctypes.c_void_p, ctypes.c_void_p, c_u64, u32p, c_u64]
    L.or_diff.restype = c_u64
    return L


# ---------------------------------------------------------------- helpers

def _as_u8(buf) -> np.ndarray:
    """A C-contiguous uint8 view of bytes / bytearray / numpy array."""
    if isinstance(buf, (bytes, bytearray, memoryview)):
        return np.frombuffer(bytes(buf), dtype=np.uint8)
    a = np.ascontiguousarray(buf)
    return a.reshape(-1).view(np.uint8)


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data if a.size else 0


def _u64s(vals):
    return (ctypes.c_uint64 * max(1, len(vals)))(*[int(v) for v in vals])


def _u32s(vals):
    return (ctypes.c_uint32 * max(1, len(vals)))(*[int(v) for v in vals])


def _ptrs(arrs):
    return (ctypes.c_void_p * max(1, len(arrs)))(*[_ptr(a) for a in arrs])


# ---------------------------------------------------------------- CRC

def crc_bitwise(poly: int, init: int, xorout: int, data) -> int:
    a = _as_u8(data)
    return int(lib().or_crc_bitwise(poly, init, xorout, _ptr(a), a.size))


def crc_table(poly: int, init: int, xorout: int, data) -> int:
    a = _as_u8(data)
    return int(lib().or_crc_table(poly, init, xorout, _ptr(a), a.size))


def crc_combine(poly: int, crc_a: int, crc_b: int, len_b: int) -> int:
    return int(lib().or_crc_combine(poly, crc_a, crc_b, len_b))


def crc32c(data) -> int:
    a = _as_u8(data)
    return int(lib().or_crc32c(_ptr(a), a.size))


def crc32c_combine(crc_a: int, crc_b: int, len_b: int) -> int:
    return int(lib().or_crc32c_combine(crc_a, crc_b, len_b))


# ---------------------------------------------------------------- fingerprint

def fp_values(data, dtype: int):
    a = _as_u8(data)
    nf = ctypes.c_uint32()
    s = ctypes.c_double()
    lib().or_fp_values(_ptr(a), a.size, dtype, ctypes.byref(nf), ctypes.byref(s))
    return int(nf.value), float(s.value)


def fingerprint_chunk(data, dtype: int):
    a = _as_u8(data)
    out = _OrFp()
    lib().or_fingerprint_chunk(_ptr(a), a.size, dtype, ctypes.byref(out))
    return int(out.crc32c), int(out.nonfinite), float(out.sumsq)


# ---------------------------------------------------------------- plan

def plan(nbytes, dtypes, chunk_bytes: int):
    """(chunks as a CHUNK_DTYPE array, packed_bytes); raises on invalid input."""
    nb, dt = _u64s(nbytes), _u32s(dtypes)
    packed = ctypes.c_uint64()
    n = lib().or_plan(nb, dt, len(nbytes), chunk_bytes, None, 0, ctypes.byref(packed))
    if n == 2**64 - 1:
        raise ValueError("invalid plan arguments")
    out = np.zeros(n, dtype=CHUNK_DTYPE)
    lib().or_plan(nb, dt, len(nbytes), chunk_bytes, _ptr(out) or None, n, ctypes.byref(packed))
    return out, int(packed.value)


def header(chunk, chunk_id: int, fp) -> bytes:
    ch = _OrChunk(int(chunk["tensor_idx"]), int(chunk["dtype"]), int(chunk["tensor_off"]),
                  int(chunk["len"]), int(chunk["payload_off"]))
    f = _OrFp(int(fp[0]), int(fp[1]), float(fp[2]))
    h = np.zeros(64, dtype=np.uint8)
    lib().or_header(ctypes.byref(ch), chunk_id, ctypes.byref(f), _ptr(h))
    return h.tobytes()


def verify_chunk(chunk, chunk_id: int, header_bytes, payload_and_padding, gap=None) -> bool:
    """The oracle's unpack verdict for one chunk (True: it fails a check).
    `payload_and_padding` holds the chunk's payload and its zero padding
    (len rounded up to 256 bytes); `gap` the zero gap after the header table,
    passed for the last chunk only."""
    ch = _OrChunk(int(chunk["tensor_idx"]), int(chunk["dtype"]), int(chunk["tensor_off"]),
                  int(chunk["len"]), int(chunk["payload_off"]))
    h = _as_u8(header_bytes)
    p = _as_u8(payload_and_padding)
    assert h.size == HEADER_BYTES
    assert p.size == (int(chunk["len"]) + PAYLOAD_ALIGN - 1) // PAYLOAD_ALIGN * PAYLOAD_ALIGN
    g = _as_u8(gap) if gap is not None else np.zeros(0, dtype=np.uint8)
    return bool(lib().or_verify_chunk(ctypes.byref(ch), chunk_id, _ptr(h), _ptr(p) or None,
                                      _ptr(g) or None, g.size))


# ---------------------------------------------------------------- whole state

def fingerprint(tensors, dtypes, chunk_bytes: int) -> np.ndarray:
    arrs = [_as_u8(t) for t in tensors]
    chunks, _ = plan([a.size for a in arrs], dtypes, chunk_bytes)
    out = np.zeros(len(chunks), dtype=FP_DTYPE)
    rc = lib().or_fingerprint(_ptrs(arrs), _u64s([a.size for a in arrs]), _u32s(dtypes), len(arrs),
                              chunk_bytes, _ptr(out) or None)
    if rc != OK:
        raise ValueError("or_fingerprint failed: %d" % rc)
    return out


def pack(tensors, dtypes, chunk_bytes: int) -> np.ndarray:
    arrs = [_as_u8(t) for t in tensors]
    _, packed = plan([a.size for a in arrs], dtypes, chunk_bytes)
    dst = np.zeros(packed, dtype=np.uint8)
    rc = lib().or_pack(_ptrs(arrs), _u64s([a.size for a in arrs]), _u32s(dtypes), len(arrs), chunk_bytes,
                       _ptr(dst) or None, packed)
    if rc != OK:
        raise ValueError("or_pack failed: %d" % rc)
    return dst


def unpack_verify(dst_tensors, dtypes, chunk_bytes: int, src, cap=None, src_bytes=None):
    """Scatter `src` into the writable uint8 arrays `dst_tensors` (in place).

    Returns (status, mismatch ids as uint32 array (first `cap`), true count)."""
    arrs = [t for t in dst_tensors]
    for a in arrs:
        assert a.dtype == np.uint8 and a.flags["C_CONTIGUOUS"] and a.flags["WRITEABLE"]
    s = _as_u8(src)
    chunks, _ = plan([a.size for a in arrs], dtypes, chunk_bytes)
    if cap is None:
        cap = len(chunks)
    ids = np.zeros(max(1, cap), dtype=np.uint32)
    n = ctypes.c_uint64()
    rc = lib().or_unpack_verify(_ptrs(arrs), _u64s([a.size for a in arrs]), _u32s(dtypes), len(arrs),
                                chunk_bytes, _ptr(s) or None, s.size if src_bytes is None else src_bytes,
                                ids.ctypes.data_as(ctypes.POINTER(ctypes.c_uint32)), cap, ctypes.byref(n))
    return rc, ids[: min(cap, n.value)].copy(), int(n.value)


def diff(a: np.ndarray, b: np.ndarray, cap=None):
    assert a.dtype == FP_DTYPE and b.dtype == FP_DTYPE and a.size == b.size
    if cap is None:
        cap = a.size
    ids = np.zeros(max(1, cap), dtype=np.uint32)
    n = lib().or_diff(_ptr(a) or None, _ptr(b) or None, a.size,
                      ids.ctypes.data_as(ctypes.POINTER(ctypes.c_uint32)), cap)
    return ids[: min(cap, n)].copy(), int(n)
