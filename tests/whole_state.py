"""Whole-state parity at any size: every chunk of the CUDA path's outputs
against the CPU oracle, the oracle's per-chunk functions spread over the host's
cores.

The oracle itself stays single-threaded: each call of `or_fingerprint_chunk`,
`or_header` or `or_verify_chunk` runs on one thread, and only this harness
runs many such calls at once, on Python threads (ctypes releases the GIL
around foreign calls).  The state is streamed through host memory in slices
of at most SLICE_BYTES, so host memory stays bounded at any state size.

Pass 1 (after fingerprint and pack) compares, for every chunk, the GPU's table
entry with the oracle's fingerprint of the chunk's bytes, the GPU's 64-byte
header with the oracle's header (written with the GPU's sum of squares once
that sum is within tolerance, since the header carries it), the payload with
the source bytes and the padding with zeros -- together, the oracle's packed
buffer byte for byte.  Pass 2 (after unpack_verify of the possibly damaged
buffer) compares the mismatch list with the oracle's per-chunk verdicts, every
restored byte with the payload the oracle would copy, the restored state's
table with the oracle's fingerprint of the restored bytes, and the GPU diff of
the two tables with the oracle's diff of its own two tables.
"""
from __future__ import annotations

import os
import time
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import torch

import oracle

SUMSQ_RTOL = 1e-9
SLICE_BYTES = 2 << 30


def host_threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def _a256(v: int) -> int:
    return (v + 255) // 256 * 256


def _slices(lens: np.ndarray, limit: int):
    """Consecutive chunk ranges [c0, c1) of at most `limit` payload bytes (a
    larger chunk stands alone)."""
    out, c0, acc = [], 0, 0
    for c, ln in enumerate(lens.tolist()):
        if c > c0 and acc + ln > limit:
            out.append((c0, c))
            c0, acc = c, 0
        acc += ln
    if len(lens) > c0:
        out.append((c0, len(lens)))
    return out


def _tasks(lens: np.ndarray, c0: int, c1: int, n: int):
    """Split [c0, c1) into about `n` ranges of similar byte counts."""
    tot = int(lens[c0:c1].sum())
    per = max(1, tot // max(1, n))
    out, a, acc = [], c0, 0
    for c in range(c0, c1):
        acc += int(lens[c])
        if acc >= per:
            out.append((a, c + 1))
            a, acc = c + 1, 0
    if a < c1:
        out.append((a, c1))
    return out


def _gather(raw, chunks, c0, c1):
    """Host copy of chunks [c0, c1)'s bytes, concatenated in chunk order, and
    each chunk's offset in it."""
    pieces, t_prev, lo, hi = [], None, 0, 0
    for c in range(c0, c1):
        t, off, ln = int(chunks["tensor_idx"][c]), int(chunks["tensor_off"][c]), int(chunks["len"][c])
        if t == t_prev and off == hi:
            hi = off + ln
            continue
        if t_prev is not None:
            pieces.append(raw[t_prev][lo:hi])
        t_prev, lo, hi = t, off, off + ln
    if t_prev is not None:
        pieces.append(raw[t_prev][lo:hi])
    dev = torch.cat(pieces) if len(pieces) > 1 else pieces[0].clone()
    host = dev.cpu().numpy()
    del dev
    lens = chunks["len"][c0:c1].astype(np.int64)
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]])
    return host, starts


class WholeState:
    """Oracle-side results of the two passes over one state."""

    def __init__(self, tensors, dtypes, chunk_bytes, threads=None):
        self.raw = [t.view(torch.uint8).reshape(-1) for t in tensors]
        self.dtypes = list(dtypes)
        self.chunk_bytes = chunk_bytes
        self.chunks, self.packed_bytes = oracle.plan([r.numel() for r in self.raw], self.dtypes, chunk_bytes)
        self.C = len(self.chunks)
        self.lens = self.chunks["len"].astype(np.int64)
        self.poff = self.chunks["payload_off"].astype(np.int64)
        self.threads = threads or host_threads()
        self.table = np.zeros(self.C, dtype=oracle.FP_DTYPE)     # oracle, of the source
        self.table_r = np.zeros(self.C, dtype=oracle.FP_DTYPE)   # oracle, of the restored bytes
        self.verdict = np.zeros(self.C, dtype=bool)
        self.seconds = {}
        oracle.crc32c(b"")  # build the oracle's CRC table before any thread uses it

    def _packed_span(self, packed, c0, c1):
        hdr = packed[64 * c0: 64 * c1].cpu().numpy()
        lo, hi = int(self.poff[c0]), int(self.poff[c1 - 1] + _a256(int(self.lens[c1 - 1])))
        return hdr, packed[lo:hi].cpu().numpy(), lo

    def check_pack(self, gpu_table: np.ndarray, packed: torch.Tensor):
        """Pass 1.  Returns a list of (chunk, what) failures (empty: parity)."""
        t0 = time.perf_counter()
        assert packed.numel() == self.packed_bytes
        fails = []
        if self.C:
            gap = packed[64 * self.C: int(self.poff[0])]
            if int(gap.count_nonzero()):
                fails.append((self.C - 1, "table gap not zero"))
        for c0, c1 in _slices(self.lens, SLICE_BYTES):
            src, s_off = _gather(self.raw, self.chunks, c0, c1)
            hdr, pay, p_lo = self._packed_span(packed, c0, c1)

            def work(a, b):
                bad = []
                for c in range(a, b):
                    ln, dt = int(self.lens[c]), int(self.chunks["dtype"][c])
                    so = int(s_off[c - c0])
                    data = src[so: so + ln]
                    crc, nf, s = oracle.fingerprint_chunk(data, dt)
                    self.table[c] = (crc, nf, s)
                    g = gpu_table[c]
                    gs = float(g["sumsq"])
                    if int(g["crc32c"]) != crc or int(g["nonfinite"]) != nf:
                        bad.append((c, "crc32c/nonfinite"))
                    if not ((s == 0.0 and gs == 0.0) or
                            (s != 0.0 and abs(gs - s) <= SUMSQ_RTOL * abs(s))):
                        bad.append((c, "sumsq %r vs %r" % (gs, s)))
                    want_h = oracle.header(self.chunks[c], c, (crc, nf, gs))
                    if hdr[64 * (c - c0): 64 * (c - c0) + 64].tobytes() != want_h:
                        bad.append((c, "header"))
                    po = int(self.poff[c]) - p_lo
                    if not np.array_equal(pay[po: po + ln], data):
                        bad.append((c, "payload"))
                    if pay[po + ln: po + _a256(ln)].any():
                        bad.append((c, "padding"))
                return bad

            with ThreadPoolExecutor(self.threads) as ex:
                for r in ex.map(lambda ab: work(*ab), _tasks(self.lens, c0, c1, 4 * self.threads)):
                    fails += r
            del src, hdr, pay
        self.seconds["pack_pass"] = time.perf_counter() - t0
        return fails

    def check_restore(self, packed: torch.Tensor, restored, gpu_table_r: np.ndarray):
        """Pass 2.  Returns (failures, oracle mismatch ids)."""
        t0 = time.perf_counter()
        raw_r = [t.view(torch.uint8).reshape(-1) for t in restored]
        fails = []
        gap = packed[64 * self.C: int(self.poff[0])].cpu().numpy() if self.C else None
        for c0, c1 in _slices(self.lens, SLICE_BYTES):
            rest, r_off = _gather(raw_r, self.chunks, c0, c1)
            hdr, pay, p_lo = self._packed_span(packed, c0, c1)

            def work(a, b):
                bad = []
                for c in range(a, b):
                    ln, dt = int(self.lens[c]), int(self.chunks["dtype"][c])
                    po = int(self.poff[c]) - p_lo
                    self.verdict[c] = oracle.verify_chunk(self.chunks[c], c, hdr[64 * (c - c0): 64 * (c - c0) + 64],
                                                          pay[po: po + _a256(ln)],
                                                          gap if c == self.C - 1 else None)
                    ro = int(r_off[c - c0])
                    data = rest[ro: ro + ln]
                    if not np.array_equal(data, pay[po: po + ln]):
                        bad.append((c, "restored bytes"))
                    crc, nf, s = oracle.fingerprint_chunk(data, dt)
                    self.table_r[c] = (crc, nf, s)
                    g = gpu_table_r[c]
                    gs = float(g["sumsq"])
                    if int(g["crc32c"]) != crc or int(g["nonfinite"]) != nf:
                        bad.append((c, "restored crc32c/nonfinite"))
                    if not ((s == 0.0 and gs == 0.0) or
                            (s != 0.0 and abs(gs - s) <= SUMSQ_RTOL * abs(s))):
                        bad.append((c, "restored sumsq %r vs %r" % (gs, s)))
                return bad

            with ThreadPoolExecutor(self.threads) as ex:
                for r in ex.map(lambda ab: work(*ab), _tasks(self.lens, c0, c1, 4 * self.threads)):
                    fails += r
            del rest, hdr, pay
        self.seconds["restore_pass"] = time.perf_counter() - t0
        return fails, np.nonzero(self.verdict)[0].astype(np.uint32)

    def oracle_diff(self):
        """The oracle's diff of its own two tables."""
        ids, n = oracle.diff(self.table, self.table_r)
        return ids, n
