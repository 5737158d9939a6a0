"""Shared helpers of the GPU parity tests: run the CUDA path through the
C-ABI binding and the CPU oracle on the same seeded inputs, and compare."""
import numpy as np
import torch

import oracle
from paper_2509_03047_gb300 import flashrec as fr
from paper_2509_03047_gb300 import synth

SUMSQ_RTOL = 1e-9  # the fp64 sums of squares agree within 1e-9 relative

# Every output buffer a test hands the library is followed by GUARD_BYTES of
# GUARD_FILL; after the call the guard must be intact, so a kernel writing
# past the end of an output is caught (compute-sanitizer is not available).
GUARD_BYTES = 4096
GUARD_FILL = 0x5A


class Guarded:
    """A uint8 output buffer of `nbytes` followed by a guard region."""

    def __init__(self, nbytes, device="cuda", pinned=False, fill=GUARD_FILL):
        self.nbytes = int(nbytes)
        self.fill = fill
        if pinned:
            self.whole = torch.empty(self.nbytes + GUARD_BYTES, dtype=torch.uint8, pin_memory=True)
            self.whole.fill_(fill)
        else:
            self.whole = torch.full((self.nbytes + GUARD_BYTES,), fill, dtype=torch.uint8, device=device)
        self.buf = self.whole[: self.nbytes]

    def view(self, dtype):
        return self.buf.view(dtype) if self.nbytes else torch.empty(0, dtype=dtype, device=self.whole.device)

    def check(self, what="output"):
        tail = self.whole[self.nbytes:]
        bad = torch.nonzero(tail != self.fill)
        assert bad.numel() == 0, "%s: %d guard bytes past the end were written (first at +%d)" % (
            what, bad.numel(), int(bad[0]))


def guarded_outputs(n_chunks, cap=None, device="cuda"):
    """Guarded fingerprint table, mismatch list (int32 x cap) and count word."""
    cap = n_chunks if cap is None else cap
    return Guarded(16 * n_chunks, device), Guarded(4 * cap, device), Guarded(8, device)


def fr_diff_guarded(a, b, n_chunks, cap=None):
    """fr_diff into guarded outputs; returns (ids, count) after checking the guards."""
    cap = n_chunks if cap is None else cap
    out, cnt = Guarded(4 * cap), Guarded(8)
    fr.fr_diff(a, b, n_chunks, out.view(torch.int32) if cap else None, cnt.view(torch.int64))
    torch.cuda.synchronize()
    out.check("diff list")
    cnt.check("diff count")
    k = int(cnt.view(torch.int64).item())
    return out.view(torch.int32)[: min(k, cap)], k


def host_bytes(tensors):
    return [t.contiguous().view(torch.uint8).cpu().numpy().reshape(-1) for t in tensors]


def table_np(table: torch.Tensor) -> np.ndarray:
    return table.cpu().numpy().view(oracle.FP_DTYPE)


def assert_tables_match(got: np.ndarray, want: np.ndarray, what=""):
    assert got.shape == want.shape, what
    bad = np.nonzero(got["crc32c"] != want["crc32c"])[0]
    assert bad.size == 0, "%s crc32c differs at chunks %s" % (what, bad[:10])
    bad = np.nonzero(got["nonfinite"] != want["nonfinite"])[0]
    assert bad.size == 0, "%s nonfinite differs at chunks %s" % (what, bad[:10])
    g, w = got["sumsq"], want["sumsq"]
    zero = w == 0.0
    assert np.array_equal(g[zero], w[zero]), "%s zero sums must be exact" % what
    rel = np.abs(g[~zero] - w[~zero]) / np.abs(w[~zero])
    assert rel.size == 0 or rel.max() <= SUMSQ_RTOL, "%s sumsq rel err %g" % (what, rel.max())


def expected_mismatch(chunks: np.ndarray, bit_positions: np.ndarray) -> np.ndarray:
    """Chunks owning a flipped byte: header k -> k; table gap -> last chunk;
    payload or its padding -> that chunk (independent of both implementations'
    verification code; from the documented layout)."""
    if bit_positions.size == 0 or chunks.size == 0:
        return np.zeros(0, dtype=np.int64)
    C = chunks.size
    b = bit_positions // 8
    starts = chunks["payload_off"].astype(np.int64)
    owner = np.where(b < 64 * C, b // 64, -1)
    gap = (b >= 64 * C) & (b < starts[0])
    owner = np.where(gap, C - 1, owner)
    pay = b >= starts[0]
    owner = np.where(pay, np.searchsorted(starts, b, side="right") - 1, owner)
    return np.unique(owner)


def payload_flip_chunks(chunks: np.ndarray, bit_positions: np.ndarray) -> np.ndarray:
    """Chunks whose payload bytes (not header or padding) took a flip."""
    if bit_positions.size == 0:
        return np.zeros(0, dtype=np.int64)
    b = bit_positions // 8
    starts = chunks["payload_off"].astype(np.int64)
    i = np.searchsorted(starts, b, side="right") - 1
    ok = (i >= 0) & (b >= starts[0])
    ii = np.clip(i, 0, None)
    ok &= b < starts[ii] + chunks["len"][ii].astype(np.int64)
    return np.unique(i[ok])


def restored_like(tensors, fill=0xA5):
    """Fresh destination tensors shaped like `tensors`, each at a 256-byte
    aligned offset of one buffer pre-filled with `fill` and followed by
    GUARD_BYTES of it.  Returns (tensors, check) where check() asserts that
    nothing outside the tensors was written."""
    offs, o = [], 0
    for t in tensors:
        offs.append(o)
        o += (t.numel() * t.element_size() + 255) // 256 * 256 + GUARD_BYTES
    whole = torch.full((max(o, 1),), fill, dtype=torch.uint8, device="cuda")
    out = []
    for t, off in zip(tensors, offs):
        nb = t.numel() * t.element_size()
        out.append(whole[off: off + nb].view(t.dtype) if nb else torch.empty(0, dtype=t.dtype, device="cuda"))

    def check():
        mask = torch.ones(whole.numel(), dtype=torch.bool, device="cuda")
        for t, off in zip(tensors, offs):
            mask[off: off + t.numel() * t.element_size()] = False
        outside = whole[mask]
        bad = int((outside != fill).sum())
        assert bad == 0, "%d bytes outside the destination tensors were written" % bad

    return out, check


def run_full(tensors, chunk_bytes, flips=None, cap=None):
    """CUDA path over `tensors`: fingerprint, pack, optional flips, unpack into
    fresh tensors, fingerprint of the restored state, diff.  Every output sits
    in front of a guard region that is checked after the calls.  Returns a
    dict."""
    plan = fr.Plan(tensors, chunk_bytes)
    C, P = plan.n_chunks, plan.packed_bytes
    g_tab, g_pack = Guarded(16 * C), Guarded(P)
    table = plan.fingerprint(out=g_tab.buf)
    packed = plan.pack(g_pack.buf)
    torch.cuda.synchronize()
    g_tab.check("fingerprint table")
    g_pack.check("packed buffer")
    if flips is not None and flips.size:
        synth.apply_flips(packed, flips)
    restored, check_restored = restored_like(tensors)
    plan_r = fr.Plan(restored, chunk_bytes)
    g_tab_r, g_ids, g_cnt = guarded_outputs(C, cap)
    ids, n = plan_r.unpack_verify(packed, mismatch=g_ids.view(torch.int32), count=g_cnt.view(torch.int64))
    status = plan_r.sync_status()
    table_r = plan_r.fingerprint(out=g_tab_r.buf)
    torch.cuda.synchronize()
    g_ids.check("mismatch list")
    g_cnt.check("mismatch count")
    g_tab_r.check("restored fingerprint table")
    check_restored()
    div, nd = fr_diff_guarded(table, table_r, C)
    out = dict(plan=plan, plan_r=plan_r, table=table, packed=packed, restored=restored, ids=ids, n=n,
               status=status, table_r=table_r, div=div, nd=nd)
    return out


def oracle_full(tensors_host, dtypes, chunk_bytes, flips=None, sumsq_override=None):
    """The oracle's results.  The packed headers carry each chunk's sum of
    squares, which the GPU matches to 1e-9 relative, not bit for bit; with
    `sumsq_override` (the GPU's sums) the oracle writes those values into its
    headers (and its header CRC over them), so every other packed byte can be
    compared exactly."""
    want_table = oracle.fingerprint(tensors_host, dtypes, chunk_bytes)
    packed = oracle.pack(tensors_host, dtypes, chunk_bytes)
    if sumsq_override is not None:
        chunks, _ = oracle.plan([h.size for h in tensors_host], dtypes, chunk_bytes)
        for c in range(chunks.size):
            fp = (int(want_table["crc32c"][c]), int(want_table["nonfinite"][c]), float(sumsq_override[c]))
            packed[64 * c: 64 * c + 64] = np.frombuffer(oracle.header(chunks[c], c, fp), dtype=np.uint8)
    if flips is not None:
        for p in flips:
            packed[p // 8] ^= np.uint8(1 << (p % 8))
    dst = [np.zeros_like(h) for h in tensors_host]
    rc, ids, n = oracle.unpack_verify(dst, dtypes, chunk_bytes, packed)
    assert rc == 0
    return dict(table=want_table, packed=packed, restored=dst, ids=ids, n=n)


def compare_full(tensors, chunk_bytes, flips=None):
    """Whole-state parity: every table entry, every packed byte, the mismatch
    list and every restored byte."""
    dtypes = [fr.fr_dtype_of(t) for t in tensors]
    got = run_full(tensors, chunk_bytes, flips)
    host = host_bytes(tensors)
    gt = table_np(got["table"])
    want = oracle_full(host, dtypes, chunk_bytes, flips, sumsq_override=gt["sumsq"])
    assert_tables_match(gt, want["table"], "fingerprint")
    gp = got["packed"].cpu().numpy()
    assert gp.size == want["packed"].size
    if not np.array_equal(gp, want["packed"]):
        diff = np.nonzero(gp != want["packed"])[0]
        raise AssertionError("packed bytes differ at %d offsets, first %s" % (diff.size, diff[:10]))
    assert got["n"] == want["n"]
    assert np.array_equal(got["ids"].cpu().numpy().astype(np.uint32), want["ids"])
    for i, (g, w) in enumerate(zip(host_bytes(got["restored"]), want["restored"])):
        assert np.array_equal(g, w), "restored tensor %d differs" % i
    assert got["status"] == fr.FR_OK
    # diff against the oracle's diff of its own two tables
    want_r = oracle.fingerprint(want["restored"], dtypes, chunk_bytes)
    ref_div, ref_nd = oracle.diff(want["table"], want_r)
    assert got["nd"] == ref_nd
    assert np.array_equal(got["div"].cpu().numpy().astype(np.uint32), ref_div)
    return got, want


def odd_tensors(seed=0, offset=0):
    """Tensors of awkward sizes (empty, a few bytes, just over and under 512-byte
    blocks and 16 KiB segments, several MiB), each a view starting `offset`
    bytes into its buffer where the element size allows (else aligned)."""
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    sizes = [(torch.float32, 0), (torch.bfloat16, 6), (torch.float32, 4), (torch.float32, 20),
             (torch.uint8, 13), (torch.bfloat16, 1000), (torch.float32, 4096), (torch.float32, 4100),
             (torch.bfloat16, 8194), (torch.float32, 3 * 1024 + 12), (torch.float32, 512),
             (torch.float32, 511 * 4), (torch.bfloat16, 70000), (torch.float32, 1 << 20),
             (torch.float32, (1 << 20) + 516), (torch.uint8, 100003), (torch.bfloat16, 262144 * 2 + 2)]
    out = []
    for dt, nbytes in sizes:
        if dt == torch.uint8:
            base = torch.randint(0, 256, (nbytes + 16,), generator=g, device="cuda", dtype=torch.uint8)
            out.append(base[offset:offset + nbytes])
            continue
        esz = 4 if dt == torch.float32 else 2
        n = nbytes // esz
        eo = offset // esz if offset % esz == 0 else 0
        base = torch.randn(n + 8, generator=g, device="cuda", dtype=torch.float32).to(dt)
        out.append(base[eo:eo + n])
    return out
