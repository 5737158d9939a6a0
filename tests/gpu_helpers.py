"""Shared helpers of the GPU parity tests: run the CUDA path through the
C-ABI binding and the CPU oracle on the same seeded inputs, and compare."""
import numpy as np
import torch

import oracle
from paper_2509_03047_gb300 import flashrec as fr
from paper_2509_03047_gb300 import synth

SUMSQ_RTOL = 1e-9  # the fp64 sums of squares agree within 1e-9 relative


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


def run_full(tensors, chunk_bytes, flips=None, cap=None):
    """CUDA path over `tensors`: fingerprint, pack, optional flips, unpack into
    fresh tensors, fingerprint of the restored state.  Returns a dict."""
    plan = fr.Plan(tensors, chunk_bytes)
    table = plan.fingerprint()
    packed = plan.pack()
    if flips is not None and flips.size:
        synth.apply_flips(packed, flips)
    restored = [torch.full_like(t.view(torch.uint8), 0xA5).view(t.dtype) if t.numel() else torch.empty_like(t)
                for t in tensors]
    plan_r = fr.Plan(restored, chunk_bytes)
    ids, n = plan_r.unpack_verify(packed, cap=cap)
    status = plan_r.sync_status()
    table_r = plan_r.fingerprint()
    torch.cuda.synchronize()
    out = dict(plan=plan, plan_r=plan_r, table=table, packed=packed, restored=restored, ids=ids, n=n,
               status=status, table_r=table_r)
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
