"""Pins of the oracle's planner, packed layout, verification and diff.

The expectations here are computed independently of the oracle's C code:
chunk counts and offsets from a plain Python restatement of the layout,
headers parsed with `struct` against the documented field offsets, and the
expected mismatch set from where the injected bit flips landed.
"""
import random
import struct

import numpy as np
import pytest

from paper_2509_03047_gb300 import synth

DT_BYTES, DT_BF16, DT_F32 = 0, 1, 2
HDR = struct.Struct("<IHHQIIQQQdII")  # magic ver dtype id tidx pcrc toff len poff sumsq nonfinite hcrc
assert HDR.size == 64


def a256(v):
    return (v + 255) // 256 * 256


def py_plan(nbytes, chunk):
    """Independent restatement: [(tensor, off, len)], payload offsets, size."""
    chunks = []
    for t, n in enumerate(nbytes):
        off = 0
        while off < n:
            chunks.append((t, off, min(chunk, n - off)))
            off += chunk
    p = a256(64 * len(chunks))
    offs = []
    for _, _, ln in chunks:
        offs.append(p)
        p += a256(ln)
    return chunks, offs, p


def owner_of_byte(b, chunks, offs):
    """Which chunk a byte of the packed buffer belongs to."""
    c = len(chunks)
    if b < 64 * c:
        return b // 64
    if b < a256(64 * c):
        return c - 1  # the gap after the header table belongs to the last chunk
    i = int(np.searchsorted(np.asarray(offs), b, side="right")) - 1
    assert offs[i] <= b < offs[i] + a256(chunks[i][2])
    return i


def adversarial_state(seed=0):
    """Tensors of awkward sizes: empty, < 16 B, = 4 mod 16, exact chunk
    multiples, and NaN/Inf content."""
    rng = np.random.default_rng(seed)
    specs = [(DT_F32, 0), (DT_BF16, 6), (DT_F32, 4), (DT_F32, 20), (DT_BF16, 1000),
             (DT_F32, 4096), (DT_BYTES, 13), (DT_F32, 4100), (DT_BF16, 8192 + 2), (DT_F32, 3 * 1024 + 12)]
    arrs = []
    for dt, n in specs:
        if dt == DT_F32:
            a = rng.standard_normal(n // 4).astype(np.float32)
            if a.size > 3:
                a[1] = np.nan
                a[2] = np.inf
        elif dt == DT_BF16:
            a = (rng.integers(0, 2**16, n // 2, dtype=np.uint32) & 0xBFFF).astype(np.uint16)
        else:
            a = rng.integers(0, 256, n, dtype=np.uint8)
        arrs.append(np.ascontiguousarray(a).view(np.uint8))
    return arrs, [dt for dt, _ in specs]


CHUNK = 1024


def test_plan_matches_independent_restatement(orc):
    arrs, dts = adversarial_state()
    nb = [a.size for a in arrs]
    for chunk in [4, 64, 1000, 1024, 4096, 1 << 20]:
        ch, packed = orc.plan(nb, dts, chunk)
        want, offs, size = py_plan(nb, chunk)
        assert packed == size
        assert [(int(c["tensor_idx"]), int(c["tensor_off"]), int(c["len"])) for c in ch] == want
        assert list(ch["payload_off"]) == offs
        assert all(o % 256 == 0 for o in offs)


def test_config_chunk_counts(orc):
    """Chunk and tail counts of the five workloads (sizes from the model shapes)."""
    expect = {"tiny": (236, 12), "gpt2s": (2121, 517), "l8b_tp8": (3806, 620), "l70b_tp8pp4": (2212, 384)}
    for name, (n, tails) in expect.items():
        cfg = synth.get_config(name)
        specs = cfg.buffer_specs()
        ch, _ = orc.plan([b for _, _, b in specs], [d for _, d, _ in specs], cfg.chunk_bytes)
        assert len(ch) == n
        assert int((ch["len"] < cfg.chunk_bytes).sum()) == tails


def test_plan_rejects_invalid(orc):
    with pytest.raises(ValueError):
        orc.plan([16], [DT_F32], 0)
    with pytest.raises(ValueError):
        orc.plan([16], [DT_F32], 6)
    with pytest.raises(ValueError):
        orc.plan([6], [DT_F32], 16)
    with pytest.raises(ValueError):
        orc.plan([3], [DT_BF16], 16)
    with pytest.raises(ValueError):
        orc.plan([16], [7], 16)


def test_header_layout_and_payloads(orc):
    arrs, dts = adversarial_state()
    buf = orc.pack(arrs, dts, CHUNK)
    chunks, offs, size = py_plan([a.size for a in arrs], CHUNK)
    assert buf.size == size
    for c, (t, off, ln) in enumerate(chunks):
        h = buf[64 * c: 64 * c + 64].tobytes()
        magic, ver, dt, cid, tidx, pcrc, toff, length, poff, sumsq, nf, hcrc = HDR.unpack(h)
        assert h[:4] == b"FRC1" and ver == 1 and dt == dts[t]
        assert (cid, tidx, toff, length, poff) == (c, t, off, ln, offs[c])
        payload = arrs[t][off:off + ln].tobytes()
        assert buf[poff:poff + ln].tobytes() == payload
        assert pcrc == orc.crc32c(payload)
        assert (nf, sumsq) == orc.fp_values(payload, dts[t])
        assert hcrc == orc.crc32c(h[:60])
        assert not buf[poff + ln: poff + a256(ln)].any()
    assert not buf[64 * len(chunks): a256(64 * len(chunks))].any()


def _fresh_dst(arrs):
    return [np.full(a.size, 0xA5, dtype=np.uint8) for a in arrs]


def test_roundtrip_bitwise(orc):
    arrs, dts = adversarial_state(1)
    buf = orc.pack(arrs, dts, CHUNK)
    dst = _fresh_dst(arrs)
    rc, ids, n = orc.unpack_verify(dst, dts, CHUNK, buf)
    assert rc == 0 and n == 0 and ids.size == 0
    for a, b in zip(arrs, dst):
        assert np.array_equal(a, b)


def _flip(buf, bit):
    b = buf.copy()
    b[bit // 8] ^= np.uint8(1 << (bit % 8))
    return b


def test_each_region_flags_its_chunk(orc):
    arrs, dts = adversarial_state(2)
    buf = orc.pack(arrs, dts, CHUNK)
    chunks, offs, _ = py_plan([a.size for a in arrs], CHUNK)
    C = len(chunks)
    probes = []
    for c in [0, 3, C - 1]:
        for field_off in [0, 4, 6, 8, 16, 20, 24, 32, 40, 48, 56, 60, 63]:  # every field, incl. header_crc
            probes.append(((64 * c + field_off) * 8 + 3, c))
        probes.append(((offs[c]) * 8, c))                      # first payload bit
        probes.append(((offs[c] + chunks[c][2] - 1) * 8 + 7, c))  # last payload bit
        if chunks[c][2] % 256:
            probes.append(((offs[c] + chunks[c][2]) * 8 + 1, c))  # padding
    if (64 * C) % 256:
        probes.append((64 * C * 8 + 5, C - 1))                  # gap after the table
    for bit, want in probes:
        dst = _fresh_dst(arrs)
        rc, ids, n = orc.unpack_verify(dst, dts, CHUNK, _flip(buf, bit))
        assert rc == 0 and list(ids) == [want], (bit, want, list(ids))


def test_two_flips_on_one_bit_cancel(orc):
    arrs, dts = adversarial_state(3)
    buf = orc.pack(arrs, dts, CHUNK)
    twice = _flip(_flip(buf, 12345), 12345)
    rc, ids, n = orc.unpack_verify(_fresh_dst(arrs), dts, CHUNK, twice)
    assert n == 0


def test_seeded_flips_give_the_injected_set(orc):
    arrs, dts = adversarial_state(4)
    buf = orc.pack(arrs, dts, CHUNK)
    chunks, offs, size = py_plan([a.size for a in arrs], CHUNK)
    for count in [1, 2, 10, 40]:
        pos = synth.flip_positions(size, count, seed=count)
        bad = buf.copy()
        for p in pos:
            bad[p // 8] ^= np.uint8(1 << (p % 8))
        want = sorted({owner_of_byte(int(p) // 8, chunks, offs) for p in pos})
        dst = _fresh_dst(arrs)
        rc, ids, n = orc.unpack_verify(dst, dts, CHUNK, bad)
        assert list(ids) == want and n == len(want)
        # restored bytes are the packed payload bytes, corrupted ones included
        for c, (t, off, ln) in enumerate(chunks):
            assert np.array_equal(dst[t][off:off + ln], bad[offs[c]:offs[c] + ln])


def test_capacity_overflow_keeps_true_count(orc):
    arrs, dts = adversarial_state(5)
    buf = orc.pack(arrs, dts, CHUNK)
    chunks, offs, _ = py_plan([a.size for a in arrs], CHUNK)
    bad = buf.copy()
    for c in range(len(chunks)):
        bad[offs[c]] ^= 1
    rc, ids, n = orc.unpack_verify(_fresh_dst(arrs), dts, CHUNK, bad, cap=3)
    assert n == len(chunks) and list(ids) == [0, 1, 2]


def test_truncated_buffer_is_rejected(orc):
    arrs, dts = adversarial_state(6)
    buf = orc.pack(arrs, dts, CHUNK)
    rc, ids, n = orc.unpack_verify(_fresh_dst(arrs), dts, CHUNK, buf, src_bytes=buf.size - 1)
    assert rc == orc.ERR_BUFFER_TOO_SMALL


def test_diff_lists_modified_chunks(orc):
    arrs, dts = adversarial_state(7)
    fa = orc.fingerprint(arrs, dts, CHUNK)
    ids, n = orc.diff(fa, fa.copy())
    assert n == 0
    chunks, _, _ = py_plan([a.size for a in arrs], CHUNK)
    rng = random.Random(8)
    pick = sorted(rng.sample(range(len(chunks)), 5))
    mod = [a.copy() for a in arrs]
    for c in pick:
        t, off, ln = chunks[c]
        mod[t][off + rng.randrange(ln)] ^= 0x10
    fb = orc.fingerprint(mod, dts, CHUNK)
    ids, n = orc.diff(fa, fb)
    assert list(ids) == pick and n == len(pick)
    ids, n = orc.diff(fa, fb, cap=2)
    assert list(ids) == pick[:2] and n == len(pick)


def test_diff_compares_sumsq_bits():
    import oracle as orc
    orc.build()
    a = np.zeros(3, dtype=orc.FP_DTYPE)
    b = a.copy()
    b["sumsq"][1] = -0.0  # equal as numbers, different as bits
    ids, n = orc.diff(a, b)
    assert list(ids) == [1]


def test_empty_state(orc):
    buf = orc.pack([], [], CHUNK)
    assert buf.size == 0
    rc, ids, n = orc.unpack_verify([], [], CHUNK, buf)
    assert rc == 0 and n == 0
    z = np.zeros(0, dtype=np.uint8)
    assert orc.pack([z], [DT_F32], CHUNK).size == 0


@pytest.mark.parametrize("field_off,width", [(0, 4), (4, 2), (6, 2), (8, 8), (16, 4), (24, 8), (32, 8), (40, 8)])
def test_wrong_field_under_a_valid_header_crc(orc, field_off, width):
    """A header whose CRC is intact but whose addressing field disagrees with
    the receiver's plan (a replayed or misdirected header) is flagged."""
    arrs, dts = adversarial_state(9)
    buf = orc.pack(arrs, dts, CHUNK)
    c = 3
    h = bytearray(buf[64 * c: 64 * c + 64].tobytes())
    v = int.from_bytes(h[field_off:field_off + width], "little") ^ 1
    h[field_off:field_off + width] = v.to_bytes(width, "little")
    h[60:64] = orc.crc32c(bytes(h[:60])).to_bytes(4, "little")
    bad = buf.copy()
    bad[64 * c: 64 * c + 64] = np.frombuffer(bytes(h), dtype=np.uint8)
    rc, ids, n = orc.unpack_verify(_fresh_dst(arrs), dts, CHUNK, bad)
    assert list(ids) == [c]


def test_swapped_headers_are_flagged(orc):
    arrs, dts = adversarial_state(10)
    buf = orc.pack(arrs, dts, CHUNK)
    bad = buf.copy()
    bad[64 * 2: 64 * 3], bad[64 * 5: 64 * 6] = buf[64 * 5: 64 * 6], buf[64 * 2: 64 * 3]
    rc, ids, n = orc.unpack_verify(_fresh_dst(arrs), dts, CHUNK, bad)
    assert list(ids) == [2, 5]


def test_per_chunk_verdicts_match_where_the_flips_landed(orc):
    """verify_chunk, given each chunk's header, payload + padding and (last
    chunk) the table gap, sliced by the independent layout restatement, flags
    exactly the owners of the flipped bytes -- the whole-buffer call's result
    chunk by chunk, so tests can spread the chunks over host threads."""
    arrs, dts = adversarial_state(7)
    buf = orc.pack(arrs, dts, CHUNK)
    chunks, offs, size = py_plan([a.size for a in arrs], CHUNK)
    ochunks, _ = orc.plan([a.size for a in arrs], dts, CHUNK)
    C = len(chunks)
    gap = (64 * C, a256(64 * C))
    assert gap[1] > gap[0]  # this layout has a gap for the probe below
    cases = [np.zeros(0, dtype=np.int64), np.array([gap[0] * 8 + 2])]
    cases += [synth.flip_positions(size, k, seed=100 + k) for k in (1, 3, 17, 60)]
    for pos in cases:
        bad = buf.copy()
        for p in pos:
            bad[p // 8] ^= np.uint8(1 << (p % 8))
        want = sorted({owner_of_byte(int(p) // 8, chunks, offs) for p in pos})
        got = [c for c in range(C)
               if orc.verify_chunk(ochunks[c], c, bad[64 * c: 64 * c + 64],
                                   bad[offs[c]: offs[c] + a256(chunks[c][2])],
                                   bad[gap[0]: gap[1]] if c == C - 1 else None)]
        assert got == want
        rc, ids, n = orc.unpack_verify(_fresh_dst(arrs), dts, CHUNK, bad)
        assert list(ids) == got
