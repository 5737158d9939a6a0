"""GPU parity: the CUDA path, called through the C ABI, against the CPU oracle
on the same seeded inputs.

Bar: bit-exact CRC-32C, non-finite counts, packed bytes, mismatch lists and
restored bytes; sums of squares within 1e-9 relative (exactly equal when the
sum is zero).  Small workloads are compared whole; the 14-31 GB workloads are
compared on sampled chunks the oracle computes one by one, plus properties
that hold at any size.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2509_03047_gb300 import synth

from gpu_helpers import (assert_tables_match, compare_full, expected_mismatch, host_bytes, odd_tensors,
                         payload_flip_chunks, run_full, table_np)

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")

KiB, MiB = 1024, 1 << 20


@pytest.fixture(autouse=True)
def _free_memory():
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


# ------------------------------------------------------------------ small, whole

def test_tiny_config_whole_state():
    cfg = synth.get_config("tiny")
    st = synth.make_state(cfg, "cuda")
    pos = synth.inject_nonfinite(cfg, st)
    plan = fr.Plan(st, cfg.chunk_bytes)
    flips = synth.flip_positions(plan.packed_bytes, cfg.flips, cfg.seed)
    plan.close()
    got, want = compare_full(st, cfg.chunk_bytes, flips)
    assert int(table_np(got["table"])["nonfinite"].sum()) == pos.size == 3
    chunks, _ = oracle.plan([t.numel() * t.element_size() for t in st],
                            [fr.fr_dtype_of(t) for t in st], cfg.chunk_bytes)
    assert np.array_equal(np.asarray(want["ids"], dtype=np.int64), expected_mismatch(chunks, flips))


def test_gpt2_small_whole_state_clean_roundtrip():
    cfg = synth.get_config("gpt2s")
    st = synth.make_state(cfg, "cuda")
    got, want = compare_full(st, cfg.chunk_bytes)
    assert got["n"] == 0
    assert torch.equal(got["table"], got["table_r"])
    for a, b in zip(st, got["restored"]):
        assert torch.equal(a.view(torch.uint8), b.view(torch.uint8))


@pytest.mark.parametrize("chunk", [4, 12, 100, 512, 1000, 4096, 64 * KiB, 1 * MiB])
def test_adversarial_sizes_and_chunks(chunk):
    compare_full(odd_tensors(1), chunk)


@pytest.mark.parametrize("dt,esz", [(torch.uint8, 1), (torch.bfloat16, 2), (torch.float32, 4)])
def test_every_tail_length(dt, esz):
    """Chunk tails (len % 512) of every length up to 64 bytes and near 512, on
    bodies of 0, 1 and several blocks, split over several warps: the body's
    CRC is folded into a word-aligned tail, shifted past any other, and
    absent when there is no tail."""
    g = torch.Generator(device="cuda")
    g.manual_seed(17)
    tails = [t for t in list(range(0, 65)) + [500, 508, 510, 511] if t % esz == 0]
    ts = []
    for i, t in enumerate(tails):
        nbytes = 512 * (0, 1, 7)[i % 3] + t
        if dt == torch.uint8:
            ts.append(torch.randint(0, 256, (nbytes,), generator=g, device="cuda", dtype=torch.uint8))
        else:
            ts.append(torch.randn(nbytes // esz, generator=g, device="cuda").to(dt))
    compare_full(ts, 4096)  # one chunk per tensor
    compare_full(ts, 1024)  # several chunks, tails only in the last


@pytest.mark.parametrize("offset", [4, 8, 2])
def test_misaligned_views(offset):
    ts = odd_tensors(2, offset)
    assert any(t.data_ptr() % 16 for t in ts if t.numel())
    compare_full(ts, 4096)
    compare_full(ts, 64 * KiB)


def test_byte_misaligned_views():
    base = torch.randint(0, 256, (3 * MiB + 64,), device="cuda", dtype=torch.uint8)
    ts = [base[1:1 + 1 * MiB + 7], base[1 * MiB + 9: 2 * MiB + 9], base[2 * MiB + 3: 3 * MiB + 3]]
    compare_full(ts, 64 * KiB)


def test_special_values():
    n = 1 << 16
    cases = [
        torch.zeros(n, device="cuda"),
        -torch.zeros(n, device="cuda"),
        torch.full((n,), 1e-40, device="cuda"),             # subnormal fp32
        torch.full((n,), 1e-25, device="cuda"),             # squares underflow fp32
        torch.full((n,), 3e19, device="cuda"),              # squares overflow fp32
        torch.full((n,), 3.0e38, device="cuda"),
        torch.full((n,), 1e17, device="cuda"),              # segment sums near fp32's top, fast path
        torch.full((n,), 2e17, device="cuda"),              # lane sums above 2^120: fp64 tree
        torch.full((n,), float("nan"), device="cuda"),
        torch.full((n,), float("inf"), device="cuda"),
        torch.full((n,), 0.5, device="cuda"),
        torch.full((n,), 1e-40, device="cuda").to(torch.bfloat16),
        torch.full((n,), 3e19, device="cuda").to(torch.bfloat16),
        torch.full((n,), float("-inf"), device="cuda").to(torch.bfloat16),
    ]
    mixed = torch.randn(n, device="cuda")
    mixed[::997] = float("nan")
    mixed[5::1013] = float("inf")
    mixed[7::1511] = 1e-30
    mixed[9::2003] = 2e30
    cases.append(mixed)
    spiky = torch.zeros(n, device="cuda")
    spiky[12345] = 1e-20
    cases.append(spiky)
    got, want = compare_full(cases, 16 * KiB)
    # the same values in tensors with a 148-byte (fp32) / 74-byte (bf16) tail,
    # on both sides of the tail's fp32 range [2^-40, 2^56]
    tails = [torch.full((4096 + 37,), v, device="cuda") for v in
             (1e-12, 8e-13, 3e16, 1e17, 3e19, 1e-25, 1e-40, float("nan"), 0.5)]
    tails += [torch.full((8192 + 37,), v, device="cuda").to(torch.bfloat16) for v in (1e-12, 3e16, 1e17, 3e19)]
    mixed_t = torch.randn(4096 + 37, device="cuda")
    mixed_t[-37::5] = 2e30
    mixed_t[-36::7] = float("inf")
    tails.append(mixed_t)
    compare_full(tails, 16 * KiB)
    t = table_np(got["table"])
    per = (n * 4) // (16 * KiB)
    assert (t["sumsq"][:per] == 0).all()
    assert (t["nonfinite"][8 * per:10 * per] == (16 * KiB) // 4).all()


def test_many_tiny_tensors():
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    sizes = torch.randint(1, 700, (20000,), generator=g, device="cuda").tolist()
    flat = torch.randn(sum(sizes) + 16, generator=g, device="cuda")
    ts, o = [], 0
    for s in sizes:
        ts.append(flat[o:o + s])
        o += s
    compare_full(ts, 1024)


def test_single_chunk_equal_to_tensor_and_one_tensor():
    t = torch.randn(1 << 18, device="cuda")
    got, _ = compare_full([t], t.numel() * 4)
    assert got["plan"].n_chunks == 1
    compare_full([t], 1 << 30)


def test_empty_inputs():
    plan = fr.Plan([], 4096)
    assert plan.n_chunks == 0 and plan.packed_bytes == 0
    table = plan.fingerprint()
    ids, n = plan.unpack_verify(torch.empty(0, dtype=torch.uint8, device="cuda"))
    assert n == 0 and ids.numel() == 0
    ids, n = fr.diff(table, table)
    assert n == 0
    compare_full([torch.empty(0, device="cuda"), torch.empty(0, device="cuda", dtype=torch.bfloat16)], 4096)


# ------------------------------------------------------------------ errors and status

def test_capacity_overflow_and_status():
    cfg = synth.get_config("tiny")
    st = synth.make_state(cfg, "cuda")
    plan = fr.Plan(st, cfg.chunk_bytes)
    packed = plan.pack()
    C = plan.n_chunks
    bits = []
    for c in range(0, C, 7):
        _, _, _, poff = fr.fr_plan_chunk(plan.handle, c)
        bits.append(poff * 8 + 3)
    synth.apply_flips(packed, np.array(bits))
    restored = [torch.empty_like(t) for t in st]
    pr = fr.Plan(restored, cfg.chunk_bytes)
    ids, n = pr.unpack_verify(packed, cap=5)
    assert n == len(bits)
    assert ids.cpu().tolist() == list(range(0, C, 7))[:5]
    assert pr.sync_status() == fr.FR_ERR_CAPACITY
    assert pr.sync_status() == fr.FR_OK
    ids, n = pr.unpack_verify(packed)
    assert n == len(bits) and pr.sync_status() == fr.FR_OK
    ta, tb = plan.fingerprint(), pr.fingerprint()
    d, k = fr.diff(ta, tb, cap=2)
    assert k == len(bits) and d.cpu().tolist() == list(range(0, C, 7))[:2]


def test_argument_errors():
    t = torch.randn(4096, device="cuda")
    with pytest.raises(fr.FlashrecError) as e:
        fr.Plan([t], 6)
    assert e.value.status == fr.FR_ERR_INVALID_ARG
    with pytest.raises(fr.FlashrecError) as e:
        fr.Plan([t], 0)
    plan = fr.Plan([t], 1024)
    short = torch.empty(plan.packed_bytes - 1, dtype=torch.uint8, device="cuda")
    with pytest.raises(fr.FlashrecError) as e:
        plan.pack(short)
    assert e.value.status == fr.FR_ERR_BUFFER_TOO_SMALL
    big = torch.empty(plan.packed_bytes + 32, dtype=torch.uint8, device="cuda")
    with pytest.raises(fr.FlashrecError) as e:
        plan.pack(big[4:])
    assert e.value.status == fr.FR_ERR_ALIGNMENT
    packed = plan.pack()
    with pytest.raises(fr.FlashrecError) as e:
        plan.unpack_verify(packed[: plan.packed_bytes - 16])
    assert e.value.status == fr.FR_ERR_BUFFER_TOO_SMALL


def test_determinism_three_runs():
    cfg = synth.get_config("gpt2s")
    st = synth.make_state(cfg, "cuda")
    st[3][::1001] = float("nan")
    plan = fr.Plan(st, cfg.chunk_bytes)
    tabs = [plan.fingerprint() for _ in range(3)]
    packs = [plan.pack() for _ in range(2)]
    torch.cuda.synchronize()
    assert torch.equal(tabs[0], tabs[1]) and torch.equal(tabs[1], tabs[2])
    assert torch.equal(packs[0], packs[1])


def test_pinned_host_transfer_buffer():
    cfg = synth.get_config("tiny")
    st = synth.make_state(cfg, "cuda")
    plan = fr.Plan(st, cfg.chunk_bytes)
    dev = plan.pack()
    host = plan.new_packed(pinned=True)
    plan.pack(host)
    torch.cuda.synchronize()
    assert torch.equal(dev.cpu(), host)
    restored = [torch.empty_like(t) for t in st]
    pr = fr.Plan(restored, cfg.chunk_bytes)
    ids, n = pr.unpack_verify(host)
    assert n == 0
    for a, b in zip(st, restored):
        assert torch.equal(a.view(torch.uint8), b.view(torch.uint8))


# ------------------------------------------------------------------ full-size workloads

def _sample_chunks(C, k, seed):
    rng = np.random.default_rng(seed)
    picks = set(rng.choice(C, size=min(k, C), replace=False).tolist()) | {0, C - 1}
    return sorted(picks)


def _check_sampled(state, chunk_bytes, table, packed, sample):
    """Per sampled chunk: the oracle's fingerprint of its bytes, its header and
    its payload + padding in the packed buffer."""
    tab = table_np(table)
    nbytes = [t.numel() * t.element_size() for t in state]
    dts = [fr.fr_dtype_of(t) for t in state]
    chunks, packed_bytes = oracle.plan(nbytes, dts, chunk_bytes)
    assert packed.numel() == packed_bytes
    raw = [t.view(torch.uint8) for t in state]
    for c in sample:
        ch = chunks[c]
        t, off, ln, poff = int(ch["tensor_idx"]), int(ch["tensor_off"]), int(ch["len"]), int(ch["payload_off"])
        data = raw[t][off:off + ln].cpu().numpy()
        crc, nf, s = oracle.fingerprint_chunk(data, dts[t])
        got = tab[c]
        assert int(got["crc32c"]) == crc and int(got["nonfinite"]) == nf, c
        assert (s == 0 and got["sumsq"] == 0) or abs(got["sumsq"] - s) <= 1e-9 * abs(s), c
        hdr = packed[64 * c: 64 * c + 64].cpu().numpy().tobytes()
        assert hdr == oracle.header(ch, c, (crc, nf, s if s == got["sumsq"] else float(got["sumsq"]))), c
        assert torch.equal(packed[poff:poff + ln], raw[t][off:off + ln]), c
        pad_end = poff + (ln + 255) // 256 * 256
        assert int(packed[poff + ln:pad_end].count_nonzero()) == 0, c
    return chunks


def _big_config(name, sample_k=48):
    cfg = synth.get_config(name)
    st = synth.make_state(cfg, "cuda")
    pos = synth.inject_nonfinite(cfg, st)
    plan = fr.Plan(st, cfg.chunk_bytes)
    table = plan.fingerprint()
    packed = plan.pack()
    torch.cuda.synchronize()
    sample = _sample_chunks(plan.n_chunks, sample_k, 7)
    chunks = _check_sampled(st, cfg.chunk_bytes, table, packed, sample)
    # any-size properties
    tab = table_np(table)
    assert int(tab["nonfinite"].sum()) == pos.size
    assert int(packed[64 * plan.n_chunks: int(chunks["payload_off"][0])].count_nonzero()) == 0
    return cfg, st, pos, plan, table, packed, chunks


def _restore_with_flips(cfg, st, plan, table, packed, chunks):
    flips = synth.flip_positions(plan.packed_bytes, cfg.flips, cfg.seed)
    synth.apply_flips(packed, flips)
    restored = [torch.empty_like(t) for t in st]
    pr = fr.Plan(restored, cfg.chunk_bytes)
    ids, n = pr.unpack_verify(packed)
    assert pr.sync_status() == fr.FR_OK
    want = expected_mismatch(chunks, flips)
    assert np.array_equal(ids.cpu().numpy().astype(np.int64), want)
    # restored bytes are the packed payload bytes: they differ from the
    # original in exactly the flipped payload bits
    pay = payload_flip_chunks(chunks, flips)
    diffbits = 0
    for a, b in zip(st, restored):
        x = torch.bitwise_xor(a.view(torch.uint8), b.view(torch.uint8))
        diffbits += int(sum(bin(i).count("1") * int(c) for i, c in
                            enumerate(torch.bincount(x.view(-1).to(torch.int64), minlength=256).tolist()) if i))
    b = flips // 8
    starts = chunks["payload_off"].astype(np.int64)
    i = np.clip(np.searchsorted(starts, b, side="right") - 1, 0, None)
    in_payload = (b >= starts[0]) & (b < starts[i] + chunks["len"][i].astype(np.int64))
    assert diffbits == int(in_payload.sum())
    tr = pr.fingerprint()
    d, k = fr.diff(table, tr)
    assert np.array_equal(d.cpu().numpy().astype(np.int64), pay)
    return pr, restored


def test_l8b_tp8_full_size_sampled():
    cfg, st, pos, plan, table, packed, chunks = _big_config("l8b_tp8")
    assert plan.n_chunks == 3806
    _restore_with_flips(cfg, st, plan, table, packed, chunks)


def test_l70b_tp8pp4_full_size_sampled():
    cfg, st, pos, plan, table, packed, chunks = _big_config("l70b_tp8pp4", sample_k=40)
    assert plan.n_chunks == 2212 and pos.size == 50
    _restore_with_flips(cfg, st, plan, table, packed, chunks)


def test_l70b_pinned_host_variant_sampled():
    cfg = synth.get_config("l70b_tp8pp4")
    st = synth.make_state(cfg, "cuda")[:40]  # the first 10 parameter tensors
    plan = fr.Plan(st, cfg.chunk_bytes)
    dev = plan.pack()
    host = plan.new_packed(pinned=True)
    plan.pack(host)
    torch.cuda.synchronize()
    assert torch.equal(dev.cpu(), host)
    restored = [torch.empty_like(t) for t in st]
    pr = fr.Plan(restored, cfg.chunk_bytes)
    ids, n = pr.unpack_verify(host)
    assert n == 0
    assert all(torch.equal(a.view(torch.uint8), b.view(torch.uint8)) for a, b in zip(st, restored))


def test_zero_frag_full_size_sampled_and_diff():
    cfg, st, pos, plan, table, packed, chunks = _big_config("zero_frag", sample_k=64)
    assert plan.n_chunks == len(chunks) and pos.size > 0
    del packed
    torch.cuda.empty_cache()
    rows = [(int(c["tensor_idx"]), int(c["tensor_off"]), int(c["len"]), int(c["dtype"])) for c in chunks]
    mod = [t.clone() for t in st]
    ids = synth.modify_for_diff(cfg, mod, rows)
    pm = fr.Plan(mod, cfg.chunk_bytes)
    tm = pm.fingerprint()
    d, k = fr.diff(table, tm)
    assert k == cfg.diff_chunks == 100
    assert np.array_equal(d.cpu().numpy().astype(np.int64), ids)


def test_chunk_larger_than_4_gib():
    """One fp32 tensor of 6 GiB + 37 elements in 5 GiB chunks: lengths,
    offsets, shift exponents and header fields beyond 32 bits.  Fingerprint
    against the oracle, headers byte-exact against the oracle's (with the
    GPU's sums), and a clean round trip."""
    n = (6 << 30) // 4 + 37
    g = torch.Generator(device="cuda")
    g.manual_seed(17)
    t = torch.randn(n, generator=g, device="cuda")
    t[123456789] = float("nan")
    t[n - 5] = float("inf")
    chunk = 5 << 30
    p = fr.Plan([t], chunk)
    assert p.n_chunks == 2
    table = table_np(p.fingerprint())
    host = host_bytes([t])
    want = oracle.fingerprint(host, [fr.FR_DT_F32], chunk)
    assert_tables_match(table, want, "6 GiB tensor")
    packed = p.pack()
    chunks, _ = oracle.plan([host[0].size], [fr.FR_DT_F32], chunk)
    head = packed[: 2 * 64].cpu().numpy()
    for c in range(2):
        fp = (int(want["crc32c"][c]), int(want["nonfinite"][c]), float(table["sumsq"][c]))
        assert np.array_equal(head[64 * c: 64 * c + 64], np.frombuffer(oracle.header(chunks[c], c, fp), dtype=np.uint8))
    del host
    out = torch.empty_like(t)
    q = fr.Plan([out], chunk)
    ids, k = q.unpack_verify(packed)
    assert k == 0
    assert torch.equal(out.view(torch.int32), t.view(torch.int32))
