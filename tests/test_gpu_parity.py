"""GPU parity: the CUDA path, called through the C ABI, against the CPU oracle
on the same seeded inputs.

Bar: bit-exact CRC-32C, non-finite counts, packed bytes, mismatch lists and
restored bytes; sums of squares within 1e-9 relative (exactly equal when the
sum is zero).  Every workload is compared whole: the small ones through the
oracle's whole-state calls, the 14-31 GB ones chunk by chunk with the oracle's
per-chunk calls spread over the host's cores (tests/whole_state.py).  Every
output buffer is followed by a guard region that must stay untouched.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2509_03047_gb300 import synth

from gpu_helpers import (Guarded, assert_tables_match, compare_full, expected_mismatch, fr_diff_guarded,
                         guarded_outputs, host_bytes, odd_tensors, payload_flip_chunks, table_np)
from whole_state import WholeState

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
    _, g_ids, g_cnt = guarded_outputs(C, cap=5)
    ids, n = pr.unpack_verify(packed, mismatch=g_ids.view(torch.int32), count=g_cnt.view(torch.int64))
    g_ids.check("mismatch list beyond cap")
    g_cnt.check("mismatch count")
    assert n == len(bits)
    assert ids.cpu().tolist() == list(range(0, C, 7))[:5]
    assert pr.sync_status() == fr.FR_ERR_CAPACITY
    assert pr.sync_status() == fr.FR_OK
    ids, n = pr.unpack_verify(packed)
    assert n == len(bits) and pr.sync_status() == fr.FR_OK
    ta, tb = plan.fingerprint(), pr.fingerprint()
    for cap in (0, 1, 2):
        d, k = fr_diff_guarded(ta, tb, C, cap=cap)
        assert k == len(bits) and d.cpu().tolist() == list(range(0, C, 7))[:cap]


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

def _whole_config(name):
    """A full-size workload through the C ABI, every chunk compared with the
    oracle (tests/whole_state.py): fingerprint table, packed headers, payloads
    and padding; then the config's bit flips, unpack_verify into fresh
    tensors, and the mismatch list, restored bytes, restored table and diff.
    Every output buffer has a guard region checked after its call."""
    cfg = synth.get_config(name)
    st = synth.make_state(cfg, "cuda")
    pos = synth.inject_nonfinite(cfg, st)
    plan = fr.Plan(st, cfg.chunk_bytes)
    C, P = plan.n_chunks, plan.packed_bytes
    g_tab, g_pack = Guarded(16 * C), Guarded(P)
    table = plan.fingerprint(out=g_tab.buf)
    packed = plan.pack(g_pack.buf)
    torch.cuda.synchronize()
    g_tab.check("fingerprint table")
    g_pack.check("packed buffer")
    ws = WholeState(st, [fr.fr_dtype_of(t) for t in st], cfg.chunk_bytes)
    assert ws.C == C and ws.packed_bytes == P
    tab = table_np(table)
    fails = ws.check_pack(tab, packed)
    assert not fails, "%d chunk checks failed, first %s" % (len(fails), fails[:5])
    assert int(tab["nonfinite"].sum()) == pos.size

    flips = synth.flip_positions(P, cfg.flips, cfg.seed)
    synth.apply_flips(packed, flips)
    restored = [torch.empty_like(t) for t in st]
    pr = fr.Plan(restored, cfg.chunk_bytes)
    g_tab_r, g_ids, g_cnt = guarded_outputs(C)
    ids, n = pr.unpack_verify(packed, mismatch=g_ids.view(torch.int32), count=g_cnt.view(torch.int64))
    assert pr.sync_status() == fr.FR_OK
    table_r = pr.fingerprint(out=g_tab_r.buf)
    torch.cuda.synchronize()
    for g, what in ((g_ids, "mismatch list"), (g_cnt, "mismatch count"), (g_tab_r, "restored table")):
        g.check(what)
    fails, want_ids = ws.check_restore(packed, restored, table_np(table_r))
    assert not fails, "%d restore checks failed, first %s" % (len(fails), fails[:5])
    got_ids = ids.cpu().numpy().astype(np.uint32)
    assert n == want_ids.size and np.array_equal(got_ids, want_ids)
    # and where the flips landed, from the documented layout alone
    assert np.array_equal(got_ids.astype(np.int64), expected_mismatch(ws.chunks, flips))
    div, nd = fr_diff_guarded(table, table_r, C)
    want_div, want_nd = ws.oracle_diff()
    assert nd == want_nd and np.array_equal(div.cpu().numpy().astype(np.uint32), want_div)
    assert np.array_equal(want_div.astype(np.int64), payload_flip_chunks(ws.chunks, flips))
    print("%s: %d chunks, oracle passes %.1f s + %.1f s on %d threads, %d mismatching, %d diverged" % (
        name, C, ws.seconds["pack_pass"], ws.seconds["restore_pass"], ws.threads, n, nd))
    return cfg, st, plan, table, ws


def test_l8b_tp8_whole_state():
    cfg, st, plan, table, ws = _whole_config("l8b_tp8")
    assert plan.n_chunks == 3806


def test_l70b_tp8pp4_whole_state():
    cfg, st, plan, table, ws = _whole_config("l70b_tp8pp4")
    assert plan.n_chunks == 2212


def test_l70b_pinned_host_variant():
    """The first 10 parameter tensors of the 70B shard packed into pinned host
    memory: the same bytes as the device pack (itself checked against the
    oracle above), guard intact, and a clean restore from the host buffer."""
    cfg = synth.get_config("l70b_tp8pp4")
    st = synth.make_state(cfg, "cuda")[:40]
    plan = fr.Plan(st, cfg.chunk_bytes)
    dev = plan.pack()
    host = Guarded(plan.packed_bytes, pinned=True)
    plan.pack(host.buf)
    torch.cuda.synchronize()
    host.check("pinned packed buffer")
    assert torch.equal(dev.cpu(), host.buf)
    restored = [torch.empty_like(t) for t in st]
    pr = fr.Plan(restored, cfg.chunk_bytes)
    ids, n = pr.unpack_verify(host.buf)
    assert n == 0
    assert all(torch.equal(a.view(torch.uint8), b.view(torch.uint8)) for a, b in zip(st, restored))


def test_zero_frag_whole_state_and_diff():
    cfg, st, plan, table, ws = _whole_config("zero_frag")
    assert ws.C == 132976
    rows = [(int(c["tensor_idx"]), int(c["tensor_off"]), int(c["len"]), int(c["dtype"])) for c in ws.chunks]
    mod = [t.clone() for t in st]
    ids = synth.modify_for_diff(cfg, mod, rows)
    pm = fr.Plan(mod, cfg.chunk_bytes)
    tm = pm.fingerprint()
    d, k = fr_diff_guarded(table, tm, plan.n_chunks)
    assert k == cfg.diff_chunks == 100
    assert np.array_equal(d.cpu().numpy().astype(np.int64), ids)
    # the oracle on the modified chunks: exactly these entries change
    want_m = ws.table.copy()
    raw = [t.view(torch.uint8) for t in mod]
    for c in ids.tolist():
        ch = ws.chunks[c]
        t, off, ln = int(ch["tensor_idx"]), int(ch["tensor_off"]), int(ch["len"])
        want_m[c] = oracle.fingerprint_chunk(raw[t][off:off + ln].cpu().numpy(), int(ch["dtype"]))
    assert_tables_match(table_np(tm)[ids], want_m[ids], "modified chunks")
    od, on = oracle.diff(ws.table, want_m)
    assert on == 100 and np.array_equal(od.astype(np.int64), ids)


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
