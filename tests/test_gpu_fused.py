"""GPU tests of the fused calls: pack, unpack and restore that also write the
fingerprint tables.  Each table must be bit-identical to what fr_fingerprint
writes for the same tensors (itself pinned to the oracle in
test_gpu_parity.py), and every other output identical to the plain call's."""
import numpy as np
import pytest
import torch

from paper_2509_03047_gb300 import synth

from gpu_helpers import assert_tables_match, expected_mismatch, odd_tensors, table_np

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")

import oracle  # noqa: E402

KiB, MiB = 1024, 1024 * 1024


@pytest.fixture(autouse=True)
def _free_memory():
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _fresh(st):
    return [torch.full_like(t.view(torch.uint8), 0x5A).view(t.dtype) for t in st]


def _same(a, b):
    return all(torch.equal(x.view(torch.uint8), y.view(torch.uint8)) for x, y in zip(a, b))


def _chunks(st, chunk):
    return oracle.plan([t.numel() * t.element_size() for t in st], [fr.fr_dtype_of(t) for t in st], chunk)[0]


def _cases():
    """(name, tensors, chunk bytes): NaN-bearing state, special values, odd views."""
    cfg = synth.get_config("tiny")
    tiny = synth.make_state(cfg, "cuda")
    synth.inject_nonfinite(cfg, tiny)
    n = 1 << 15
    special = [torch.full((n,), v, device="cuda") for v in (0.0, 1e-40, 1e-25, 3e19, 3.0e38, 2e17, float("nan"))]
    special += [torch.full((n,), v, device="cuda").to(torch.bfloat16) for v in (1e-40, 3e19, float("-inf"))]
    mixed = torch.randn(n, device="cuda")
    mixed[::997] = float("nan")
    mixed[9::2003] = 2e30
    special.append(mixed)
    base = torch.randn((3 << 20) + 64, device="cuda")
    views = [base[1:1 + 700001], base[800001:800001 + 333333].to(torch.bfloat16).contiguous(),
             base[2000000:2000000 + 1000003], torch.randint(0, 256, (99999,), device="cuda", dtype=torch.uint8)]
    return [("tiny", tiny, cfg.chunk_bytes), ("special", special, 16 * KiB), ("views", views, 12288)]


CASES = ["tiny", "special", "views"]


def _case(name):
    return {c[0]: c for c in _cases()}[name]


@pytest.mark.parametrize("name", CASES)
def test_pack_fp_equals_pack_and_fingerprint(name):
    _, st, chunk = _case(name)
    p = fr.Plan(st, chunk)
    want_table = p.fingerprint()
    want_packed = p.pack()
    got_packed = torch.full_like(want_packed, 0xCC)
    got_table = torch.full_like(want_table, 0xEE)
    fr.fr_pack_fp(p.handle, got_packed, got_table)
    torch.cuda.synchronize()
    assert torch.equal(got_packed, want_packed)
    assert torch.equal(got_table, want_table)


@pytest.mark.parametrize("name", CASES)
def test_unpack_verify_fp_equals_unpack_then_fingerprint(name):
    _, st, chunk = _case(name)
    src = fr.Plan(st, chunk)
    packed = src.pack()
    flips = synth.flip_positions(src.packed_bytes, 9, seed=11)
    synth.apply_flips(packed, flips)
    a_t, b_t = _fresh(st), _fresh(st)
    a, b = fr.Plan(a_t, chunk), fr.Plan(b_t, chunk)
    ids_a, n_a = a.unpack_verify(packed)
    got_table = torch.full((b.n_chunks * 16,), 0xEE, dtype=torch.uint8, device="cuda")
    ids_b = torch.empty(b.n_chunks, dtype=torch.int32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    fr.fr_unpack_verify_fp(b.handle, packed, ids_b, cnt, got_table)
    n_b = int(cnt.item())
    assert n_a == n_b and torch.equal(ids_a, ids_b[:n_b])
    assert np.array_equal(ids_a.cpu().numpy().astype(np.int64), expected_mismatch(_chunks(st, chunk), flips))
    assert _same(a_t, b_t)
    # the table is the fingerprint of what was written, failing chunks included
    assert torch.equal(got_table, b.fingerprint())


@pytest.mark.parametrize("offset,chunk", [(0, 4), (0, 12), (0, 1000), (0, 64 * KiB), (2, 4096), (4, 12288),
                                          (8, 100)])
def test_fused_calls_on_odd_sizes_and_views(offset, chunk):
    """Every piece shape the fused sweeps meet -- sub-block tails, chunks of a
    few bytes, tensors shorter than a lane's unit, misaligned views -- against
    the plain calls and, for the tables, the oracle."""
    st = odd_tensors(5, offset)
    src = fr.Plan(st, chunk)
    want_table, want_packed = src.fingerprint(), src.pack()
    packed = torch.full_like(want_packed, 0xCC)
    ta = torch.full_like(want_table, 0xEE)
    fr.fr_pack_fp(src.handle, packed, ta)
    torch.cuda.synchronize()
    assert torch.equal(packed, want_packed) and torch.equal(ta, want_table)
    chunks = _chunks(st, chunk)
    host = [t.contiguous().view(torch.uint8).cpu().numpy().reshape(-1) for t in st]
    want_fp = oracle.fingerprint(host, [fr.fr_dtype_of(t) for t in st], chunk)
    assert_tables_match(table_np(ta), want_fp, "pack_fp")

    flips = synth.flip_positions(src.packed_bytes, 5, seed=offset + chunk)
    synth.apply_flips(packed, flips)
    dst_t = _fresh(st)
    dst = fr.Plan(dst_t, chunk)
    ids = torch.empty(dst.n_chunks, dtype=torch.int32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    tb = torch.full_like(want_table, 0xDD)
    fr.fr_unpack_verify_fp(dst.handle, packed, ids, cnt, tb)
    n = int(cnt.item())
    assert np.array_equal(ids[:n].cpu().numpy().astype(np.int64), expected_mismatch(chunks, flips))
    assert torch.equal(tb, dst.fingerprint())
    # chunks whose payload took no flip are restored bit-exactly, with equal entries
    d, k = fr.diff(ta, tb)
    assert set(d.cpu().tolist()) <= set(ids[:n].cpu().tolist())


@pytest.mark.parametrize("where,n_batches", [("device", 1), ("device", 7), ("pinned", 5)])
def test_restore_fp_tables(where, n_batches):
    cfg = synth.get_config("gpt2s")
    st = synth.make_state(cfg, "cuda")
    st[1][::7777] = float("nan")
    src = fr.Plan(st, cfg.chunk_bytes, n_batches=n_batches)
    dst_t = _fresh(st)
    dst = fr.Plan(dst_t, cfg.chunk_bytes, n_batches=n_batches)
    staging = src.new_packed(pinned=(where == "pinned"))
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    fa = torch.full((src.n_chunks * 16,), 0xEE, dtype=torch.uint8, device="cuda")
    fb = torch.full_like(fa, 0xDD)
    cnt = torch.full((1,), -1, dtype=torch.int64, device="cuda")
    fr.fr_restore_fp(src.handle, dst.handle, staging, 1, None, cnt, fa, fb, s1, s2)
    s2.synchronize()
    assert int(cnt.item()) == 0
    assert _same(st, dst_t)
    want = src.fingerprint()
    torch.cuda.synchronize()
    assert torch.equal(fa, want) and torch.equal(fb, want)
    d, k = fr.diff(fa, fb)
    assert k == 0
    assert int(table_np(fa)["nonfinite"].sum()) == st[1][::7777].numel()


def test_resend_fp_rewrites_the_resent_entries():
    _, st, chunk = _case("tiny")
    src = fr.Plan(st, chunk)
    dst_t = _fresh(st)
    dst = fr.Plan(dst_t, chunk)
    staging = src.new_packed()
    fa = torch.full((src.n_chunks * 16,), 0xEE, dtype=torch.uint8, device="cuda")
    fr.fr_pack_fp(src.handle, staging, fa)
    flips = synth.flip_positions(src.packed_bytes, 20, seed=4)
    synth.apply_flips(staging, flips)  # damage in transit
    fb = torch.full_like(fa, 0xDD)
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    fr.fr_unpack_verify_fp(dst.handle, staging, None, cnt, fb)
    bad = int(cnt.item())
    assert bad == expected_mismatch(_chunks(st, chunk), flips).size > 0
    # before the re-send the restored table reflects the damaged bytes
    assert torch.equal(fb, dst.fingerprint())
    n = fr.fr_resend_fp(src.handle, dst.handle, staging, fa, fb)
    assert n == bad
    torch.cuda.synchronize()
    assert _same(st, dst_t)
    assert torch.equal(fa, src.fingerprint())
    assert torch.equal(fb, fa)


def test_plan_methods_for_the_fused_calls():
    _, st, chunk = _case("tiny")
    a = fr.Plan(st, chunk)
    packed, ta = a.pack_fp()
    assert torch.equal(ta, a.fingerprint()) and torch.equal(packed, a.pack())
    out = _fresh(st)
    b = fr.Plan(out, chunk)
    ids, n, tb = b.unpack_verify_fp(packed)
    assert n == 0 and torch.equal(ta, tb) and _same(st, out)


@pytest.mark.parametrize("name", ["l70b_tp8pp4", "zero_frag"])
def test_fused_calls_at_full_size(name):
    """The bench's workloads at full size, with its flips: the fused tables
    are bit-identical to fr_fingerprint's (sampled against the oracle in
    test_gpu_parity.py), the failure list to the plain call's."""
    cfg = synth.get_config(name)
    st = synth.make_state(cfg, "cuda")
    synth.inject_nonfinite(cfg, st)
    a = fr.Plan(st, cfg.chunk_bytes)
    packed, ta = a.pack_fp()
    assert torch.equal(ta, a.fingerprint())
    flips = synth.flip_positions(a.packed_bytes, max(cfg.flips, 10), cfg.seed)
    synth.apply_flips(packed, flips)
    out = [torch.empty_like(t) for t in st]
    b = fr.Plan(out, cfg.chunk_bytes)
    ids, n, tb = b.unpack_verify_fp(packed)
    assert np.array_equal(ids.cpu().numpy().astype(np.int64), expected_mismatch(_chunks(st, cfg.chunk_bytes), flips))
    assert torch.equal(tb, b.fingerprint())
    d, k = fr.diff(ta, tb)
    assert k >= 1 and set(d.cpu().numpy().tolist()) <= set(ids.cpu().numpy().tolist())
