"""GPU tests of the streamed restore: batched plans, batch-level pack/unpack,
re-sending failed chunks, and the pipelined fr_restore over a device or a
pinned-host transfer buffer.  Everything is compared with the whole-state
calls (themselves pinned to the oracle in test_gpu_parity.py) and with the
original tensors."""
import numpy as np
import pytest
import torch

import oracle
from paper_2509_03047_gb300 import synth

from gpu_helpers import expected_mismatch, odd_tensors, table_np

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")


@pytest.fixture(autouse=True)
def _free_memory():
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _state(name="gpt2s", nan=True):
    cfg = synth.get_config(name)
    st = synth.make_state(cfg, "cuda")
    if nan:
        st[1][::7777] = float("nan")
    return cfg, st


def _fresh(st):
    return [torch.full_like(t.view(torch.uint8), 0x5A).view(t.dtype) for t in st]


def _same(a, b):
    return all(torch.equal(x.view(torch.uint8), y.view(torch.uint8)) for x, y in zip(a, b))


def _chunks(st, chunk):
    return oracle.plan([t.numel() * t.element_size() for t in st], [fr.fr_dtype_of(t) for t in st], chunk)[0]


@pytest.mark.parametrize("n_batches", [2, 7, 64])
def test_batches_cover_the_chunks_in_order(n_batches):
    cfg, st = _state("tiny", nan=False)
    p = fr.Plan(st, cfg.chunk_bytes, n_batches=n_batches)
    nb = p.n_batches
    assert nb == min(n_batches, p.n_chunks)
    nxt, sizes = 0, []
    for b in range(nb):
        _, first, n = fr.fr_plan_batch(p.handle, b)
        assert first == nxt and n >= 1
        nxt += n
        sizes.append(sum(fr.fr_plan_chunk(p.handle, c)[2] for c in range(first, first + n)))
    assert nxt == p.n_chunks
    if nb == 2:  # about equal bytes
        assert max(sizes) < 0.7 * sum(sizes)


def test_batch_pack_equals_whole_pack_and_fingerprint_unchanged():
    cfg, st = _state()
    whole = fr.Plan(st, cfg.chunk_bytes)
    batched = fr.Plan(st, cfg.chunk_bytes, n_batches=9)
    a = whole.pack()
    b = torch.full_like(a, 0xCC)
    for i in range(batched.n_batches):
        fr.fr_pack_batch(batched.handle, i, b)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    assert torch.equal(whole.fingerprint(), batched.fingerprint())
    c = batched.pack()
    assert torch.equal(a, c)


def test_batch_unpack_equals_whole_unpack_with_faults():
    cfg, st = _state()
    src = fr.Plan(st, cfg.chunk_bytes)
    packed = src.pack()
    flips = synth.flip_positions(src.packed_bytes, 25, seed=3)
    synth.apply_flips(packed, flips)
    r1, r2 = _fresh(st), _fresh(st)
    p1 = fr.Plan(r1, cfg.chunk_bytes)
    p2 = fr.Plan(r2, cfg.chunk_bytes, n_batches=5)
    ids1, n1 = p1.unpack_verify(packed)
    for i in range(p2.n_batches):
        fr.fr_unpack_verify_batch(p2.handle, i, packed)
    out = torch.empty(p2.n_chunks, dtype=torch.int32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    fr.fr_unpack_collect(p2.handle, out, cnt)
    n2 = int(cnt.item())
    assert n1 == n2 and torch.equal(ids1, out[:n2])
    assert np.array_equal(ids1.cpu().numpy().astype(np.int64), expected_mismatch(_chunks(st, cfg.chunk_bytes), flips))
    assert _same(r1, r2)


def test_resend_repairs_transit_corruption():
    cfg, st = _state()
    src = fr.Plan(st, cfg.chunk_bytes, n_batches=6)
    dst_t = _fresh(st)
    dst = fr.Plan(dst_t, cfg.chunk_bytes, n_batches=6)
    staging = src.new_packed()
    for i in range(src.n_batches):
        fr.fr_pack_batch(src.handle, i, staging)
    flips = synth.flip_positions(src.packed_bytes, 40, seed=9)
    synth.apply_flips(staging, flips)  # damage in transit
    for i in range(dst.n_batches):
        fr.fr_unpack_verify_batch(dst.handle, i, staging)
    out = torch.empty(dst.n_chunks, dtype=torch.int32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    fr.fr_unpack_collect(dst.handle, out, cnt)
    bad = int(cnt.item())
    want = expected_mismatch(_chunks(st, cfg.chunk_bytes), flips)
    assert bad == want.size > 0
    n = fr.fr_resend(src.handle, dst.handle, staging)
    assert n == bad
    fr.fr_unpack_collect(dst.handle, out, cnt)
    assert int(cnt.item()) == 0
    torch.cuda.synchronize()
    assert _same(st, dst_t)
    assert fr.fr_resend(src.handle, dst.handle, staging) == 0


@pytest.mark.parametrize("where,n_batches", [("device", 1), ("device", 8), ("pinned", 8), ("pinned", 31)])
def test_restore_pipelined(where, n_batches):
    cfg, st = _state()
    src = fr.Plan(st, cfg.chunk_bytes, n_batches=n_batches)
    dst_t = _fresh(st)
    dst = fr.Plan(dst_t, cfg.chunk_bytes, n_batches=n_batches)
    staging = src.new_packed(pinned=(where == "pinned"))
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    out = torch.empty(dst.n_chunks, dtype=torch.int32, device="cuda")
    cnt = torch.full((1,), -1, dtype=torch.int64, device="cuda")
    fr.fr_restore(src.handle, dst.handle, staging, 2, out, cnt, s1, s2)
    s2.synchronize()
    assert int(cnt.item()) == 0
    assert _same(st, dst_t)
    # the transfer buffer holds exactly what fr_pack writes
    ref = src.pack()
    torch.cuda.synchronize()
    assert torch.equal(ref.cpu() if where == "pinned" else ref, staging)
    assert torch.equal(src.fingerprint(), dst.fingerprint())


@pytest.mark.parametrize("offset,chunk,n_batches", [(2, 4096, 5), (4, 12288, 3), (0, 1000, 9)])
def test_restore_every_class_in_batches(offset, chunk, n_batches):
    """Batches that hold chunks of every (element type, alignment) class --
    byte, bf16 and fp32 tensors, some views misaligned -- go through the
    pipelined restore with its re-sends, both fingerprint tables included."""
    st = odd_tensors(9, offset)
    src = fr.Plan(st, chunk, n_batches=n_batches)
    dst_t = _fresh(st)
    dst = fr.Plan(dst_t, chunk, n_batches=n_batches)
    staging = src.new_packed()
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


def test_restore_of_tensors_without_a_body():
    """Every tensor shorter than one 512-byte block: batches with no sweep
    work at all, only tails."""
    g = torch.Generator(device="cuda")
    g.manual_seed(3)
    st = [torch.randn(int(n), generator=g, device="cuda") for n in (1, 5, 64, 127, 100, 3, 90)]
    st += [torch.randint(0, 256, (int(n),), generator=g, device="cuda", dtype=torch.uint8) for n in (7, 511, 300)]
    src = fr.Plan(st, 64, n_batches=4)
    dst_t = _fresh(st)
    dst = fr.Plan(dst_t, 64, n_batches=4)
    staging = src.new_packed()
    cnt = torch.full((1,), -1, dtype=torch.int64, device="cuda")
    fr.fr_restore(src.handle, dst.handle, staging, 1, None, cnt)
    torch.cuda.synchronize()
    assert int(cnt.item()) == 0
    assert _same(st, dst_t)
    assert torch.equal(src.fingerprint(), dst.fingerprint())


def test_restore_rejects_a_different_layout():
    cfg, st = _state("tiny", nan=False)
    src = fr.Plan(st, cfg.chunk_bytes, n_batches=4)
    other = fr.Plan(_fresh(st)[:-1], cfg.chunk_bytes, n_batches=4)
    staging = src.new_packed()
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    with pytest.raises(fr.FlashrecError) as e:
        fr.fr_restore(src.handle, other.handle, staging, 0, None, cnt)
    assert e.value.status == fr.FR_ERR_PLAN_MISMATCH
    with pytest.raises(fr.FlashrecError) as e:
        fr.fr_resend(src.handle, fr.Plan(_fresh(st), cfg.chunk_bytes, n_batches=3).handle, staging)
    assert e.value.status == fr.FR_ERR_PLAN_MISMATCH


def test_restore_full_size_pinned_host():
    """The 31.8 GB Llama-70B shard through pinned host memory, 16 batches."""
    cfg = synth.get_config("l70b_tp8pp4")
    st = synth.make_state(cfg, "cuda")
    synth.inject_nonfinite(cfg, st)
    src = fr.Plan(st, cfg.chunk_bytes, n_batches=16)
    dst_t = [torch.empty_like(t) for t in st]
    dst = fr.Plan(dst_t, cfg.chunk_bytes, n_batches=16)
    staging = src.new_packed(pinned=True)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    cnt = torch.full((1,), -1, dtype=torch.int64, device="cuda")
    fr.fr_restore(src.handle, dst.handle, staging, 1, None, cnt, s1, s2)
    s2.synchronize()
    assert int(cnt.item()) == 0
    ta, tb = src.fingerprint(), dst.fingerprint()
    d, k = fr.diff(ta, tb)
    assert k == 0
    assert int(table_np(ta)["nonfinite"].sum()) == cfg.nan_count
