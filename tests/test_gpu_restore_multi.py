"""Restoration from several replicas at once (the partitioned form of the
restore): batch b is packed by replica b % R.  Checked byte for byte, by the
restored state's fingerprint table, and by making one replica differ in one
of its batches so the result shows which replica sent what."""
import pytest
import torch

from paper_2509_03047_gb300 import synth

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")


@pytest.fixture(autouse=True)
def _free_memory():
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _same(a, b):
    return all(torch.equal(x.view(torch.uint8), y.view(torch.uint8)) for x, y in zip(a, b))


@pytest.mark.parametrize("n_src,n_batches,where", [(1, 4, "device"), (3, 7, "device"), (4, 4, "pinned"),
                                                   (5, 3, "device")])
def test_restore_from_several_replicas(n_src, n_batches, where):
    cfg = synth.get_config("tiny")
    base = synth.make_state(cfg, "cuda")
    synth.inject_nonfinite(cfg, base)
    reps = [[t.clone() for t in base] for _ in range(n_src)]
    src = [fr.Plan(r, cfg.chunk_bytes, n_batches=n_batches) for r in reps]
    out = [torch.full_like(t.view(torch.uint8), 0x5A).view(t.dtype) for t in base]
    dst = fr.Plan(out, cfg.chunk_bytes, n_batches=n_batches)
    staging = src[0].new_packed(pinned=(where == "pinned"))
    streams = [torch.cuda.Stream() for _ in range(n_src)]
    s_dst = torch.cuda.Stream()
    fb = dst.new_table()
    cnt = torch.full((1,), -1, dtype=torch.int64, device="cuda")
    fr.fr_restore_multi([p.handle for p in src], dst.handle, staging, 1, None, cnt, fb, streams, s_dst)
    s_dst.synchronize()
    assert int(cnt.item()) == 0
    assert _same(base, out)
    assert torch.equal(fb, src[0].fingerprint())


def test_each_replica_sends_its_own_batches():
    cfg = synth.get_config("tiny")
    base = synth.make_state(cfg, "cuda")
    reps = [[t.clone() for t in base] for _ in range(3)]
    src = [fr.Plan(r, cfg.chunk_bytes, n_batches=6) for r in reps]
    _, first, n = fr.fr_plan_batch(src[0].handle, 4)  # batch 4 comes from replica 4 % 3 = 1
    t_idx, t_off, length, _ = fr.fr_plan_chunk(src[0].handle, first)
    reps[1][t_idx].view(torch.uint8)[t_off] ^= 1  # replica 1 differs there (a consistent state of its own)
    reps[2][t_idx].view(torch.uint8)[t_off] ^= 2  # replica 2 differs too, but does not send batch 4
    out = [torch.empty_like(t) for t in base]
    dst = fr.Plan(out, cfg.chunk_bytes, n_batches=6)
    staging = src[0].new_packed()
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    fr.fr_restore_multi([p.handle for p in src], dst.handle, staging, 0, None, cnt)
    torch.cuda.synchronize()
    assert int(cnt.item()) == 0
    assert _same(reps[1], out)
    ta, tb = src[0].fingerprint(), dst.fingerprint()
    ids, k = fr.diff(ta, tb)
    assert k == 1 and int(ids[0]) == first


def test_restore_multi_rejects_bad_arguments():
    cfg = synth.get_config("tiny")
    base = synth.make_state(cfg, "cuda")
    a = fr.Plan(base, cfg.chunk_bytes, n_batches=4)
    b = fr.Plan([torch.empty_like(t) for t in base], cfg.chunk_bytes, n_batches=3)
    staging = a.new_packed()
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    with pytest.raises(fr.FlashrecError) as e:
        fr.fr_restore_multi([a.handle], b.handle, staging, 0, None, cnt)
    assert e.value.status == fr.FR_ERR_PLAN_MISMATCH
    with pytest.raises(fr.FlashrecError) as e:
        fr.fr_restore_multi([], a.handle, staging, 0, None, cnt)
    assert e.value.status == fr.FR_ERR_INVALID_ARG
