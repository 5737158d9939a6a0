"""GPU tests of the work units that pack and unpack warps claim at run time.

A pack or unpack launch leaves the last few percent of each class's segments
out of the warps' own ranges and cuts them into units that warps claim
through per-class counters; the last warp to leave zeroes the counters for
the next launch on the plan.  The state here has four classes (bf16, fp32,
an fp32 view that is not 16-byte aligned, bytes), each large enough to have
several units.  Its outputs must equal the oracle's, and stay equal over many
launches queued back to back with no host synchronization between them (a
counter left non-zero would make a later launch skip units: stale payload
bytes and wrong checksums), for the whole-state calls and for the batched
restore, whose batches each have their own counters."""
import numpy as np
import pytest
import torch

from gpu_helpers import compare_full, host_bytes, table_np

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")

KiB, MiB = 1024, 1024 * 1024


@pytest.fixture(autouse=True)
def _free_memory():
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _state():
    g = torch.Generator(device="cuda")
    g.manual_seed(11)
    base = torch.randn((6 << 20) + 8, generator=g, device="cuda")
    return [
        torch.randn(5 << 20, generator=g, device="cuda").to(torch.bfloat16),  # 10 MiB bf16
        torch.randn((3 << 20) + 77, generator=g, device="cuda"),             # 12 MiB fp32, ragged
        base[1:1 + (5 << 20)],                                                # fp32, 4-byte aligned view
        torch.randint(0, 256, ((7 << 20) + 5,), generator=g, device="cuda", dtype=torch.uint8),
        torch.randn(12345, generator=g, device="cuda"),                       # smaller than one chunk
    ]


def test_claimed_units_match_the_oracle():
    compare_full(_state(), 1 * MiB, flips=np.array([8 * 4096 + 3, 8 * (9 << 20) + 1], dtype=np.int64))


def test_many_launches_back_to_back():
    st = _state()
    plan = fr.Plan(st, 1 * MiB)
    ref = plan.pack()
    ref_tab = plan.fingerprint()
    torch.cuda.synchronize()
    n = 12
    packed = [plan.new_packed() for _ in range(n)]
    restored = [[torch.empty_like(t) for t in st] for _ in range(n)]
    plans_r = [fr.Plan(r, 1 * MiB) for r in restored]
    counts = torch.empty(n, dtype=torch.int64, device="cuda")
    tabs = [plan_r.new_table() for plan_r in plans_r]
    for i in range(n):  # no synchronization between the launches
        fr.fr_pack(plan.handle, packed[i])
        fr.fr_unpack_verify_fp(plans_r[i].handle, packed[i], None, counts[i:i + 1], tabs[i])
    torch.cuda.synchronize()
    want = host_bytes(st)
    assert counts.tolist() == [0] * n
    for i in range(n):
        assert torch.equal(packed[i], ref), "launch %d: packed buffer differs" % i
        assert torch.equal(tabs[i], ref_tab), "launch %d: restored table differs" % i
        for j, (g, w) in enumerate(zip(host_bytes(restored[i]), want)):
            assert np.array_equal(g, w), "launch %d: restored tensor %d differs" % (i, j)
    for p in plans_r:
        p.close()
    plan.close()


def test_batched_restore_repeated():
    st = _state()
    src = fr.Plan(st, 1 * MiB, n_batches=3)
    out = [torch.empty_like(t) for t in st]
    dst = fr.Plan(out, 1 * MiB, n_batches=3)
    staging = src.new_packed()
    fa, fb = src.new_table(), dst.new_table()
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    ref_tab = fr.Plan(st, 1 * MiB).fingerprint()
    want = host_bytes(st)
    for k in range(4):
        for t in out:
            t.view(torch.uint8).fill_(0xA5)
        fr.fr_restore_fp(src.handle, dst.handle, staging, 1, None, cnt, fa, fb)
        torch.cuda.synchronize()
        assert int(cnt.item()) == 0, "round %d" % k
        assert torch.equal(fa, ref_tab) and torch.equal(fb, ref_tab), "round %d: tables" % k
        for j, (g, w) in enumerate(zip(host_bytes(out), want)):
            assert np.array_equal(g, w), "round %d: restored tensor %d differs" % (k, j)
    assert table_np(fa).shape[0] == src.n_chunks
    src.close()
    dst.close()
