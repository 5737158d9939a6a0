"""GPU tests of ZeRO / FSDP restoration (Sec. III-A, III-E): a restarted
rank's shard assembled from differently sharded replicas with one pipelined
fr_restore, checked byte for byte against the flat state and by fingerprint
diff; and the cross-replica consistency check finding exactly the chunk a
corrupted replica disagrees in."""
import pytest
import torch

from paper_2509_03047_gb300 import shards

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")


@pytest.fixture(autouse=True)
def _free_memory():
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def flat_state(n=3_000_017, seed=0):
    """Flat groups of a ZeRO optimizer: bf16 parameters, fp32 master, Adam m, v."""
    g = torch.Generator(device="cuda").manual_seed(seed)
    master = torch.randn(n, generator=g, device="cuda") * 0.02
    weight = master.to(torch.bfloat16)
    master = weight.float()
    m = torch.randn(n, generator=g, device="cuda") * 1e-3
    v = (torch.randn(n, generator=g, device="cuda") * 1e-3) ** 2
    return [weight, master, m, v]


def _bytes_equal(a, b):
    return torch.equal(a.view(torch.uint8), b.view(torch.uint8))


@pytest.mark.parametrize("n_dst,rank,n_src", [(4, 1, 3), (4, 3, 7), (4, 0, 1), (4, 2, 4), (8, 7, 3), (3, 2, 8),
                                              (2, 1, 5)])
def test_restore_shard_from_other_sharding(n_dst, rank, n_src):
    full = flat_state()
    n_elems = [t.numel() for t in full]
    sources = [shards.make_shards(full, n_src, j) for j in range(n_src)]
    want = shards.make_shards(full, n_dst, rank)
    dst = [torch.full_like(w.view(torch.uint8), 0x5A).view(w.dtype) for w in want]
    left, diverged, (ps, pd) = shards.restore_shard(n_elems, dst, n_dst, rank, sources, n_src,
                                                    chunk_bytes=256 * 1024, n_batches=5)
    assert left == 0 and diverged.numel() == 0
    for w, d in zip(want, dst):
        assert _bytes_equal(w, d)
    assert ps.n_chunks == pd.n_chunks and ps.state_bytes == sum(w.numel() * w.element_size() for w in want)


def test_restore_shard_through_pinned_host():
    full = flat_state(1_000_003, seed=2)
    n_elems = [t.numel() for t in full]
    sources = [shards.make_shards(full, 5, j) for j in range(5)]
    want = shards.make_shards(full, 2, 0)
    dst = [torch.empty_like(w) for w in want]
    src_reg, _ = shards.shard_regions(n_elems, dst, 2, 0, sources, 5)
    staging = fr.Plan(src_reg, 64 * 1024, n_batches=7).new_packed(pinned=True)
    left, diverged, _ = shards.restore_shard(n_elems, dst, 2, 0, sources, 5, chunk_bytes=64 * 1024, n_batches=7,
                                             staging=staging)
    assert left == 0 and diverged.numel() == 0
    assert all(_bytes_equal(w, d) for w, d in zip(want, dst))


def test_empty_shard_needs_nothing():
    full = [t[:5] for t in flat_state(16)]
    n_elems = [t.numel() for t in full]
    sources = [shards.make_shards(full, 2, j) for j in range(2)]
    dst = shards.make_shards(full, 8, 7)  # 5 elements over 8 shards: shard 7 is empty
    assert all(t.numel() == 0 for t in dst)
    left, diverged, plans = shards.restore_shard(n_elems, dst, 8, 7, sources, 2, chunk_bytes=4096)
    assert left == 0 and plans is None


@pytest.mark.parametrize("n_a,n_b", [(3, 5), (2, 8), (4, 4)])
def test_cross_check_finds_the_corrupted_replica_chunk(n_a, n_b):
    full = flat_state(2_000_003, seed=1)
    n_elems = [t.numel() for t in full]
    eb = [t.element_size() for t in full]
    a = [shards.make_shards(full, n_a, j) for j in range(n_a)]
    b = [shards.make_shards(full, n_b, j) for j in range(n_b)]
    cb = 128 * 1024
    ids, _ = shards.cross_check(n_elems, eb, 4, 1, a, n_a, b, n_b, cb)
    assert ids.numel() == 0
    # change one element of group 2 (Adam m) inside shard 1 of 4 in replica group A
    lo, hi = shards.shard_range(n_elems[2], 4, 1)
    e = lo + (hi - lo) * 2 // 3
    j = e // -(-n_elems[2] // n_a)
    off = e - shards.shard_range(n_elems[2], n_a, j)[0]
    a[j][2][off] += 1.0
    ids, regions = shards.cross_check(n_elems, eb, 4, 1, a, n_a, b, n_b, cb)
    assert ids.numel() == 1
    # the one listed chunk is the one holding the changed element
    plan = fr.Plan(regions, cb)
    t_idx, t_off, length = fr.fr_plan_chunk(plan.handle, int(ids[0]))[:3]
    r = regions[t_idx]
    addr = a[j][2].data_ptr() + off * 4
    assert r.data_ptr() + t_off <= addr < r.data_ptr() + t_off + length
