"""GPU tests of the ordered compaction behind fr_diff and the unpack failure
list, on both of its launch forms: one CTA for up to one tile (8,192 ids) and
a cluster of CTAs, sharing their tile counts through distributed shared
memory, beyond that.  The expected ids come from numpy on the same tables."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")

TILE = 8192


def _tables(n, frac, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    a = torch.randint(0, 256, (n * 16,), generator=g, device="cuda", dtype=torch.uint8)
    b = a.clone()
    hit = torch.rand(n, generator=g, device="cuda") < frac
    idx = torch.nonzero(hit).flatten()
    # flip one seeded byte of each chosen 16-byte entry
    byte = torch.randint(0, 16, (idx.numel(),), generator=g, device="cuda")
    pos = idx * 16 + byte
    b[pos] ^= 0x40
    return a, b, idx.cpu().numpy().astype(np.int64)


@pytest.mark.parametrize("n", [TILE, TILE + 1, 3 * TILE - 7, 8 * TILE, 8 * TILE + 1, 17 * TILE + 123, 132_976])
@pytest.mark.parametrize("frac", [0.003, 0.5])
def test_diff_across_tiles_and_rounds(n, frac):
    a, b, want = _tables(n, frac, seed=n)
    got, k = fr.diff(a, b)
    torch.cuda.synchronize()
    assert k == want.size
    assert np.array_equal(got.cpu().numpy().astype(np.int64), want)


@pytest.mark.parametrize("n", [TILE + 1, 8 * TILE + 5000, 40 * TILE])
def test_diff_beyond_capacity_keeps_the_first_ids_and_the_true_count(n):
    a, b, want = _tables(n, 0.2, seed=7 + n)
    cap = want.size // 3
    out = torch.full((cap,), -1, dtype=torch.int32, device="cuda")
    cnt = torch.empty(1, dtype=torch.int64, device="cuda")
    fr.fr_diff(a, b, n, out, cnt)
    torch.cuda.synchronize()
    assert int(cnt.item()) == want.size
    assert np.array_equal(out.cpu().numpy().astype(np.int64), want[:cap])


def test_diff_of_equal_tables_is_empty_at_every_size():
    for n in (1, TILE, TILE + 1, 9 * TILE + 3):
        a = torch.randint(0, 256, (n * 16,), device="cuda", dtype=torch.uint8)
        got, k = fr.diff(a, a.clone())
        assert k == 0 and got.numel() == 0


def test_unpack_failure_list_over_many_chunks():
    """More chunks than one tile: the verdict compaction takes the cluster
    form; the list is the chunks whose payload took a flip."""
    t = torch.randn(40 * TILE * 64 // 4, device="cuda")  # 40 tiles of 64-byte chunks
    p = fr.Plan([t], 64)
    assert p.n_chunks == 40 * TILE
    packed = p.pack()
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    bad = torch.randperm(p.n_chunks, generator=g, device="cuda")[:777].sort().values
    # payload k sits at a 256-byte-aligned offset after the 64-byte headers
    payload0 = (p.n_chunks * 64 + 255) // 256 * 256
    packed[payload0 + bad * 256 + 3] ^= 0x01
    dst = fr.Plan([torch.empty_like(t)], 64)
    ids, n = dst.unpack_verify(packed)
    torch.cuda.synchronize()
    assert n == 777
    assert torch.equal(ids.to(torch.int64), bad.to(torch.int64))
