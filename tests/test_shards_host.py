"""Host logic of ZeRO / FSDP restoration (Sec. III-A, III-E): the library's
fr_shard_pieces against a brute-force map of which shard owns each element,
and the region lists built from it, on CPU tensors (no device work)."""
import itertools

import numpy as np
import pytest
import torch

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")
from paper_2509_03047_gb300 import shards  # noqa: E402


def owners(n, k):
    """Brute force: the shard that owns each element when n elements are cut
    into k shards of ceil(n/k) elements (the last non-empty one shorter)."""
    if n == 0:
        return np.zeros(0, dtype=np.int64)
    q = -(-n // k)
    return np.arange(n) // q


def brute_pieces(n, eb, n_dst, rank, n_src):
    od, os_ = owners(n, n_dst), owners(n, n_src)
    mine = np.nonzero(od == rank)[0]
    out = []
    for e in mine:
        j = int(os_[e])
        src_off = (e - np.nonzero(os_ == j)[0][0]) * eb
        dst_off = (e - mine[0]) * eb
        if out and out[-1][0] == j and out[-1][1] + out[-1][3] == src_off and out[-1][2] + out[-1][3] == dst_off:
            out[-1] = (j, out[-1][1], out[-1][2], out[-1][3] + eb)
        else:
            out.append((j, int(src_off), int(dst_off), eb))
    return out


CASES = [(n, eb, nd, ns) for n in (0, 1, 5, 17, 64, 101) for eb in (2, 4) for nd in (1, 3, 4, 8, 13)
         for ns in (1, 2, 4, 7, 13)]


@pytest.mark.parametrize("n,eb,n_dst,n_src", CASES)
def test_pieces_match_brute_force(n, eb, n_dst, n_src):
    for rank in range(n_dst):
        got = fr.fr_shard_pieces(n, eb, n_dst, rank, n_src)
        assert got == brute_pieces(n, eb, n_dst, rank, n_src)
        a, b = shards.shard_range(n, n_dst, rank)
        assert sum(p[3] for p in got) == (b - a) * eb
        assert len(got) <= n_src


def test_equal_sharding_is_one_piece_from_the_same_rank():
    for rank in range(6):
        assert fr.fr_shard_pieces(1000, 4, 6, rank, 6) == [(rank, 0, 0, shards.shard_range(1000, 6, rank)[1] * 4
                                                            - shards.shard_range(1000, 6, rank)[0] * 4)]


def test_capacity_keeps_the_true_count():
    import ctypes

    n = ctypes.c_uint64(0)
    arr = (fr.fr_piece * 2)()
    st = fr.lib.fr_shard_pieces(1000, 4, 1, 0, 5, arr, 2, ctypes.byref(n))
    assert st == fr.FR_ERR_CAPACITY and n.value == 5
    assert (arr[0].source, arr[1].source) == (0, 1)


@pytest.mark.parametrize("args", [(10, 0, 2, 0, 2), (10, 4, 0, 0, 2), (10, 4, 2, 2, 2), (10, 4, 2, 0, 0),
                                  (2 ** 63, 4, 2, 0, 2)])
def test_invalid_arguments(args):
    with pytest.raises(fr.FlashrecError) as e:
        fr.fr_shard_pieces(*args)
    assert e.value.status == fr.FR_ERR_INVALID_ARG


def _flat_groups(seed=0):
    g = torch.Generator().manual_seed(seed)
    n = 1037
    master = torch.randn(n, generator=g) * 0.02
    return [master.to(torch.bfloat16), master, torch.randn(n, generator=g), torch.randn(n, generator=g)]


@pytest.mark.parametrize("n_dst,n_src", list(itertools.product((1, 3, 4, 8), (1, 2, 5, 8))))
def test_regions_reassemble_the_shard(n_dst, n_src):
    full = _flat_groups()
    n_elems = [t.numel() for t in full]
    srcs = [shards.make_shards(full, n_src, j) for j in range(n_src)]
    for rank in range(n_dst):
        want = shards.make_shards(full, n_dst, rank)
        dst = [torch.empty_like(t) for t in want]
        src_reg, dst_reg = shards.shard_regions(n_elems, dst, n_dst, rank, srcs, n_src)
        assert [r.numel() for r in src_reg] == [r.numel() for r in dst_reg]
        for s, d in zip(src_reg, dst_reg):  # a plain host copy stands in for the device transfer
            d.copy_(s)
        for w, d in zip(want, dst):
            assert torch.equal(w.view(torch.uint8) if w.dtype != torch.bfloat16 else w.view(torch.int16),
                               d.view(torch.uint8) if d.dtype != torch.bfloat16 else d.view(torch.int16))


@pytest.mark.parametrize("n_a,n_b", [(3, 5), (2, 8), (4, 4), (1, 7)])
def test_common_regions_line_up(n_a, n_b):
    full = _flat_groups(1)
    n_elems = [t.numel() for t in full]
    eb = [t.element_size() for t in full]
    a = [shards.make_shards(full, n_a, j) for j in range(n_a)]
    b = [shards.make_shards(full, n_b, j) for j in range(n_b)]
    for rank in range(3):
        ra, rb = shards.common_regions(n_elems, eb, 3, rank, a, n_a, b, n_b)
        assert len(ra) == len(rb)
        assert len(ra) <= sum(len(fr.fr_shard_pieces(n, e, 3, rank, n_a)) + len(fr.fr_shard_pieces(n, e, 3, rank, n_b))
                              for n, e in zip(n_elems, eb))
        for x, y in zip(ra, rb):
            assert x.dtype == y.dtype and torch.equal(x.view(torch.uint8), y.view(torch.uint8))
        # together they cover the shard's bytes of every group, in order
        got = [torch.cat([r.view(torch.uint8) for r in ra if r.dtype == dt])
               for dt in (torch.bfloat16, torch.float32)]
        want = shards.make_shards(full, 3, rank)
        assert torch.equal(got[0], want[0].view(torch.uint8))
        assert torch.equal(got[1], torch.cat([w.view(torch.uint8) for w in want[1:]]))
