"""Restoring a ZeRO / FSDP shard from differently sharded replicas.

ZeRO / FSDP flatten the model states into flat groups (one per element type:
bf16 parameters, fp32 master weights, Adam m, Adam v) and give every
data-parallel rank one shard of each group (Sec. III-A).  The paper restores
a restarted rank's states from data-parallel replicas for vanilla DP and for
ZeRO / FSDP alike (Sec. III-E, "Model states Restoration", and the ZeRO/FSDP
panel of its restoration figure).  When the surviving copies are sharded
another way -- another data-parallel degree, another ZeRO group -- the shard
is assembled from pieces of several peers' shards.

The library's fr_shard_pieces gives those pieces for one flat group.  This
module turns them into two tensor lists of identical layout: regions inside
the source shards and the matching regions of the restarted rank's shard.
One plan over each list then drives one pipelined fr_restore for the whole
shard, from all sources at once, and the fingerprints of the two plans,
compared with fr_diff, confirm the result.  `cross_check` compares two
differently sharded replica groups chunk by chunk over the same shard.

Host-side composition only: every byte is moved, checksummed and compared by
the library's kernels.  On one GPU the "peers" are buffers on that GPU (or in
pinned host memory); across GPUs each source would pack its own pieces.
"""
from __future__ import annotations

from typing import List, Optional, Sequence, Tuple

import torch

from . import flashrec as fr


def shard_range(n_elems: int, n_shards: int, rank: int) -> Tuple[int, int]:
    """Element range of shard `rank` under the library's sharding rule
    (ceil-sized shards, the last non-empty one holding the rest)."""
    q = -(-n_elems // n_shards)
    a = min(rank * q, n_elems)
    return a, min(a + q, n_elems)


def make_shards(flat_groups: Sequence[torch.Tensor], n_shards: int, rank: int) -> List[torch.Tensor]:
    """Rank `rank`'s shard (a copy) of each flat group."""
    out = []
    for g in flat_groups:
        a, b = shard_range(g.numel(), n_shards, rank)
        out.append(g[a:b].clone())
    return out


def _elem(t: torch.Tensor) -> int:
    return t.element_size()


def shard_regions(n_elems: Sequence[int], dst: Sequence[torch.Tensor], n_dst: int, rank: int,
                  sources: Sequence[Sequence[torch.Tensor]], n_src: int):
    """(source regions, destination regions): matching 1-D views, one per
    piece, over every flat group in order.  `dst[g]` is the restarted rank's
    shard of group g; `sources[j][g]` is source shard j of group g (entries of
    sources that no piece needs may be None)."""
    src_reg, dst_reg = [], []
    for g, n in enumerate(n_elems):
        eb = _elem(dst[g])
        a, b = shard_range(n, n_dst, rank)
        if dst[g].numel() != b - a:
            raise ValueError("destination shard %d holds %d elements, the rule gives %d" % (g, dst[g].numel(), b - a))
        for j, so, do, nb in fr.fr_shard_pieces(n, eb, n_dst, rank, n_src):
            s = sources[j][g]
            if s is None or s.dtype != dst[g].dtype:
                raise ValueError("source shard %d of group %d is missing or of another type" % (j, g))
            sa, sb = shard_range(n, n_src, j)
            if s.numel() != sb - sa:
                raise ValueError("source shard %d of group %d has the wrong size" % (j, g))
            src_reg.append(s[so // eb:(so + nb) // eb])
            dst_reg.append(dst[g][do // eb:(do + nb) // eb])
    return src_reg, dst_reg


def restore_shard(n_elems: Sequence[int], dst: Sequence[torch.Tensor], n_dst: int, rank: int,
                  sources: Sequence[Sequence[torch.Tensor]], n_src: int, chunk_bytes: int,
                  n_batches: int = 8, max_retries: int = 2, staging: Optional[torch.Tensor] = None,
                  stream_src=None, stream_dst=None, verify: bool = True):
    """Assemble the restarted rank's shard from `n_src` differently sharded
    sources with one pipelined fr_restore; with `verify`, fingerprint both
    sides and return the chunks whose fingerprints differ (empty when every
    byte arrived).  Returns (n_still_failing, diverged_ids, plans)."""
    src_reg, dst_reg = shard_regions(n_elems, dst, n_dst, rank, sources, n_src)
    if not dst_reg:
        return 0, torch.empty(0, dtype=torch.int32), None
    ps = fr.Plan(src_reg, chunk_bytes, n_batches=n_batches)
    pd = fr.Plan(dst_reg, chunk_bytes, n_batches=n_batches)
    if staging is None:
        staging = ps.new_packed()
    dev = dst_reg[0].device
    s_src = stream_src or torch.cuda.Stream(device=dev)
    s_dst = stream_dst or torch.cuda.Stream(device=dev)
    cnt = torch.empty(1, dtype=torch.int64, device=dev)
    s_src.wait_stream(torch.cuda.current_stream(dev))
    s_dst.wait_stream(torch.cuda.current_stream(dev))
    fr.fr_restore(ps.handle, pd.handle, staging, max_retries, None, cnt, s_src, s_dst)
    diverged = torch.empty(0, dtype=torch.int32)
    with torch.cuda.stream(s_dst):
        if verify:
            ta = ps.fingerprint(stream=s_dst)
            tb = pd.fingerprint(stream=s_dst)
            diverged, _ = fr.diff(ta, tb, stream=s_dst)
    s_dst.synchronize()
    return int(cnt.item()), diverged, (ps, pd)


def _cuts(n_elems: int, eb: int, n_dst: int, rank: int, n_src: int):
    return [do for _, _, do, _ in fr.fr_shard_pieces(n_elems, eb, n_dst, rank, n_src)]


def common_regions(n_elems: Sequence[int], elem_bytes: Sequence[int], n_dst: int, rank: int,
                   a_sources: Sequence[Sequence[torch.Tensor]], n_a: int,
                   b_sources: Sequence[Sequence[torch.Tensor]], n_b: int):
    """Matching regions of two replica groups (sharded `n_a` and `n_b` ways)
    over the bytes of shard `rank` of `n_dst`: each region lies inside one
    shard of each group, cut at every piece boundary of both."""
    ra, rb = [], []
    for g, n in enumerate(n_elems):
        eb = elem_bytes[g]
        a0, b0 = shard_range(n, n_dst, rank)
        length = (b0 - a0) * eb
        if length == 0:
            continue
        pa = fr.fr_shard_pieces(n, eb, n_dst, rank, n_a)
        pb = fr.fr_shard_pieces(n, eb, n_dst, rank, n_b)
        cuts = sorted(set(_cuts(n, eb, n_dst, rank, n_a)) | set(_cuts(n, eb, n_dst, rank, n_b)) | {length})
        ia = ib = 0
        for lo, hi in zip(cuts[:-1], cuts[1:]):
            while pa[ia][2] + pa[ia][3] <= lo:
                ia += 1
            while pb[ib][2] + pb[ib][3] <= lo:
                ib += 1
            for (j, so, do, _), srcs, out in ((pa[ia], a_sources, ra), (pb[ib], b_sources, rb)):
                off = (so + lo - do) // eb
                out.append(srcs[j][g][off:off + (hi - lo) // eb])
    return ra, rb


def cross_check(n_elems: Sequence[int], elem_bytes: Sequence[int], n_dst: int, rank: int,
                a_sources, n_a: int, b_sources, n_b: int, chunk_bytes: int, stream=None):
    """Chunks (of the common-region plan) where replica groups A and B
    disagree over shard `rank`'s bytes.  Returns (diverged ids, regions of A)."""
    ra, rb = common_regions(n_elems, elem_bytes, n_dst, rank, a_sources, n_a, b_sources, n_b)
    if not ra:
        return torch.empty(0, dtype=torch.int32), ra
    pa, pb = fr.Plan(ra, chunk_bytes), fr.Plan(rb, chunk_bytes)
    ids, _ = fr.diff(pa.fingerprint(stream=stream), pb.fingerprint(stream=stream), stream=stream)
    return ids, ra
