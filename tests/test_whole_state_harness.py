"""The whole-state harness (tests/whole_state.py) on the CPU: fed the oracle's
own outputs it reports no failure, and every planted mistake in a "device"
output (here CPU tensors standing in for the GPU's) is reported at exactly its
chunk.  Small slices force the state through several host slices and many
thread tasks."""
import numpy as np
import pytest
import torch

import oracle
import whole_state
from paper_2509_03047_gb300 import synth


def expected_owner(chunks, bit_positions):
    """Chunks owning a flipped byte, from the documented layout: header k ->
    k, the gap after the header table -> the last chunk, payload or padding ->
    its chunk."""
    C = len(chunks)
    starts = chunks["payload_off"].astype(np.int64)
    owners = set()
    for b in (bit_positions // 8).tolist():
        if b < 64 * C:
            owners.add(b // 64)
        elif b < starts[0]:
            owners.add(C - 1)
        else:
            owners.add(int(np.searchsorted(starts, b, side="right")) - 1)
    return np.array(sorted(owners), dtype=np.int64)


def _state():
    g = torch.Generator().manual_seed(3)
    ts = [torch.randn(n, generator=g) for n in (1000, 70000, 4, 33333)]
    ts.insert(1, torch.randn(50001, generator=g).to(torch.bfloat16))
    ts.insert(3, torch.randint(0, 256, (9999,), generator=g, dtype=torch.uint8))
    ts.append(torch.zeros(0))
    ts[2][17] = float("nan")
    dts = [oracle.DT_F32, oracle.DT_BF16, oracle.DT_F32, oracle.DT_BYTES, oracle.DT_F32, oracle.DT_F32,
           oracle.DT_F32]
    return ts, dts


@pytest.fixture(autouse=True)
def _small_slices(monkeypatch):
    monkeypatch.setattr(whole_state, "SLICE_BYTES", 40000)


def _oracle_outputs(ts, dts, chunk):
    host = [t.view(torch.uint8).numpy() for t in ts]
    table = oracle.fingerprint(host, dts, chunk)
    packed = torch.from_numpy(oracle.pack(host, dts, chunk))
    return table, packed


def test_clean_state_passes_and_tables_fill():
    ts, dts = _state()
    chunk = 4096
    table, packed = _oracle_outputs(ts, dts, chunk)
    ws = whole_state.WholeState(ts, dts, chunk, threads=3)
    assert ws.check_pack(table, packed) == []
    assert np.array_equal(ws.table, table)
    restored = [torch.empty_like(t) for t in ts]
    dst = [r.view(torch.uint8).numpy() for r in restored]
    rc, ids, n = oracle.unpack_verify(dst, dts, chunk, packed.numpy())
    fails, want_ids = ws.check_restore(packed, restored, table)
    assert fails == [] and want_ids.size == 0 and n == 0
    d, k = ws.oracle_diff()
    assert k == 0


def test_planted_mistakes_are_reported_at_their_chunk():
    ts, dts = _state()
    chunk = 4096
    table, packed = _oracle_outputs(ts, dts, chunk)
    ws = whole_state.WholeState(ts, dts, chunk, threads=4)
    C = ws.C
    bad_tab = table.copy()
    bad_tab["crc32c"][5] ^= 1
    bad_tab["sumsq"][9] *= 1 + 1e-8
    bad_pack = packed.clone()
    poff, ln = int(ws.chunks["payload_off"][12]), int(ws.chunks["len"][12])
    bad_pack[poff + ln // 2] ^= 4                       # payload of chunk 12
    bad_pack[64 * 20 + 33] ^= 1                         # header of chunk 20
    t_last = int(ws.chunks["len"][C - 1])
    if t_last % 256:
        bad_pack[int(ws.chunks["payload_off"][C - 1]) + t_last] = 7  # padding of the last chunk
    fails = ws.check_pack(bad_tab, bad_pack)
    where = sorted({c for c, _ in fails})
    want = sorted({5, 9, 12, 20} | ({C - 1} if t_last % 256 else set()))
    assert where == want, fails
    assert any(c == 9 and w.startswith("sumsq") for c, w in fails)
    assert (12, "payload") in fails and (20, "header") in fails


def test_restore_pass_finds_flips_and_wrong_restored_bytes():
    ts, dts = _state()
    chunk = 2048
    table, packed = _oracle_outputs(ts, dts, chunk)
    ws = whole_state.WholeState(ts, dts, chunk, threads=2)
    assert ws.check_pack(table, packed) == []
    flips = synth.flip_positions(packed.numel(), 25, seed=11)
    synth.apply_flips(packed, flips)
    restored = [torch.empty_like(t) for t in ts]
    dst = [r.view(torch.uint8).numpy() for r in restored]
    rc, ids, n = oracle.unpack_verify(dst, dts, chunk, packed.numpy())
    table_r = oracle.fingerprint(dst, dts, chunk)
    fails, want_ids = ws.check_restore(packed, restored, table_r)
    assert fails == []
    assert np.array_equal(want_ids, ids)
    assert np.array_equal(want_ids.astype(np.int64), expected_owner(ws.chunks, flips))
    d, k = ws.oracle_diff()
    assert np.array_equal(d, oracle.diff(table, table_r)[0])
    # a restored byte that is not the packed payload byte is caught
    ws2 = whole_state.WholeState(ts, dts, chunk, threads=2)
    ws2.check_pack(table, packed)
    c = 7
    t, off = int(ws.chunks["tensor_idx"][c]), int(ws.chunks["tensor_off"][c])
    restored[t].view(torch.uint8)[off + 3] ^= 0x10
    fails, _ = ws2.check_restore(packed, restored, table_r)
    assert {cc for cc, _ in fails} == {c}
