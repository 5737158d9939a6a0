"""The restoration step captured once in a CUDA graph and replayed: the plain
calls only enqueue kernels on the given stream (no allocation, no host sync),
so a whole fingerprint -> pack -> unpack_verify -> fingerprint -> diff step can
be replayed without per-call launch overhead.  Replays must give exactly the
eager results."""
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


@pytest.mark.parametrize("fused", [False, True])
def test_restore_step_replays_from_a_cuda_graph(fused):
    cfg = synth.get_config("tiny")
    src = synth.make_state(cfg, "cuda")
    synth.inject_nonfinite(cfg, src)
    dst = [torch.empty_like(t) for t in src]
    a, b = fr.Plan(src, cfg.chunk_bytes), fr.Plan(dst, cfg.chunk_bytes)
    C = a.n_chunks
    packed = a.new_packed()
    ta, tb = a.new_table(), b.new_table()
    mism = torch.empty(C, dtype=torch.int32, device="cuda")
    nmis = torch.empty(1, dtype=torch.int64, device="cuda")
    div = torch.empty(C, dtype=torch.int32, device="cuda")
    ndiv = torch.empty(1, dtype=torch.int64, device="cuda")

    def step(s):
        if fused:
            fr.fr_pack_fp(a.handle, packed, ta, s)
            fr.fr_unpack_verify_fp(b.handle, packed, mism, nmis, tb, s)
        else:
            fr.fr_fingerprint(a.handle, ta, s)
            fr.fr_pack(a.handle, packed, s)
            fr.fr_unpack_verify(b.handle, packed, mism, nmis, s)
            fr.fr_fingerprint(b.handle, tb, s)
        fr.fr_diff(ta, tb, C, div, ndiv, s)

    # eager reference
    step(torch.cuda.current_stream())
    torch.cuda.synchronize()
    want = (ta.clone(), tb.clone(), packed.clone(), int(nmis.item()), int(ndiv.item()))
    assert want[3] == 0 and want[4] == 0

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        step(s)
    torch.cuda.synchronize()
    for k in range(3):
        for t in dst:  # the receiver starts from garbage every replay
            t.view(torch.uint8).fill_(0x5A + k)
        for x in (ta, tb, packed):
            x.fill_(0xEE)
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(ta, want[0]) and torch.equal(tb, want[1]) and torch.equal(packed, want[2])
        assert int(nmis.item()) == 0 and int(ndiv.item()) == 0
        assert all(torch.equal(x.view(torch.uint8), y.view(torch.uint8)) for x, y in zip(src, dst))
