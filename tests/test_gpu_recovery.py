"""A recovery end to end on one GPU (Sec. III-E): four data-parallel replicas
of one state, a failure reported to the step-tag controller, the failed
rank's state rebuilt from the replica the controller picks with the fused,
pipelined restore, and the whole group's fingerprints compared."""
import pytest
import torch

from paper_2509_03047_gb300 import steptag, synth

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")


@pytest.fixture(autouse=True)
def _free_memory():
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("phase", ["forward_backward", "optimizer"])
@pytest.mark.parametrize("where", ["device", "pinned"])
def test_failed_rank_is_restored_from_the_chosen_replica(phase, where):
    cfg = synth.get_config("tiny")
    base = synth.make_state(cfg, "cuda")
    synth.inject_nonfinite(cfg, base)
    replicas = [[t.clone() for t in base] for _ in range(4)]
    plans = [fr.Plan(r, cfg.chunk_bytes, n_batches=5) for r in replicas]

    # rank 1 fails; the others report the step they hold
    ctl = steptag.Controller(4, [[0, 1, 2, 3]])
    ctl.heartbeat(1, steptag.OPTIMIZER if phase == "optimizer" else 6)
    ctl.report_failure(1)
    for r in (0, 2, 3):
        ctl.heartbeat(r, 7 if phase == "optimizer" else 6)
    d = ctl.decide()
    assert d.restore == [1] and d.phase == phase and d.resume_step == (7 if phase == "optimizer" else 6)
    src = d.source[1]

    # the restarted process starts from garbage
    for t in replicas[1]:
        t.view(torch.uint8).fill_(0xA5)
    staging = plans[src].new_packed(pinned=(where == "pinned"))
    fa, fb = plans[src].new_table(), plans[1].new_table()
    cnt = torch.full((1,), -1, dtype=torch.int64, device="cuda")
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    fr.fr_restore_fp(plans[src].handle, plans[1].handle, staging, 1, None, cnt, fa, fb, s1, s2)
    s2.synchronize()
    assert int(cnt.item()) == 0
    assert fr.diff(fa, fb)[1] == 0

    # every replica of the group now agrees, chunk for chunk
    tables = [p.fingerprint() for p in plans]
    for t in tables[1:]:
        assert fr.diff(tables[0], t)[1] == 0
    assert torch.equal(tables[1], fb)
    for a, b in zip(replicas[0], replicas[1]):
        assert torch.equal(a.view(torch.uint8), b.view(torch.uint8))
