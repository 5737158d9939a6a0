"""The step-tag protocol (Sec. III-E): resume at step i after a forward/backward
failure, at step i+1 after an optimizer failure, never while an optimizer step
runs, and from a surviving data-parallel replica.  Ranks are CPU processes;
the fault is made on the host (a rank exits)."""
import pytest

from paper_2509_03047_gb300 import steptag as st

GROUPS = [[0, 2], [1, 3]]  # two data-parallel groups of two replicas


def test_decision_waits_for_the_optimizer_and_for_agreement():
    c = st.Controller(4, GROUPS)
    for r in range(4):
        c.heartbeat(r, 5)
    assert c.decide() is None  # no failure
    c.report_failure(1)
    c.heartbeat(0, st.OPTIMIZER)
    assert c.decide() is None  # rank 0 is inside an optimizer step
    c.heartbeat(0, 6)
    assert c.decide() is None  # ranks disagree (6 vs 5): heartbeats in flight
    c.heartbeat(2, 6)
    c.heartbeat(3, 6)
    d = c.decide()
    assert d.resume_step == 6 and d.stop == [0, 2, 3] and d.restore == [1] and d.source == {1: 3}


def test_phase_comes_from_the_failed_ranks_last_tag():
    c = st.Controller(4, GROUPS)
    for r in range(4):
        c.heartbeat(r, st.OPTIMIZER)
    c.report_failure(2)
    for r in (0, 1, 3):
        c.heartbeat(r, 8)
    d = c.decide()
    assert d.phase == "optimizer" and d.resume_step == 8 and d.source == {2: 0}


def test_all_replicas_lost_needs_a_checkpoint():
    c = st.Controller(4, GROUPS)
    for r in range(4):
        c.heartbeat(r, 3)
    c.report_failure(1)
    c.report_failure(3)
    with pytest.raises(st.NoReplicaError):
        c.decide()


def test_groups_must_cover_every_rank():
    with pytest.raises(ValueError):
        st.Controller(4, [[0, 1], [2]])


@pytest.mark.parametrize("phase,fail_step,resume", [("forward_backward", 3, 3), ("optimizer", 3, 4)])
def test_simulated_failure_resumes_at_the_right_step(phase, fail_step, resume):
    decision, held = st.simulate(world=4, dp_groups=GROUPS, n_steps=8, fail_rank=1, fail_step=fail_step,
                                 fail_phase=phase)
    assert decision.phase == phase
    assert decision.resume_step == resume
    assert decision.restore == [1] and decision.source == {1: 3}
    # every normal replica holds exactly the state of the resume step, so the
    # failed rank restored from its replica agrees with everyone
    assert set(held.values()) == {resume}


def test_heartbeat_timeout_declares_a_silent_rank_failed():
    c = st.Controller(4, GROUPS, heartbeat_timeout=1.0)
    for r in range(4):
        c.beat(r, 1, now=0.0)
        c.heartbeat(r, 7)
    for r in (0, 2, 3):
        c.beat(r, 5, now=0.8)  # ranks 0, 2, 3 keep beating; rank 1 falls silent
        c.beat(r, 5, now=0.9)  # an unchanged counter is not a beat
    assert c.check_timeouts(now=0.95) == []
    assert c.check_timeouts(now=1.05) == [1]
    d = c.decide()
    assert d.restore == [1] and d.resume_step == 7 and d.source == {1: 3}
    assert c.check_timeouts(now=1.75) == []
    assert c.check_timeouts(now=1.85) == [0, 2, 3]  # silent since 0.8


@pytest.mark.parametrize("phase,resume", [("forward_backward", 2), ("optimizer", 3)])
def test_simulated_hang_is_found_by_its_silent_heartbeat(phase, resume):
    decision, held = st.simulate(world=4, dp_groups=GROUPS, n_steps=6, fail_rank=2, fail_step=2, fail_phase=phase,
                                 fail_mode="hang", heartbeat_timeout=2.0)
    assert decision.restore == [2] and decision.source == {2: 0}
    assert decision.resume_step == resume and decision.phase == phase
    assert set(held.values()) == {resume}
