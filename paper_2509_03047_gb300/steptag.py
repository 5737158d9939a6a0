"""Step tags: when to stop, clean and reset, and at which step to resume.

FlashRecovery (arXiv 2509.03047, Sec. III-E) resumes a failed job at step i or
step i+1 depending on where the failure hit, and learns both from tags the
training processes report through their heartbeats:

* a process sets tag = i when step i's forward pass starts;
* a barrier, merged with the gradient all-reduce, precedes the optimizer
  step, so either every process is still in forward/backward of step i or
  every process has entered the optimizer step of step i;
* a process sets tag = -1 when its optimizer step starts and tag = i+1 when
  that step ends.

So once every normal process reports the same non-negative tag T, none of
them is inside an optimizer step and all hold the model state after T
updates: the controller can stop, clean and reset them at once, restore the
failed processes' state from a data-parallel replica (with the library's
fr_restore) and resume at step T -- step i after a forward/backward failure,
step i+1 after an optimizer failure.  While any normal process reports -1 the
controller waits for its optimizer step to finish.  If every replica of a
failed process is lost too, only a checkpoint can help (the paper's first
limitation, Sec. III-G).

Failures reach the controller two ways (Sec. III-C): a report (the process
is gone, or a device plugin says so), or a heartbeat that stops -- a rank
that hangs without exiting is declared failed once it has been silent for
`heartbeat_timeout` seconds.

This module is host logic only: the Controller, and a simulation that runs
ranks as separate CPU processes reporting tags and heartbeats through a
torch TCPStore, with faults made on the host (a rank exits, or hangs without
exiting).  No GPU is involved.
"""
from __future__ import annotations

import os
import time
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence

OPTIMIZER = -1


class NoReplicaError(RuntimeError):
    """Every data-parallel replica of a failed rank is lost."""


@dataclass
class Decision:
    resume_step: int                 # the step training resumes at
    phase: str                       # "forward_backward" or "optimizer": where the failure hit
    stop: List[int]                  # normal ranks to stop, clean and reset
    restore: List[int]               # failed ranks to restore
    source: Dict[int, int] = field(default_factory=dict)  # failed rank -> replica rank


class Controller:
    """Collects step tags and failure reports; decides when and where to resume.

    `dp_groups`: lists of ranks that hold replicas of the same model state."""

    def __init__(self, world_size: int, dp_groups: Sequence[Sequence[int]],
                 heartbeat_timeout: Optional[float] = None):
        self.world_size = world_size
        self.heartbeat_timeout = heartbeat_timeout
        self.beats: Dict[int, tuple] = {}  # rank -> (heartbeat count, time it last changed)
        self.group_of: Dict[int, List[int]] = {}
        for g in dp_groups:
            for r in g:
                self.group_of[r] = list(g)
        if sorted(self.group_of) != list(range(world_size)):
            raise ValueError("the data-parallel groups must cover every rank once")
        self.tags: Dict[int, int] = {}
        self.failed: set = set()

    def heartbeat(self, rank: int, tag: int) -> None:
        self.tags[rank] = tag

    def report_failure(self, rank: int) -> None:
        self.failed.add(rank)

    def beat(self, rank: int, count: int, now: float) -> None:
        """A rank's heartbeat counter as last read; only a change counts as a
        beat, and a rank's clock starts with its first beat (a process still
        starting up is not silent)."""
        if count == 0:
            return
        old = self.beats.get(rank)
        if old is None or old[0] != count:
            self.beats[rank] = (count, now)

    def check_timeouts(self, now: float) -> List[int]:
        """Declare failed every rank silent for longer than the timeout; returns them."""
        if self.heartbeat_timeout is None:
            return []
        out = [r for r, (_, t) in self.beats.items()
               if r not in self.failed and now - t > self.heartbeat_timeout]
        for r in out:
            self.report_failure(r)
        return out

    def decide(self) -> Optional[Decision]:
        """A decision once it is safe to stop the normal ranks, else None."""
        if not self.failed:
            return None
        normal = [r for r in range(self.world_size) if r not in self.failed]
        tags = [self.tags.get(r) for r in normal]
        if any(t is None for t in tags):
            return None  # not heard from every normal rank yet
        if any(t == OPTIMIZER for t in tags):
            return None  # an optimizer step is running: let it finish
        if len(set(tags)) != 1:
            return None  # the tags still disagree (heartbeats in flight)
        resume = tags[0]
        phase = "optimizer" if any(self.tags.get(f) == OPTIMIZER for f in self.failed) else "forward_backward"
        source = {}
        for f in sorted(self.failed):
            alive = [r for r in self.group_of[f] if r not in self.failed]
            if not alive:
                raise NoReplicaError("rank %d has no surviving data-parallel replica" % f)
            source[f] = alive[0]
        return Decision(resume, phase, normal, sorted(self.failed), source)


# ---------------------------------------------------------------- simulation

def _rank_main(rank: int, world: int, host: str, port: int, n_steps: int, fail_step: int, fail_phase: str,
               step_time: float, fail_mode: str = "exit") -> None:
    """One simulated training process.  Its 'model state' is the number of
    optimizer updates it applied, reported with every tag; it beats its
    heartbeat counter with every tag and while it waits.  fail_mode "exit":
    the process dies; "hang": it stays alive but goes silent until stopped."""
    from datetime import timedelta

    import torch.distributed as dist

    store = dist.TCPStore(host, port, world + 1, False, timeout=timedelta(seconds=60))
    updates = 0

    def beat():
        store.add("hb/%d" % rank, 1)

    def tag(t):
        store.set("state/%d" % rank, str(updates))
        store.set("tag/%d" % rank, str(t))
        beat()

    def stopped():
        return store.check(["stop"])

    def fail():
        if fail_mode == "exit":
            os._exit(3)  # the fault: this process dies
        while not stopped():  # the fault: alive, silent
            time.sleep(0.005)

    for i in range(n_steps):
        tag(i)
        if fail_phase == "forward_backward" and i == fail_step:
            return fail()
        time.sleep(step_time)  # forward and backward
        # barrier merged with the gradient all-reduce
        store.add("barrier/%d" % i, 1)
        while int(store.add("barrier/%d" % i, 0)) < world:
            if stopped():
                return
            beat()
            time.sleep(0.005)
        tag(OPTIMIZER)
        if fail_phase == "optimizer" and i == fail_step:
            return fail()
        time.sleep(step_time / 2)  # the optimizer step
        updates += 1
        tag(i + 1)
    while not stopped():
        beat()
        time.sleep(0.005)


def simulate(world: int, dp_groups: Sequence[Sequence[int]], n_steps: int, fail_rank: int, fail_step: int,
             fail_phase: str, step_time: float = 0.02, timeout: float = 60.0, fail_mode: str = "exit",
             heartbeat_timeout: float = 5.0):
    """Run `world` CPU ranks; rank `fail_rank` dies ("exit") or goes silent
    ("hang") in `fail_phase` of step `fail_step`.  Returns (decision, {rank:
    updates held when stopped})."""
    import multiprocessing as mp
    import socket
    from datetime import timedelta

    import torch.distributed as dist

    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    store = dist.TCPStore("127.0.0.1", port, world + 1, True, timeout=timedelta(seconds=60),
                          wait_for_workers=False)
    ctx = mp.get_context("spawn")
    procs = []
    for r in range(world):
        fs, fp = (fail_step, fail_phase) if r == fail_rank else (-1, "")
        procs.append(ctx.Process(target=_rank_main,
                                 args=(r, world, "127.0.0.1", port, n_steps, fs, fp, step_time, fail_mode)))
    for p in procs:
        p.start()
    ctl = Controller(world, dp_groups, heartbeat_timeout=heartbeat_timeout)
    decision = None
    t0 = time.time()
    try:
        while decision is None:
            if time.time() - t0 > timeout:
                raise TimeoutError("no decision")
            now = time.time()
            for r, p in enumerate(procs):
                if p.exitcode not in (None, 0):
                    ctl.report_failure(r)  # the monitoring side: the process is gone
                if store.check(["tag/%d" % r]):
                    ctl.heartbeat(r, int(store.get("tag/%d" % r)))
                ctl.beat(r, int(store.add("hb/%d" % r, 0)), now)
            ctl.check_timeouts(now)  # silent ranks
            decision = ctl.decide()
            time.sleep(0.01)
        store.set("stop", "1")
        for r in decision.stop:
            procs[r].join(timeout=30)
        held = {r: int(store.get("state/%d" % r)) for r in decision.stop}
    finally:
        for p in procs:
            if p.is_alive():
                p.kill()
            p.join(timeout=5)
    return decision, held
