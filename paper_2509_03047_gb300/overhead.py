"""FlashRecovery's recovery-overhead model (arXiv 2509.03047).

Sec. II models the time a training job loses to failures over a period d with
m failures, per-failure recovery overhead s0, checkpoint interval t (steps)
and checkpoint dump time k0:

    F(t)  = m (s0 + t/2) + (d/t) k0                   (Eq. 1; s1 ~ t/2 recomputation)
    F'(t) = m/2 - d k0 / t^2                          (Eq. 2)
    t*    = sqrt(2 d k0 / m)                          (Eq. 3)
    Fmin  = m s0 + sqrt(2 d k0 m)                     (Eq. 4)

With checkpoint-free recovery from data-parallel replicas (Sec. III-F) the
checkpoint term vanishes and recomputation is bounded by one step:

    F     = m (s0' + s1')                             (Eq. 5)

Sec. II and III-A also give the probability arguments for replicas:
(1 - p)^n that n devices all survive, p^N that all N replicas of a state are
lost.  Table III accounts each recovery as detection + restart + step/2.
Host-side arithmetic only; nothing here runs on the GPU.
"""
from __future__ import annotations

import math


def total_overhead(t: float, m: float, s0: float, d: float, k0: float) -> float:
    """Eq. 1: recovery time plus checkpointing time over the period d."""
    if t <= 0:
        raise ValueError("the checkpoint interval must be positive")
    return m * (s0 + t / 2.0) + (d / t) * k0


def overhead_slope(t: float, m: float, d: float, k0: float) -> float:
    """Eq. 2: dF/dt."""
    return m / 2.0 - d * k0 / (t * t)


def optimal_interval(m: float, d: float, k0: float) -> float:
    """Eq. 3: the interval where Eq. 2 vanishes."""
    if m <= 0:
        raise ValueError("no failures: the optimum is an infinite interval")
    return math.sqrt(2.0 * d * k0 / m)


def minimal_overhead(m: float, s0: float, d: float, k0: float) -> float:
    """Eq. 4: Eq. 1 at the optimal interval."""
    return m * s0 + math.sqrt(2.0 * d * k0 * m)


def checkpoint_free_overhead(m: float, s0_opt: float, s1_opt: float) -> float:
    """Eq. 5: no checkpoint term; s1' is at most one training step."""
    return m * (s0_opt + s1_opt)


def all_survive(p_fail: float, n: int) -> float:
    """Probability that n devices with failure probability p_fail all work."""
    return (1.0 - p_fail) ** n


def all_replicas_lost(p_fail: float, dp: int) -> float:
    """Probability that all dp data-parallel replicas of a state fail."""
    return p_fail ** dp


def recovery_time(detect: float, restart: float, step: float) -> float:
    """One recovery as Table III accounts it: detection + restart + half a
    step of redone training."""
    return detect + restart + step / 2.0
