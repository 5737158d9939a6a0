"""The recovery-overhead model against the numbers the paper prints and the
closed forms of Eq. 1-5 (tests/golden/paper_numbers.json)."""
import json
import math
import os
import random

import pytest

from paper_2509_03047_gb300 import overhead as ov

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_numbers.json")))


def test_printed_survival_probabilities():
    for row in GOLD["all_survive"]:
        assert round(ov.all_survive(row["p_fail"], row["n"]), 5) == row["printed"]


def test_printed_replica_loss_probability():
    for row in GOLD["all_replicas_lost"]:
        assert math.isclose(ov.all_replicas_lost(row["p_fail"], row["dp"]), row["printed"], rel_tol=1e-12)


def test_table_iii_accounting():
    for params, devices, detect, restart, step, half, total in GOLD["table_iii"]["rows"]:
        assert half == step / 2
        assert ov.recovery_time(detect, restart, step) == total


def test_scale_claims():
    rows = GOLD["table_iii"]["rows"]
    first, last = rows[0], rows[-1]
    assert round(100 * (last[6] / first[6] - 1)) == GOLD["scale_claims"]["growth_percent"]
    assert last[1] / first[1] == GOLD["scale_claims"]["device_ratio"]


def test_optimum_of_eq1_matches_eq3_and_eq4():
    rng = random.Random(0)
    for _ in range(200):
        m, s0, d, k0 = rng.uniform(0.5, 50), rng.uniform(10, 2000), rng.uniform(1e3, 1e6), rng.uniform(1, 600)
        t = ov.optimal_interval(m, d, k0)
        assert abs(ov.overhead_slope(t, m, d, k0)) <= 1e-9 * (m + d * k0 / t ** 2)
        assert math.isclose(ov.total_overhead(t, m, s0, d, k0), ov.minimal_overhead(m, s0, d, k0), rel_tol=1e-12)
        for f in (0.5, 0.9, 1.1, 2.0):  # a minimum, not a maximum
            assert ov.total_overhead(f * t, m, s0, d, k0) > ov.minimal_overhead(m, s0, d, k0)


def test_checkpoint_free_removes_the_checkpoint_term():
    # Eq. 5 is Eq. 1 with k0 = 0 and s1 bounded by one step (t = 2 s1')
    for m, s0, s1 in [(3, 90, 3), (10, 120, 24.5)]:
        assert ov.checkpoint_free_overhead(m, s0, s1) == ov.total_overhead(2 * s1, m, s0, 1.0, 0.0)


def test_invalid_arguments():
    with pytest.raises(ValueError):
        ov.total_overhead(0, 1, 1, 1, 1)
    with pytest.raises(ValueError):
        ov.optimal_interval(0, 1, 1)
