"""Pins of the acceptance rules for end-to-end losses (oracle/rounding.py)
against their stated meaning.  CPU only."""
import numpy as np

from oracle import rounding


def test_within_is_the_relative_bound_or_the_furthest_member():
    ref = 2.0
    ens = np.array([2.01, 1.97, 2.02])
    assert rounding.within(2.0 + 1.9e-3, ref, ens)           # 1e-3 relative
    assert rounding.within(1.97, ref, ens)                  # as far as the furthest member
    assert rounding.within(2.03, ref, ens)                  # the other side, same distance
    assert not rounding.within(2.0301, ref, ens)
    assert not rounding.within(1.9699, ref, ens)
    assert not rounding.within(2.01, ref, np.array([]))     # no members: the relative bound only


def test_consistent_false_alarm_rate_matches_student_t():
    """For a value drawn from the same normal distribution as the oracle and
    its 8 members, (value - mean) / (sd sqrt(1 + 1/9)) is Student-t with 8
    degrees of freedom, so k = 5 rejects it with probability
    2 P(t_8 > 5 / sqrt(10/9)) ~ 1.5e-3."""
    rng = np.random.default_rng(0)
    n, trials = 8, 40000
    x = rng.standard_normal((trials, n + 2))
    rejected = sum(not rounding.consistent(x[t, 0], x[t, 1], x[t, 2:]) for t in range(trials))
    rate = rejected / trials
    assert 0.0003 < rate < 0.004, rate


def test_consistent_rejects_a_shifted_value():
    rng = np.random.default_rng(1)
    ens = rng.standard_normal(8) * 0.1 + 3.0
    assert not rounding.consistent(3.0 + 2.0, 3.0, ens)
    assert rounding.consistent(3.05, 3.0, ens)


def test_agrees_is_either_rule_and_summary_reports_z():
    ref, ens = 1.0, np.array([1.1, 0.9, 1.05, 0.95, 1.0, 1.02, 0.98, 1.01])
    assert rounding.agrees(1.2, ref, ens)                   # outside the members, inside 5 sd
    assert not rounding.agrees(1.5, ref, ens)
    s = rounding.summary(1.2, ref, ens)
    allv = np.concatenate([[ref], ens])
    assert abs(s["z"] - (1.2 - allv.mean()) / allv.std(ddof=1)) < 1e-12
    assert s["ens_max_dev"] == max(abs(ens - ref))
