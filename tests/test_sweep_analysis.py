"""Host-side analysis of the threshold sweep (no GPU): trace differences,
the settling step, the fixed-line criterion and transition schedules."""

import math

import pytest

from paper_2607_12358_gb300 import sweep as W


def test_differences_of_a_quadratic():
    # s_t = t^2: first differences 2t - 1, second differences 2
    tr = [math.nan] + [float(t * t) for t in range(1, 7)]
    d1, d2 = W.differences(tr)
    assert all(math.isnan(x) for x in d1[:2]) and d1[2:] == [3.0, 5.0, 7.0, 9.0, 11.0]
    assert all(math.isnan(x) for x in d2[:3]) and d2[3:] == [2.0, 2.0, 2.0, 2.0]


def test_stable_from():
    tr = [math.nan, 0.5, 0.2, 0.1, 0.11, 0.1, 0.105]
    # differences from step 2: -0.3, -0.1, 0.01, -0.01, 0.005
    assert W.stable_from(tr, 0.02) == 4
    assert W.stable_from(tr, 0.2) == 3
    assert W.stable_from(tr, 1.0) == 2
    assert W.stable_from(tr, 0.001) is None
    assert W.stable_from([math.nan, 1.0], 0.1) == 2


def test_beats_fixed_line():
    lo = {"computed": 30, "rel_l2": 0.01}
    hi = {"computed": 10, "rel_l2": 0.05}
    # the line through (10, 0.05) and (30, 0.01) passes (20, 0.03)
    assert W.beats_fixed_line({"computed": 20, "rel_l2": 0.029}, lo, hi)
    assert not W.beats_fixed_line({"computed": 20, "rel_l2": 0.031}, lo, hi)
    assert W.beats_fixed_line({"computed": 10, "rel_l2": 0.04}, lo, hi)
    same = {"computed": 10, "rel_l2": 0.02}
    assert W.beats_fixed_line({"computed": 10, "rel_l2": 0.01}, same, dict(same, rel_l2=0.03))


@pytest.mark.parametrize("k", [0, 1, 7, 10])
def test_transition_schedule(k):
    s = W.transition_schedule(10, k, 0.05, 0.2)
    assert len(s) == 10 and s[:k] == [0.05] * k and s[k:] == [0.2] * (10 - k)
