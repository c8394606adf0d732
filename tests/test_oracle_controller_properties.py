"""Property-based checks of the oracle's controller (Algorithm 1, Sec. 3.3)
on arbitrary non-negative signal sequences.

For a fixed signal sequence the threshold chosen at step t depends on the
signals alone (|s_t - s_prev| against delta), so Algorithm 1 is a greedy
reset rule under a per-step threshold tau_t in [tau_low, tau_high]:
accumulate, skip while the sum stays within tau_t, otherwise compute and
reset.  A greedy rule under pointwise larger thresholds never computes more
often: by induction on k, its k-th compute never comes before the other
rule's k-th compute.  Once the other rule has restarted its sum no later,
that sum covers at least as many non-negative signals, against a threshold
no larger.  Hence the compute counts sit between those of the fixed
thresholds.  The other properties are special
cases of the rule: equal thresholds, a negative delta, zero signals, and a
power-of-two rescaling of every quantity (exact in binary floating point).
"""

import pytest

import oracle as O

hyp = pytest.importorskip("hypothesis")
st = pytest.importorskip("hypothesis.strategies")
given, settings = hyp.given, hyp.settings

signals = st.lists(st.floats(min_value=0.0, max_value=1.0, allow_nan=False, allow_infinity=False),
                   min_size=1, max_size=60)
thresholds = st.tuples(st.floats(min_value=0.0, max_value=2.0), st.floats(min_value=0.0, max_value=2.0)).map(sorted)
deltas = st.floats(min_value=0.0, max_value=0.5)
warmups = st.integers(min_value=0, max_value=3)


def _count(seq, warmup, lo, hi, delta):
    return sum(O.controller_decisions(seq, warmup, lo, hi, delta))


@settings(max_examples=300, deadline=None)
@given(signals, warmups, thresholds, deltas)
def test_compute_count_between_fixed_thresholds(seq, warmup, th, delta):
    lo, hi = th
    n = _count(seq, warmup, lo, hi, delta)
    assert _count(seq, warmup, hi, hi, delta) <= n <= _count(seq, warmup, lo, lo, delta)


@settings(max_examples=200, deadline=None)
@given(signals, warmups, st.floats(min_value=0.0, max_value=2.0), deltas)
def test_equal_thresholds_are_fixed_tau(seq, warmup, tau, delta):
    """With tau_low = tau_high the delta rule has nothing to choose: the
    decisions are those of fixed-tau caching, whatever delta is."""
    assert O.controller_decisions(seq, warmup, tau, tau, delta) == O.controller_decisions(seq, warmup, tau, tau, 1e9)


@settings(max_examples=200, deadline=None)
@given(signals, warmups, thresholds)
def test_negative_delta_is_fixed_low(seq, warmup, th):
    lo, hi = th
    assert O.controller_decisions(seq, warmup, lo, hi, -1.0) == O.controller_decisions(seq, warmup, lo, lo, 0.0)


@settings(max_examples=100, deadline=None)
@given(st.integers(min_value=1, max_value=60), warmups, thresholds, deltas)
def test_zero_signal_skips_every_non_warmup_step(n, warmup, th, delta):
    lo, hi = th
    dec = O.controller_decisions([0.0] * n, warmup, lo, hi, delta)
    assert dec == [True] * min(n, warmup) + [False] * max(0, n - warmup)


@settings(max_examples=200, deadline=None)
@given(signals, warmups, thresholds, deltas, st.integers(min_value=0, max_value=8))
def test_power_of_two_rescaling_changes_nothing(seq, warmup, th, delta, e):
    """Multiplying the signals, both thresholds and delta by 2^e changes no
    decision: every sum, difference and comparison scales exactly.  Scaling
    up keeps this exact even for subnormal inputs; scaling down could
    underflow, so e >= 0."""
    lo, hi = th
    c = 2.0 ** e
    assert O.controller_decisions([c * s for s in seq], warmup, c * lo, c * hi, c * delta) == \
        O.controller_decisions(seq, warmup, lo, hi, delta)
