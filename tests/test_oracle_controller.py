"""Pins for the oracle's controller (Algorithm 1, Sec. 3.3) and step loop.

The golden cases in tests/golden/controller_cases.json were worked by hand
from Algorithm 1; the invariants below follow from it (proofs in the
docstrings) and do not re-run the oracle's own formula.
"""

import json
import math
import os

import numpy as np
import pytest

import acid_synth as S
import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "controller_cases.json")


def _run(signals, warmup, tl, th, delta):
    ctl = O.AcidController(tl, th, delta)
    comp, taus, sig = [], [], []
    for i, s in enumerate(signals):
        if i < warmup:
            comp.append(True)
            taus.append(None)
            sig.append(None)
            continue
        skip, tau, sg, _ = ctl.step(s)
        comp.append(not skip)
        taus.append(tau)
        sig.append(sg)
    return comp, taus, sig


@pytest.mark.parametrize("case", json.load(open(GOLDEN))["cases"], ids=lambda c: c["name"])
def test_golden_cases(case):
    comp, taus, sig = _run(case["signals"], case["warmup"], case["tau_low"], case["tau_high"],
                           case["delta"])
    assert comp == case["computed"]
    for a, b in zip(taus, case["tau"]):
        assert (a is None and b is None) or a == pytest.approx(b, abs=1e-12)
    for a, b in zip(sig, case["sigma"]):
        assert (a is None and b is None) or a == pytest.approx(b, abs=1e-12)


def _fixed_tau(signals, warmup, tau):
    """Fixed-threshold caching skeleton (Sec. 2, 'The Fixed Threshold...'):
    accumulate, reuse while the sum stays within tau, else run and reset."""
    acc = 0.0
    out = []
    for i, s in enumerate(signals):
        if i < warmup:
            out.append(True)
            continue
        acc += s
        if acc <= tau:
            out.append(False)
        else:
            out.append(True)
            acc = 0.0
    return out


def _random_signals(rng, n):
    # piecewise-smooth non-negative sequences with occasional jumps
    base = rng.uniform(0.0, 0.1)
    s = []
    for _ in range(n):
        if rng.uniform() < 0.25:
            base = rng.uniform(0.0, 0.15)
        s.append(max(0.0, base + rng.normal(0, 0.01)))
    return s


@pytest.mark.parametrize("seed", range(40))
def test_equal_thresholds_reduce_to_fixed_tau(seed):
    """tau_low == tau_high: the threshold no longer depends on the signal's
    rate of change, so ACID is the fixed-threshold method (Sec. 3.3)."""
    rng = np.random.default_rng(seed)
    s = _random_signals(rng, 50)
    tau = rng.uniform(0.02, 0.3)
    delta = rng.uniform(-0.05, 0.05)
    w = int(rng.integers(0, 3))
    assert O.controller_decisions(s, w, tau, tau, delta) == _fixed_tau(s, w, tau)


@pytest.mark.parametrize("seed", range(40))
def test_negative_delta_is_fixed_low(seed):
    """delta < 0 makes |s_t - s_prev| <= delta impossible: always tau_low."""
    rng = np.random.default_rng(100 + seed)
    s = _random_signals(rng, 50)
    tl, th = sorted(rng.uniform(0.02, 0.4, size=2))
    assert O.controller_decisions(s, 1, tl, th, -1.0) == _fixed_tau(s, 1, tl)


@pytest.mark.parametrize("seed", range(40))
def test_compute_count_between_fixed_thresholds(seed):
    """For non-negative signals the active threshold tau_t lies in
    [tau_low, tau_high] and depends on the signals only (s_prev is updated on
    every non-warmup step).  Greedy accumulate-and-reset with pointwise larger
    thresholds never computes earlier: if the k-th compute under the larger
    schedule is at e', the smaller schedule has accumulated at least the same
    segment sum by e' and so has computed k times by then.  Hence
    #computed(fixed tau_high) <= #computed(ACID) <= #computed(fixed tau_low)."""
    rng = np.random.default_rng(200 + seed)
    s = _random_signals(rng, 60)
    tl, th = sorted(rng.uniform(0.01, 0.4, size=2))
    delta = rng.uniform(0.0, 0.05)
    a = sum(O.controller_decisions(s, 1, tl, th, delta))
    lo = sum(_fixed_tau(s, 1, tl))
    hi = sum(_fixed_tau(s, 1, th))
    assert hi <= a <= lo


def test_zero_signal_skips_everything():
    d = O.controller_decisions([0.0] * 20, 2, 0.05, 0.2, 0.01)
    assert d == [True, True] + [False] * 18


def test_infinite_signal_forces_compute():
    d = O.controller_decisions([0.0, math.inf, 0.0, math.inf], 1, 1e9, 1e9, 1.0)
    assert d == [True, True, False, True]


def test_forced_decision_overrides_and_updates_state():
    ctl = O.AcidController(0.1, 0.1, 0.0)
    skip, _, sg, _ = ctl.step(0.5, forced=False)  # would compute; forced reuse keeps Sigma
    assert skip and sg == 0.5 and ctl.sigma == 0.5
    skip, _, sg, _ = ctl.step(0.0, forced=True)  # would skip? 0.5 > 0.1 computes anyway
    assert not skip and ctl.sigma == 0.0
    skip, _, _, _ = ctl.step(0.01, forced=True)
    assert not skip and ctl.sigma == 0.0


# ---------------------------------------------------------------------------
# Loop-level pins on the toy workload
# ---------------------------------------------------------------------------

@pytest.fixture(scope="module")
def toy():
    cfg = S.get_config("toy", steps=6)
    return cfg, S.model_weights(cfg, 0), S.latent(cfg, 0)


def _plain_sampler(cfg, w, lat, n):
    """No caching: every step evaluates the denoiser (Eq. 2 as Euler)."""
    sig = O.sigmas(n)
    x = lat.astype(np.float64)
    for i in range(n):
        v = O.denoiser(cfg, w, x, 1000.0 * sig[i], None)
        x = x + (sig[i + 1] - sig[i]) * v
    return x


def test_loop_negative_threshold_is_uncached(toy):
    cfg, w, lat = toy
    r = O.denoise_loop(cfg, w, lat, None, tau_low=-1.0, tau_high=-1.0)
    assert all(r.computed)
    np.testing.assert_allclose(r.latent, _plain_sampler(cfg, w, lat, cfg.steps), rtol=0, atol=1e-12)


def test_loop_huge_threshold_reuses_first_residual(toy):
    """With every non-warmup step skipped, TeaCache output is the final layer
    applied to H_in(x_t) + R_0, where R_0 is the block-stack residual of the
    first step."""
    cfg, w, lat = toy
    r = O.denoise_loop(cfg, w, lat, None, tau_low=1e9, tau_high=1e9)
    assert r.computed == [True] + [False] * (cfg.steps - 1)
    sig = O.sigmas(cfg.steps)
    x = lat.astype(np.float64)
    si = O.step_inputs(cfg, w, x, 1000.0 * sig[0])
    R0 = O.block_stack(cfg, w, si.h_in, si.mods, None) - si.h_in
    for i in range(cfg.steps):
        si = O.step_inputs(cfg, w, x, 1000.0 * sig[i])
        v = O.final_layer(cfg, w, si.h_in + R0, si.final_mod)
        x = x + (sig[i + 1] - sig[i]) * v
    np.testing.assert_allclose(r.latent, x, rtol=0, atol=1e-12)


def test_force_last_computes_the_final_step(toy):
    """force_last overrides a skip on the final step only: with every other
    non-warmup step reused, the last step runs the block stack (and is marked
    forced), which the replay below does by hand."""
    cfg, w, lat = toy
    r = O.denoise_loop(cfg, w, lat, None, tau_low=1e9, tau_high=1e9, force_last=True)
    assert r.computed == [True] + [False] * (cfg.steps - 2) + [True]
    assert r.records[-1].forced and not any(rec.forced for rec in r.records[:-1])
    sig = O.sigmas(cfg.steps)
    x = lat.astype(np.float64)
    si = O.step_inputs(cfg, w, x, 1000.0 * sig[0])
    R0 = O.block_stack(cfg, w, si.h_in, si.mods, None) - si.h_in
    for i in range(cfg.steps):
        si = O.step_inputs(cfg, w, x, 1000.0 * sig[i])
        h = O.block_stack(cfg, w, si.h_in, si.mods, None) if i == cfg.steps - 1 else si.h_in + R0
        x = x + (sig[i + 1] - sig[i]) * O.final_layer(cfg, w, h, si.final_mod)
    np.testing.assert_allclose(r.latent, x, rtol=0, atol=1e-12)


def test_loop_signals_are_consecutive_temni_drifts(toy):
    cfg, w, lat = toy
    r = O.denoise_loop(cfg, w, lat, None)
    # recompute the TEMNI sequence along the oracle's own trajectory via forced replay
    forced = [rec.computed for rec in r.records]
    r2 = O.denoise_loop(cfg, w, lat, None, forced=[None] + forced[1:])
    assert [x.computed for x in r2.records] == forced
    np.testing.assert_allclose(r2.latent, r.latent, rtol=0, atol=0)
    assert all(rec.signal > 0 for rec in r.records[1:])


def test_teacache_signals_follow_consecutive_steps_through_skips(toy):
    """TeaCache's signal compares the TEMNIs of consecutive steps, whether the
    earlier one was computed or reused (Sec. 2).  With every non-warmup step
    reused the trajectory can be replayed by hand (final layer on
    H_in + R_0), and each recorded s_t must equal rel_l1(TEMNI_{t-1},
    TEMNI_t) along it; comparing against the last computed step's TEMNI
    instead fails from step 2 on."""
    cfg, w, lat = toy
    r = O.denoise_loop(cfg, w, lat, None, tau_low=1e9, tau_high=1e9)
    assert r.computed == [True] + [False] * (cfg.steps - 1)
    sig = O.sigmas(cfg.steps)
    x = lat.astype(np.float64)
    si = O.step_inputs(cfg, w, x, 1000.0 * sig[0])
    R0 = O.block_stack(cfg, w, si.h_in, si.mods, None) - si.h_in
    temni = []
    for i in range(cfg.steps):
        si = O.step_inputs(cfg, w, x, 1000.0 * sig[i])
        temni.append(O.block0_temni(cfg, w, si.h_in, si.temb))
        x = x + (sig[i + 1] - sig[i]) * O.final_layer(cfg, w, si.h_in + R0, si.final_mod)
    for i in range(1, cfg.steps):
        assert r.records[i].signal == pytest.approx(O.rel_l1(temni[i - 1], temni[i]), rel=1e-12)


def test_easycache_state_through_a_skip_then_compute():
    """EasyCache's rate k and its previous input and output are those of the
    step before, whether that step was computed or reused (R9: k = output
    change over input change between steps c-1 and c, refreshed on every
    computed step).  Forced decisions compute, compute (warm-up), skip,
    compute, skip, skip; the hand replay below keeps x_{t-1}, v_{t-1} of the
    previous step and refreshes k at step 3 against the reused step 2."""
    cfg = S.get_config("toy", steps=6, method="easycache", tau_low=0.02, tau_high=0.04)
    w = S.model_weights(cfg, 3)
    lat = S.latent(cfg, 3)
    forced = [None, None, False, True, False, False]
    r = O.denoise_loop(cfg, w, lat, None, forced=forced)
    assert r.computed == [True, True, False, True, False, False]
    sig = O.sigmas(cfg.steps)
    x = lat.astype(np.float64)
    xs, vs, s_hand = [], [], {}
    k = x_c = v_c = None
    for i in range(cfg.steps):
        if i >= 2:
            dx = np.abs(x - xs[-1]).mean()
            s_hand[i] = k * dx / np.abs(vs[-1]).mean()
        if r.computed[i]:
            v = O.denoiser(cfg, w, x, 1000.0 * sig[i], None)
            if i >= 1:
                k = np.abs(v - vs[-1]).mean() / np.abs(x - xs[-1]).mean()
            x_c, v_c = x, v
        else:
            v = x + (v_c - x_c)
        xs.append(x)
        vs.append(v)
        x = x + (sig[i + 1] - sig[i]) * v
    for i in range(2, cfg.steps):
        assert r.records[i].signal == pytest.approx(s_hand[i], rel=1e-12), i
    np.testing.assert_allclose(r.latent, x, rtol=0, atol=1e-12)


def test_easycache_rate_with_an_unchanged_input():
    """The zero-denominator reading of the drift applies to the rate too: an
    unchanged input with a changed output gives k = inf, with an unchanged
    output k = 0."""
    rng = np.random.default_rng(8)
    x, v1, v2 = rng.normal(size=(3, 5)), rng.normal(size=(3, 5)), rng.normal(size=(3, 5))
    assert math.isinf(O.easycache_rate(x, x, v1, v2))
    assert O.easycache_rate(x, x, v1, v1) == 0.0


def test_force_last_leaves_an_explicit_decision_alone(toy):
    """A decision forced for the last step wins over force_last: an explicit
    skip stays a skip."""
    cfg, w, lat = toy
    forced = [None] * (cfg.steps - 1) + [False]
    r = O.denoise_loop(cfg, w, lat, None, tau_low=-1.0, tau_high=-1.0, forced=forced, force_last=True)
    assert r.computed == [True] * (cfg.steps - 1) + [False]
    assert r.records[-1].forced


def test_easycache_affine_model_is_exact():
    """EasyCache (Sec. 2): if the model's output is its input plus a constant
    offset, k = 1 and the reuse x_t + (v_c - x_c) is exact, so any decision
    sequence yields the uncached trajectory."""
    rng = np.random.default_rng(0)
    c = rng.normal(size=(3, 4))
    x_c = rng.normal(size=(3, 4))
    x_prev = x_c - 0.1 * rng.normal(size=(3, 4))
    k = O.easycache_rate(x_c, x_prev, x_c + c, x_prev + c)
    assert k == pytest.approx(1.0, abs=1e-15)
    x_t = x_c + rng.normal(size=(3, 4))
    np.testing.assert_allclose(O.easycache_reuse(x_t, x_c, x_c + c), x_t + c, atol=1e-15)
    s = O.easycache_signal(2.0, x_t, x_c, x_c + c)
    assert s == pytest.approx(2.0 * np.abs(x_t - x_c).mean() / np.abs(x_c + c).mean())


def test_easycache_rate_of_a_steeper_affine_model():
    """A model whose output moves three times as far as its input, v = 3 x +
    c: the transformation rate is 3 (output change over input change), the
    drift estimate is 3 mean|x_t - x_{t-1}| / mean|v_{t-1}|, and a rate read
    the other way round (1/3) or with the roles of input and output swapped
    fails here."""
    rng = np.random.default_rng(5)
    c = rng.normal(size=(4, 6))
    x_prev = rng.normal(size=(4, 6))
    x_c = x_prev + 0.25 * rng.normal(size=(4, 6))
    k = O.easycache_rate(x_c, x_prev, 3.0 * x_c + c, 3.0 * x_prev + c)
    assert k == pytest.approx(3.0, rel=1e-14)
    # the same step seen backwards has the same rate
    assert O.easycache_rate(x_prev, x_c, 3.0 * x_prev + c, 3.0 * x_c + c) == pytest.approx(3.0, rel=1e-14)
    x_t = x_c + 0.5  # every element moves by 0.5: mean|x_t - x_c| = 0.5
    v_c = 3.0 * x_c + c
    assert O.easycache_signal(k, x_t, x_c, v_c) == pytest.approx(1.5 / np.abs(v_c).mean(), rel=1e-14)


def test_easycache_loop_runs_and_warms_up_two_steps():
    cfg = S.get_config("toy", steps=6, method="easycache", tau_low=0.02, tau_high=0.04)
    w = S.model_weights(cfg, 1)
    r = O.denoise_loop(cfg, w, S.latent(cfg, 1), None)
    assert r.computed[:2] == [True, True]
    assert all(np.isfinite(rec.signal) for rec in r.records[2:])


# ---------------------------------------------------------------------------
# DiCache reading (Sec. 2, "DiCache")
# ---------------------------------------------------------------------------

def test_dicache_reuse_exact_on_straight_trajectory():
    """Probe and deep part moving along one straight line with proportional
    steps: the trajectory extrapolation is exact."""
    rng = np.random.default_rng(21)
    p2, dp = rng.normal(size=(5, 7)), rng.normal(size=(5, 7))
    d2, dd = rng.normal(size=(5, 7)), rng.normal(size=(5, 7))
    p1, d1 = p2 + dp, d2 + dd
    for a in (0.5, 1.0, 2.5):
        pt = p1 + a * dp
        assert O.dicache_gamma(pt, p1, p2) == pytest.approx(a)
        np.testing.assert_allclose(O.dicache_reuse(pt, p1, p2, d1, d2), pt + d1 + a * dd, atol=1e-12)


def test_dicache_single_cached_step_reuses_deep_part():
    rng = np.random.default_rng(22)
    p, d, pt = rng.normal(size=(3, 4)), rng.normal(size=(3, 4)), rng.normal(size=(3, 4))
    assert O.dicache_gamma(pt, p, p) == 0.0
    np.testing.assert_allclose(O.dicache_reuse(pt, p, p, d, d), pt + d, atol=0)


def test_dicache_reuses_along_the_last_two_computed_steps():
    """After computed steps 0, 1 and 2 a skipped step extrapolates from the
    probe and deep parts of steps 2 (latest) and 1: the hand replay below
    keeps those two, so keeping only the latest (gamma = 0) or the first
    computed step fails."""
    cfg = S.get_config("toy", steps=5)
    w = S.model_weights(cfg, 12)
    lat = S.latent(cfg, 12)
    forced = [None, True, True, False, False]
    r = O.denoise_loop(cfg, w, lat, None, method="dicache", probe_blocks=1, forced=forced)
    assert r.computed == [True, True, True, False, False]
    sig = O.sigmas(cfg.steps)
    x = lat.astype(np.float64)
    hist = []  # (probe, deep part) of computed steps, latest last
    for i in range(cfg.steps):
        si = O.step_inputs(cfg, w, x, 1000.0 * sig[i])
        probe = O.run_block_range(cfg, w, si.h_in, si.mods, None, 0, 1)
        if r.computed[i]:
            h = O.run_block_range(cfg, w, probe, si.mods, None, 1, cfg.n_blocks)
            hist.append((probe, h - probe))
        else:
            (p2, d2), (p1, d1) = hist[-2], hist[-1]
            g = np.abs(probe - p1).sum() / np.abs(p1 - p2).sum()
            h = probe + d1 + g * (d1 - d2)
        x = x + (sig[i + 1] - sig[i]) * O.final_layer(cfg, w, h, si.final_mod)
    np.testing.assert_allclose(r.latent, x, rtol=0, atol=1e-12)


def test_dicache_full_depth_probe_is_uncached():
    """A probe as deep as the whole stack leaves no deep part (D = 0), so every
    reuse reproduces the model output exactly, whatever the decisions."""
    cfg = S.get_config("toy", steps=6)
    w = S.model_weights(cfg, 8)
    lat = S.latent(cfg, 8)
    r = O.denoise_loop(cfg, w, lat, None, method="dicache", probe_blocks=cfg.n_blocks, tau_low=1e9, tau_high=1e9)
    assert r.computed == [True] + [False] * (cfg.steps - 1)
    np.testing.assert_allclose(r.latent, _plain_sampler(cfg, w, lat, cfg.steps), atol=1e-12)


def test_dicache_negative_threshold_is_uncached():
    cfg = S.get_config("toy", steps=5)
    w = S.model_weights(cfg, 9)
    lat = S.latent(cfg, 9)
    r = O.denoise_loop(cfg, w, lat, None, method="dicache", tau_low=-1.0, tau_high=-1.0)
    assert all(r.computed)
    np.testing.assert_allclose(r.latent, _plain_sampler(cfg, w, lat, cfg.steps), atol=1e-12)


# ---------------------------------------------------------------------------
# Signal rescaling hook (TeaCache-style polynomial; identity by default)
# ---------------------------------------------------------------------------

def test_rescale_polynomial_closed_forms():
    assert O.rescale_signal(0.3) == 0.3 and O.rescale_signal(0.3, []) == 0.3
    assert O.rescale_signal(0.3, [0.0, 2.0]) == 0.6
    assert O.rescale_signal(0.5, [1.0, 0.0, 4.0]) == pytest.approx(2.0)
    assert O.rescale_signal(2.0, [0.5]) == 0.5


@pytest.mark.parametrize("method", ["teacache", "dicache"])
def test_scaled_signal_with_scaled_thresholds_is_unchanged(method):
    """Doubling the signal, both thresholds and delta leaves every comparison
    of Algorithm 1 unchanged (doubling is exact in floating point)."""
    cfg = S.get_config("toy", steps=8)
    w = S.model_weights(cfg, 10)
    lat = S.latent(cfg, 10)
    a = O.denoise_loop(cfg, w, lat, None, method=method, delta=0.005)
    b = O.denoise_loop(cfg, w, lat, None, method=method, delta=0.01, tau_low=2 * cfg.tau_low,
                       tau_high=2 * cfg.tau_high, signal_poly=[0.0, 2.0])
    assert a.computed == b.computed and 0 < sum(a.computed) < cfg.steps
    np.testing.assert_array_equal(a.latent, b.latent)


def test_constant_polynomial_fixes_the_schedule():
    cfg = S.get_config("toy", steps=6)
    w = S.model_weights(cfg, 11)
    lat = S.latent(cfg, 11)
    assert all(O.denoise_loop(cfg, w, lat, None, signal_poly=[1.0]).computed)
    assert O.denoise_loop(cfg, w, lat, None, signal_poly=[0.0]).computed == [True] + [False] * 5


# ---------------------------------------------------------------------------
# Fixed threshold schedule (the transition-point experiment of Sec. 3.2)
# ---------------------------------------------------------------------------

def test_schedule_worked_example():
    """Worked by hand.  Signals 0.25 after one warmup step, delta = -1 (the
    rule alone would always pick tau_low), schedule 0.4 before step 4 and 0.8
    from step 4 on.  Sigma: 0.25 skip; 0.5 > 0.4 compute; 0.25 skip;
    0.5 <= 0.8 skip; 0.75 skip; 1.0 > 0.8 compute."""
    s = [0.0] + [0.25] * 6
    sched = [0.4] * 4 + [0.8] * 3
    d = O.controller_decisions(s, 1, 0.4, 0.8, -1.0, tau_schedule=sched)
    assert d == [True, False, True, False, False, False, True]
    ctl = O.AcidController(0.4, 0.8, -1.0)
    taus = [ctl.step(x, tau_fixed=t)[1] for x, t in zip(s[1:], sched[1:])]
    assert taus == sched[1:]


@pytest.mark.parametrize("seed", range(20))
def test_nan_schedule_is_algorithm1_and_constant_schedule_is_fixed_tau(seed):
    rng = np.random.default_rng(300 + seed)
    s = _random_signals(rng, 50)
    tl, th = sorted(rng.uniform(0.02, 0.4, size=2))
    delta = rng.uniform(0.0, 0.05)
    assert O.controller_decisions(s, 1, tl, th, delta, tau_schedule=[math.nan] * 50) == \
        O.controller_decisions(s, 1, tl, th, delta)
    tau = rng.uniform(0.02, 0.4)
    assert O.controller_decisions(s, 1, tl, th, delta, tau_schedule=[tau] * 50) == _fixed_tau(s, 1, tau)


@pytest.mark.parametrize("seed", range(20))
def test_transition_schedule_prefix_and_count(seed):
    """Low until step k, high after: the controller is causal, so steps before
    k decide as fixed tau_low does; the thresholds lie pointwise between the
    two fixed ones, so the compute count does too (same greedy argument as
    test_compute_count_between_fixed_thresholds)."""
    rng = np.random.default_rng(400 + seed)
    n = 50
    s = _random_signals(rng, n)
    tl, th = sorted(rng.uniform(0.02, 0.4, size=2))
    k = int(rng.integers(1, n))
    d = O.controller_decisions(s, 1, tl, th, 0.01, tau_schedule=[tl] * k + [th] * (n - k))
    lo = _fixed_tau(s, 1, tl)
    assert d[:k] == lo[:k]
    assert sum(_fixed_tau(s, 1, th)) <= sum(d) <= sum(lo)


def test_loop_schedule_of_low_threshold_is_fixed_low(toy):
    cfg, w, lat = toy
    a = O.denoise_loop(cfg, w, lat, None, tau_schedule=[cfg.tau_low] * cfg.steps)
    b = O.denoise_loop(cfg, w, lat, None, tau_high=cfg.tau_low)
    assert a.computed == b.computed
    np.testing.assert_array_equal(a.latent, b.latent)
