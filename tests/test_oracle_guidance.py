"""Pins for the oracle's classifier-free-guidance loop: two sampler branches
(conditional, unconditional text) with independent Algorithm 1 state and
caches, combined as v = v_u + g (v_c - v_u) before the Euler step."""

import numpy as np
import pytest

import acid_synth as S
import oracle as O


def _cfg(method="teacache", **kw):
    over = dict(n_text=12, d_text=64, steps=8)
    if method == "easycache":
        over.update(method="easycache", tau_low=0.02, tau_high=0.04)
    over.update(kw)
    return S.get_config("toy", **over)


@pytest.fixture(scope="module")
def setup():
    cfg = _cfg()
    w = S.model_weights(cfg, 30)
    return cfg, w, S.latent(cfg, 30), S.text(cfg, 30), S.text(cfg, 31)


def test_guidance_combination_closed_form():
    vc, vu = np.array([1.0, -2.0, 3.0]), np.array([0.5, 0.5, -1.0])
    np.testing.assert_array_equal(O.guided_velocity(vc, vu, 0.0), vu)
    np.testing.assert_array_equal(O.guided_velocity(vc, vu, 1.0), vc)
    np.testing.assert_array_equal(O.guided_velocity(vc, vu, 2.0), [1.5, -4.5, 7.0])


@pytest.mark.parametrize("method", ["teacache", "easycache", "dicache"])
def test_identical_texts_give_the_plain_loop(method):
    """v_c == v_u bitwise, so v = v_u + g * 0 = v_u for any g: the guided
    loop is the plain loop, with the same decisions in both branches."""
    cfg = _cfg(method)
    w = S.model_weights(cfg, 32)
    lat, text = S.latent(cfg, 32), S.text(cfg, 32)
    g = O.denoise_loop_guided(cfg, w, lat, text, text, 5.0, method=method)
    p = O.denoise_loop(cfg, w, lat, text, method=method)
    np.testing.assert_array_equal(g.latent, p.latent)
    assert [r.computed for r in g.cond] == [r.computed for r in g.uncond] == p.computed


@pytest.mark.parametrize("scale,which", [(1.0, "cond"), (0.0, "uncond")])
def test_unit_and_zero_scale_follow_one_branch(setup, scale, which):
    """g = 1 gives v_c, g = 0 gives v_u (up to one rounding of the
    combination), so the latent follows the plain loop of that branch."""
    cfg, w, lat, tc, tu = setup
    g = O.denoise_loop_guided(cfg, w, lat, tc, tu, scale)
    p = O.denoise_loop(cfg, w, lat, tc if which == "cond" else tu)
    np.testing.assert_allclose(g.latent, p.latent, rtol=1e-12, atol=1e-12)
    assert [r.computed for r in getattr(g, which)] == p.computed


def test_teacache_branches_decide_alike(setup):
    """TEMNI is block 0's modulated input of the video tokens, which the
    text does not enter, so both TeaCache branches see the same s_t and take
    the same decisions."""
    cfg, w, lat, tc, tu = setup
    g = O.denoise_loop_guided(cfg, w, lat, tc, tu, 4.0)
    assert [r.signal for r in g.cond][1:] == [r.signal for r in g.uncond][1:]
    assert [r.computed for r in g.cond] == [r.computed for r in g.uncond]
    assert 0 < sum(r.computed for r in g.cond) < cfg.steps


def test_branch_state_is_independent(setup):
    """Forcing the unconditional branch to compute on every step does not
    touch the conditional branch's controller: at g = 1 its records equal the
    plain conditional loop's."""
    cfg, w, lat, tc, tu = setup
    g = O.denoise_loop_guided(cfg, w, lat, tc, tu, 1.0, forced_uncond=[True] * cfg.steps)
    p = O.denoise_loop(cfg, w, lat, tc)
    assert all(r.computed for r in g.uncond)
    assert [r.computed for r in g.cond] == p.computed
    for a, b in zip(g.cond[1:], p.records[1:]):
        assert a.sigma == pytest.approx(b.sigma, rel=1e-9)


def test_easycache_branches_can_decide_differently():
    """EasyCache's signal divides by the branch's own |v_{t-1}|, so the two
    branches' signals differ once the texts do."""
    cfg = _cfg("easycache", steps=10)
    w = S.model_weights(cfg, 33)
    g = O.denoise_loop_guided(cfg, w, S.latent(cfg, 33), S.text(cfg, 33), S.text(cfg, 34), 4.0)
    sc = [r.signal for r in g.cond][cfg.warmup:]
    su = [r.signal for r in g.uncond][cfg.warmup:]
    assert all(a != b for a, b in zip(sc, su))
