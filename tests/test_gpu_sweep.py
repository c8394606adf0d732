"""The threshold sweep on the GPU (toy workload, and small bf16 CogVideoX-
and HunyuanVideo-shaped joint models): every run's decisions must be what
the oracle's Algorithm 1 takes on that run's own logged signals, and the
every-step run must compute every step."""

import math

import numpy as np
import pytest

import acid_synth as S
import oracle as O

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def acid():
    import __graft_entry__ as g

    g.build()
    from paper_2607_12358_gb300 import acid as a

    return a


@pytest.mark.parametrize("graph", [True, False])
def test_toy_sweep_decisions_replay(acid, graph):
    from paper_2607_12358_gb300 import sweep as W

    cfg = S.get_config("toy", steps=12)
    w = S.model_weights(cfg, 20)
    res = W.sweep(cfg, w, S.latent(cfg, 20), transitions=[2, 6], deltas=[-1.0, 0.01, 1e9], graph=graph)
    assert res["full"]["computed"] == 12 and res["full"]["rel_l2"] == 0.0
    tl, th = cfg.tau_low, cfg.tau_high

    def replay(run, lo, hi, delta, sched=None):
        s = [0.0 if math.isnan(x) else x for x in run["signal"]]
        return [int(d) for d in O.controller_decisions(s, cfg.warmup, lo, hi, delta, tau_schedule=sched)]

    assert res["fixed_low"]["decisions"] == replay(res["fixed_low"], tl, tl, cfg.delta)
    assert res["fixed_high"]["decisions"] == replay(res["fixed_high"], th, th, cfg.delta)
    for r in res["runs"]:
        if r["kind"] == "transition":
            sched = W.transition_schedule(12, r["k"], tl, th)
            assert r["decisions"] == replay(r, tl, th, cfg.delta, sched)
        else:
            assert r["decisions"] == replay(r, tl, th, r["delta"])
        assert np.isfinite(r["rel_l2"])
    by = {r["name"]: r for r in res["runs"]}
    # delta < 0 never selects tau_high: the same generation as fixed tau_low
    assert by["adaptive delta=-1.0"]["decisions"] == res["fixed_low"]["decisions"]
    assert by["adaptive delta=-1.0"]["rel_l2"] == res["fixed_low"]["rel_l2"]


@pytest.mark.parametrize("workload", ["cog", "hv"])
def test_joint_model_sweep_decisions_replay(acid, workload):
    """Small bf16 joint [text; video] models, graph-launched: CogVideoX-shaped
    (EasyCache, head dim 64) and HunyuanVideo-shaped (TeaCache, one dual- and
    one single-stream block).  Thresholds on the random-weight signal's scale
    so that runs both skip and compute."""
    from paper_2607_12358_gb300 import sweep as W

    small = dict(d=256, ffn=512, n_blocks=1, latent_f=3, latent_h=16, latent_w=22, n_text=40, d_text=256,
                 steps=10)
    if workload == "cog":
        cfg = S.get_config("cog", heads=4, **small)
        tl, th, deltas = 0.6, 2.0, [0.01, 0.2]
    else:
        cfg = S.get_config("hv", heads=2, n_single=1, **small)
        tl, th, deltas = 0.05, 0.2, [0.002, 0.05]
    w = S.model_weights(cfg, 21)
    res = W.sweep(cfg, w, S.latent(cfg, 21), S.text(cfg, 21), tau_low=tl, tau_high=th, transitions=[4],
                  deltas=deltas, graph=True)
    assert res["full"]["computed"] == cfg.steps and res["full"]["rel_l2"] == 0.0

    def replay(run, lo, hi, delta, sched=None):
        s = [0.0 if math.isnan(x) else x for x in run["signal"]]
        return [int(d) for d in O.controller_decisions(s, cfg.warmup, lo, hi, delta, tau_schedule=sched)]

    assert res["fixed_low"]["decisions"] == replay(res["fixed_low"], tl, tl, cfg.delta)
    assert res["fixed_high"]["decisions"] == replay(res["fixed_high"], th, th, cfg.delta)
    for r in res["runs"]:
        if r["kind"] == "transition":
            assert r["decisions"] == replay(r, tl, th, cfg.delta, W.transition_schedule(cfg.steps, r["k"], tl, th))
        else:
            assert r["decisions"] == replay(r, tl, th, r["delta"])
        assert np.isfinite(r["rel_l2"])
    computed = [r["computed"] for r in [res["fixed_low"], res["fixed_high"]] + res["runs"]]
    assert min(computed) < cfg.steps, computed  # some run skips
