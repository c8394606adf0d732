"""The threshold sweep on the GPU (toy workload): every run's decisions must
be what the oracle's Algorithm 1 takes on that run's own logged signals, and
the every-step run must compute every step."""

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
