"""acid_denoise_loop_graph: the whole generation as one CUDA graph with the
drift signal and Algorithm 1's decision taken on the device.  Its decisions
and latents must equal the host-driven loop's (same kernels, same order) and
the oracle's."""

import numpy as np
import pytest

import acid_synth as S
import oracle as O

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
DEV = "cuda"


@pytest.fixture(scope="module")
def acid():
    import __graft_entry__ as g

    g.build()
    from paper_2607_12358_gb300 import acid as a

    return a


def _both(acid, cfg, w, lat, text=None, **kw):
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg, **kw)
    tt = None if text is None else torch.from_numpy(text).to(DEV, model.wdtype)
    a = torch.from_numpy(lat).to(DEV)
    b = torch.from_numpy(lat).to(DEV)
    la = acid.acid_denoise_loop(model, c, a, tt)
    lb = acid.acid_denoise_loop(model, c, b, tt, graph=True)
    acid.check_device_error()
    return a.cpu().numpy(), b.cpu().numpy(), la, lb


def _same_logs(la, lb):
    for x, y in zip(la, lb):
        assert x["computed"] == y["computed"] and x["warmup"] == y["warmup"] and x["forced"] == y["forced"]
        for k in ("signal", "dsignal", "tau", "sigma", "t"):
            assert (np.isnan(x[k]) and np.isnan(y[k])) or x[k] == y[k], (k, x, y)


@pytest.mark.parametrize("method", ["teacache", "easycache", "dicache"])
def test_toy_graph_equals_host_loop_and_oracle(acid, method):
    over = dict(method="easycache", tau_low=0.02, tau_high=0.04) if method == "easycache" else {}
    if method == "dicache":
        over = dict(method="dicache")
    cfg = S.get_config("toy", **over)
    w = S.model_weights(cfg, 5)
    lat = S.latent(cfg, 5)
    host, graph, la, lb = _both(acid, cfg, w, lat, method=method)
    _same_logs(la, lb)
    np.testing.assert_array_equal(graph, host)
    ref = O.denoise_loop(cfg, w, lat, None, method=method)
    assert [bool(x["computed"]) for x in lb] == ref.computed
    assert np.abs(graph - ref.latent).max() <= 1e-4 * np.abs(ref.latent).max()
    assert 0 < sum(ref.computed) < cfg.steps


def test_toy_graph_rescaled_signal(acid):
    cfg = S.get_config("toy")
    w = S.model_weights(cfg, 14)
    host, graph, la, lb = _both(acid, cfg, w, S.latent(cfg, 14), signal_poly=[0.002, 1.5, 4.0])
    _same_logs(la, lb)
    np.testing.assert_array_equal(graph, host)


def test_toy_graph_transition_schedule(acid):
    cfg = S.get_config("toy")
    w = S.model_weights(cfg, 16)
    sched = [cfg.tau_low] * 5 + [float("nan")] * 2 + [cfg.tau_high] * 3
    host, graph, la, lb = _both(acid, cfg, w, S.latent(cfg, 16), tau_schedule=sched)
    _same_logs(la, lb)
    np.testing.assert_array_equal(graph, host)


def test_toy_graph_forced_and_force_last(acid):
    cfg = S.get_config("toy", steps=7)
    w = S.model_weights(cfg, 6)
    lat = S.latent(cfg, 6)
    forced = [None, False, True, None, False, None, None]
    host, graph, la, lb = _both(acid, cfg, w, lat, forced=forced, force_last=True, tau_low=1e9, tau_high=1e9)
    _same_logs(la, lb)
    np.testing.assert_array_equal(graph, host)
    assert [x["computed"] for x in lb] == [1, 0, 1, 0, 0, 0, 1]


@pytest.mark.parametrize("kind", ["wan", "cog", "hv", "hv-dicache"])
def test_bf16_graph_equals_host_loop(acid, kind):
    method = None
    if kind == "hv-dicache":
        kind, method = "hv", "dicache"
    over = dict(d=256, heads=2, ffn=512, latent_f=3, latent_h=16, latent_w=22, steps=8)
    if kind == "wan":
        cfg = S.get_config("wan", n_blocks=2, n_text=40, d_text=256, **over)
    elif kind == "cog":
        over["heads"] = 4
        cfg = S.get_config("cog", n_blocks=2, n_text=30, d_text=256, **over)
    else:
        cfg = S.get_config("hv", n_blocks=1, n_single=1, n_text=30, d_text=256, **over)
    w = S.model_weights(cfg, 7)
    kw = {} if method is None else dict(method=method, probe_blocks=1, tau_low=0.05, tau_high=0.2)
    host, graph, la, lb = _both(acid, cfg, w, S.latent(cfg, 7), S.text(cfg, 7), **kw)
    _same_logs(la, lb)
    np.testing.assert_array_equal(graph, host)


def test_graph_at_its_step_limit(acid):
    """The graph keeps its per-step tables (noise levels, forced decisions,
    thresholds, logs) for at most 1024 steps: a 1024-step generation runs as
    one graph and equals the host-driven loop bit for bit, decisions
    included; 1025 steps are refused before anything is launched."""
    from paper_2607_12358_gb300._capi import AcidError

    cfg = S.get_config("toy", steps=1024)
    w = S.model_weights(cfg, 60)
    a, b, la, lb = _both(acid, cfg, w, S.latent(cfg, 60))
    _same_logs(la, lb)
    np.testing.assert_array_equal(a, b)
    assert len(lb) == 1024 and 0 < sum(l["computed"] for l in lb) < 1024
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg, n_steps=1025)
    n0 = acid.launch_count()
    with pytest.raises(AcidError, match="at most 1024 steps"):
        acid.acid_denoise_loop(model, c, torch.from_numpy(S.latent(cfg, 60)).to(DEV), None, graph=True)
    assert acid.launch_count() == n0
