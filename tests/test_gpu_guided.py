"""Classifier-free guidance through the C ABI (acid_denoise_loop_guided /
acid_guided_step): two branches with independent Algorithm 1 state and
caches against the oracle's guided loop.

* fp32 toy with text (TeaCache, EasyCache, DiCache): decisions of both
  branches identical to the oracle's except at ambiguous steps (the
  accumulated drift within 1e-3 relative of the threshold, or |s_t - s_prev|
  within 1e-3 of delta), where the oracle is re-run with the GPU's decision
  forced for that branch; latent within 1e-4 relative.
* identical texts: the guided generation is bit-identical to the plain one.
* step-wise driving equals the whole-loop call.
* bf16 small Wan shape: each branch's decisions are what the oracle
  controller takes on that branch's own logged signals.
* acid_denoise_loop_guided_graph (one CUDA graph, both decisions on the
  device) equals the host-driven guided loop bit for bit.
"""

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


def _toy(method, steps=8):
    over = dict(n_text=12, d_text=64, steps=steps)
    if method == "easycache":
        over.update(method="easycache", tau_low=0.02, tau_high=0.04)
    return S.get_config("toy", **over)


def _ambiguous(rec, delta):
    if rec.tau != rec.tau:
        return False
    if abs(rec.sigma - rec.tau) <= 1e-3 * max(abs(rec.tau), 1e-12):
        return True
    return rec.dsignal == rec.dsignal and abs(rec.dsignal - delta) <= 1e-3 * max(abs(delta), 1e-6)


def _run_gpu(acid, cfg, w, lat, tc, tu, scale, method, **kw):
    model = acid.DeviceModel(cfg, w, DEV)
    cc, kc = acid.loop_cfg(cfg, method=method, **kw)
    cu, ku = acid.loop_cfg(cfg, method=method, **kw)
    x = torch.from_numpy(lat).to(DEV)
    t_c = torch.from_numpy(tc).to(DEV, model.wdtype)
    t_u = torch.from_numpy(tu).to(DEV, model.wdtype)
    lc, lu = acid.acid_denoise_loop_guided(model, cc, cu, scale, x, t_c, t_u)
    acid.check_device_error()
    return x.cpu().numpy(), lc, lu


@pytest.mark.parametrize("method", ["teacache", "easycache", "dicache"])
def test_toy_guided_against_oracle(acid, method):
    cfg = _toy(method)
    w = S.model_weights(cfg, 40)
    lat, tc, tu = S.latent(cfg, 40), S.text(cfg, 40), S.text(cfg, 41)
    scale = 3.0
    got, lc, lu = _run_gpu(acid, cfg, w, lat, tc, tu, scale, method)
    dc = [bool(l["computed"]) for l in lc]
    du = [bool(l["computed"]) for l in lu]
    fc, fu = [None] * cfg.steps, [None] * cfg.steps
    ref = O.denoise_loop_guided(cfg, w, lat, tc, tu, scale, method=method)
    for i in range(cfg.steps):
        for recs, dec, forced in ((ref.cond, dc, fc), (ref.uncond, du, fu)):
            if recs[i].computed != dec[i]:
                assert _ambiguous(recs[i], cfg.delta), (i, recs[i])
                forced[i] = dec[i]
                ref = O.denoise_loop_guided(cfg, w, lat, tc, tu, scale, method=method, forced_cond=fc,
                                            forced_uncond=fu)
    assert [r.computed for r in ref.cond] == dc and [r.computed for r in ref.uncond] == du
    for logs, recs in ((lc, ref.cond), (lu, ref.uncond)):
        for l, r in zip(logs, recs):
            if not r.warmup:
                assert abs(l["signal"] - r.signal) <= 1e-3 * abs(r.signal) + 1e-12, (l, r)
    assert np.abs(got - ref.latent).max() <= 1e-4 * np.abs(ref.latent).max()
    if method == "teacache":
        assert dc == du  # the text does not enter TEMNI


@pytest.mark.parametrize("method", ["teacache", "easycache"])
def test_identical_texts_equal_plain_loop(acid, method):
    cfg = _toy(method)
    w = S.model_weights(cfg, 42)
    lat, tc = S.latent(cfg, 42), S.text(cfg, 42)
    got, lc, lu = _run_gpu(acid, cfg, w, lat, tc, tc, 6.0, method)
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg, method=method)
    x = torch.from_numpy(lat).to(DEV)
    logs = acid.acid_denoise_loop(model, c, x, torch.from_numpy(tc).to(DEV, model.wdtype))
    np.testing.assert_array_equal(got, x.cpu().numpy())
    assert [l["computed"] for l in lc] == [l["computed"] for l in lu] == [l["computed"] for l in logs]


def test_stepwise_equals_loop(acid):
    cfg = _toy("dicache")
    w = S.model_weights(cfg, 43)
    lat, tc, tu = S.latent(cfg, 43), S.text(cfg, 43), S.text(cfg, 44)
    got, lc, lu = _run_gpu(acid, cfg, w, lat, tc, tu, 2.5, "dicache")
    model = acid.DeviceModel(cfg, w, DEV)
    cc, kc = acid.loop_cfg(cfg, method="dicache")
    cu, ku = acid.loop_cfg(cfg, method="dicache")
    t_c = torch.from_numpy(tc).to(DEV)
    t_u = torch.from_numpy(tu).to(DEV)
    gl = acid.GuidedLoop(model, cc, cu, 2.5, t_c, t_u, DEV)
    x = torch.from_numpy(lat).to(DEV)
    for i in range(cfg.steps):
        a, b = gl.step(x)
        assert a.computed == lc[i]["computed"] and b.computed == lu[i]["computed"]
        assert a.signal == lc[i]["signal"] or (a.signal != a.signal and lc[i]["signal"] != lc[i]["signal"])
    np.testing.assert_array_equal(x.cpu().numpy(), got)


def test_guided_rejects_mismatched_branches(acid):
    cfg = _toy("teacache")
    w = S.model_weights(cfg, 45)
    model = acid.DeviceModel(cfg, w, DEV)
    cc, kc = acid.loop_cfg(cfg)
    cu, ku = acid.loop_cfg(cfg, n_steps=cfg.steps + 1)
    x = torch.from_numpy(S.latent(cfg, 45)).to(DEV)
    t = torch.from_numpy(S.text(cfg, 45)).to(DEV)
    with pytest.raises(Exception, match="same n_steps"):
        acid.acid_denoise_loop_guided(model, cc, cu, 2.0, x, t, t)


@pytest.mark.parametrize("method", ["teacache", "easycache"])
def test_bf16_guided_replay(acid, method):
    over = dict(d=256, heads=2, ffn=512, latent_f=3, latent_h=16, latent_w=22, steps=8)
    if method == "easycache":
        over.update(method="easycache", tau_low=0.02, tau_high=0.04)
    cfg = S.get_config("wan", n_blocks=2, n_text=40, d_text=256, **over)
    w = S.model_weights(cfg, 46)
    got, lc, lu = _run_gpu(acid, cfg, w, S.latent(cfg, 46), S.text(cfg, 46), S.text(cfg, 47), 5.0, method)
    W = cfg.warmup
    for logs in (lc, lu):
        s = [l["signal"] if i >= W else 0.0 for i, l in enumerate(logs)]
        assert O.controller_decisions(s, W, cfg.tau_low, cfg.tau_high, cfg.delta) == \
            [bool(l["computed"]) for l in logs]
    if method == "teacache":
        assert [l["signal"] for l in lc][W:] == [l["signal"] for l in lu][W:]
    assert np.isfinite(got).all()


def _same_logs(la, lb):
    for x, y in zip(la, lb):
        assert x["computed"] == y["computed"] and x["warmup"] == y["warmup"] and x["forced"] == y["forced"]
        for k in ("signal", "dsignal", "tau", "sigma", "t"):
            assert (x[k] != x[k] and y[k] != y[k]) or x[k] == y[k], (k, x, y)


@pytest.mark.parametrize("method", ["teacache", "easycache", "dicache"])
def test_toy_guided_graph_equals_host_loop(acid, method):
    """The graph-launched guided generation (decisions on the device) runs the
    same kernels in the same order as the host-driven one: identical logs and
    a bit-identical latent."""
    cfg = _toy(method, steps=10)
    w = S.model_weights(cfg, 48)
    lat, tc, tu = S.latent(cfg, 48), S.text(cfg, 48), S.text(cfg, 49)
    model = acid.DeviceModel(cfg, w, DEV)
    outs = []
    for graph in (False, True):
        cc, kc = acid.loop_cfg(cfg, method=method)
        cu, ku = acid.loop_cfg(cfg, method=method, forced=[None] * 7 + [True] + [None] * 2)
        x = torch.from_numpy(lat).to(DEV)
        t_c = torch.from_numpy(tc).to(DEV)
        t_u = torch.from_numpy(tu).to(DEV)
        lc, lu = acid.acid_denoise_loop_guided(model, cc, cu, 3.5, x, t_c, t_u, graph=graph)
        acid.check_device_error()
        outs.append((x.cpu().numpy(), lc, lu))
    (xa, lca, lua), (xb, lcb, lub) = outs
    _same_logs(lca, lcb)
    _same_logs(lua, lub)
    np.testing.assert_array_equal(xa, xb)
    assert lub[7]["forced"] and lub[7]["computed"]


def test_bf16_guided_graph_equals_host_loop(acid):
    over = dict(d=256, heads=2, ffn=512, latent_f=3, latent_h=16, latent_w=22, steps=8)
    cfg = S.get_config("wan", n_blocks=2, n_text=40, d_text=256, **over)
    w = S.model_weights(cfg, 50)
    model = acid.DeviceModel(cfg, w, DEV)
    t_c = torch.from_numpy(S.text(cfg, 50)).to(DEV, torch.bfloat16)
    t_u = torch.from_numpy(S.text(cfg, 51)).to(DEV, torch.bfloat16)
    outs = []
    for graph in (False, True):
        cc, kc = acid.loop_cfg(cfg)
        cu, ku = acid.loop_cfg(cfg)
        x = torch.from_numpy(S.latent(cfg, 50)).to(DEV)
        lc, lu = acid.acid_denoise_loop_guided(model, cc, cu, 5.0, x, t_c, t_u, graph=graph)
        acid.check_device_error()
        outs.append((x.cpu().numpy(), lc, lu))
    _same_logs(outs[0][1], outs[1][1])
    _same_logs(outs[0][2], outs[1][2])
    np.testing.assert_array_equal(outs[0][0], outs[1][0])
