"""GPU parity of the step loop (acid_denoise_loop / acid_denoise_step through
the C ABI) against the oracle's Algorithm 1 loop.

* fp32 toy workload (2 blocks, d=256, 10 Euler steps, TeaCache signal,
  tau_low=0.05, tau_high=0.2): whole loop against the oracle; decisions
  identical except at ambiguous steps (accumulated drift within 1e-3
  relative of the threshold, or |s_t - s_prev| within 1e-3 of delta), where
  the oracle is re-run with the GPU's decision forced.
* EasyCache variant of the toy loop, same protocol.
* bf16 small Wan-shaped loop: teacher-forced signal check (the oracle
  recomputes s_t from the GPU's own latents, within 1e-3) and controller
  replay (the oracle controller fed the GPU's signals takes the same
  decisions).
"""

import math

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


def _ambiguous(rec_sigma, rec_tau, ds, delta):
    if rec_tau != rec_tau:  # warmup
        return False
    if abs(rec_sigma - rec_tau) <= 1e-3 * max(abs(rec_tau), 1e-12):
        return True
    return ds == ds and abs(ds - delta) <= 1e-3 * max(abs(delta), 1e-6)


def _compare_loop(acid, cfg, w, lat, text=None, **kw):
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg, **kw)
    tl = torch.from_numpy(lat).to(DEV)
    tt = None if text is None else torch.from_numpy(text).to(DEV, model.wdtype)
    logs = acid.acid_denoise_loop(model, c, tl, tt)
    acid.check_device_error()
    gpu_dec = [bool(l["computed"]) for l in logs]
    okw = {k: v for k, v in kw.items()
           if k in ("tau_low", "tau_high", "delta", "method", "n_steps", "probe_blocks", "signal_poly",
                     "tau_schedule")}
    ref = O.denoise_loop(cfg, w, lat, text, **okw)
    forced = [None] * len(gpu_dec)
    for i in range(len(gpu_dec)):
        rec = ref.records[i]
        if rec.computed != gpu_dec[i]:
            assert _ambiguous(rec.sigma, rec.tau, rec.dsignal, c.delta), (i, rec, logs[i])
            forced[i] = gpu_dec[i]
            ref = O.denoise_loop(cfg, w, lat, text, forced=forced, **okw)
    assert [r.computed for r in ref.records] == gpu_dec
    for l, r in zip(logs, ref.records):
        if not r.warmup:
            assert abs(l["signal"] - r.signal) <= 1e-3 * abs(r.signal) + 1e-12, (l, r)
    return tl.cpu().numpy(), ref, logs


def test_toy_loop_teacache(acid):
    cfg = S.get_config("toy")
    w = S.model_weights(cfg, 0)
    lat = S.latent(cfg, 0)
    got, ref, logs = _compare_loop(acid, cfg, w, lat)
    err = np.abs(got - ref.latent).max() / np.abs(ref.latent).max()
    assert err <= 1e-4, err
    assert 0 < sum(ref.computed) < cfg.steps  # the workload exercises both branches


@pytest.mark.parametrize("tau", [(-1.0, -1.0), (1e9, 1e9), (0.05, 0.05)])
def test_toy_loop_threshold_extremes(acid, tau):
    cfg = S.get_config("toy", steps=6)
    w = S.model_weights(cfg, 1)
    lat = S.latent(cfg, 1)
    got, ref, _ = _compare_loop(acid, cfg, w, lat, tau_low=tau[0], tau_high=tau[1])
    assert np.abs(got - ref.latent).max() <= 1e-4 * np.abs(ref.latent).max()


def test_toy_loop_easycache(acid):
    cfg = S.get_config("toy", method="easycache", tau_low=0.02, tau_high=0.04, steps=10)
    w = S.model_weights(cfg, 2)
    lat = S.latent(cfg, 2)
    got, ref, _ = _compare_loop(acid, cfg, w, lat, method="easycache")
    assert np.abs(got - ref.latent).max() <= 1e-4 * np.abs(ref.latent).max()


@pytest.mark.parametrize("probe_blocks,tau", [(1, (0.05, 0.2)), (1, (0.02, 0.04)), (2, (1e9, 1e9))])
def test_toy_loop_dicache(acid, probe_blocks, tau):
    """DiCache (probe-feature drift, trajectory reuse) against the oracle; a
    probe as deep as the stack makes every reuse exact."""
    cfg = S.get_config("toy", steps=10)
    w = S.model_weights(cfg, 12)
    lat = S.latent(cfg, 12)
    got, ref, _ = _compare_loop(acid, cfg, w, lat, method="dicache", probe_blocks=probe_blocks, tau_low=tau[0],
                                tau_high=tau[1])
    assert np.abs(got - ref.latent).max() <= 1e-4 * np.abs(ref.latent).max()
    if tau[0] < 1:
        assert 0 < sum(ref.computed) < cfg.steps


@pytest.mark.parametrize("method", ["teacache", "easycache"])
def test_toy_loop_rescaled_signal(acid, method):
    """TeaCache-style polynomial rescaling of the raw signal before Algorithm 1."""
    over = dict(method="easycache", tau_low=0.02, tau_high=0.04) if method == "easycache" else {}
    cfg = S.get_config("toy", **over)
    w = S.model_weights(cfg, 13)
    lat = S.latent(cfg, 13)
    got, ref, logs = _compare_loop(acid, cfg, w, lat, method=method, signal_poly=[0.002, 1.5, 4.0])
    assert np.abs(got - ref.latent).max() <= 1e-4 * np.abs(ref.latent).max()


@pytest.mark.parametrize("k", [1, 4, 8])
def test_toy_loop_transition_schedule(acid, k):
    """Fixed low-to-high threshold schedule switching at step k (Sec. 3.2)."""
    cfg = S.get_config("toy")
    w = S.model_weights(cfg, 15)
    lat = S.latent(cfg, 15)
    sched = [cfg.tau_low] * k + [cfg.tau_high] * (cfg.steps - k)
    got, ref, logs = _compare_loop(acid, cfg, w, lat, tau_schedule=sched)
    assert np.abs(got - ref.latent).max() <= 1e-4 * np.abs(ref.latent).max()
    assert [l["tau"] for l in logs[cfg.warmup:]] == sched[cfg.warmup:]


@pytest.mark.parametrize("method", ["teacache", "easycache", "dicache"])
def test_checkpoint_resume_is_exact(acid, method):
    """A generation stopped after k steps, checkpointed (controller struct and
    loop workspace), dropped and restored into a fresh workspace continues bit
    for bit like an uninterrupted one."""
    over = dict(method="easycache", tau_low=0.02, tau_high=0.04) if method == "easycache" else {}
    cfg = S.get_config("toy", steps=10, **over)
    w = S.model_weights(cfg, 17)
    lat = S.latent(cfg, 17)
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg, method=method)
    ref = torch.from_numpy(lat).to(DEV)
    full = acid.Loop(model, c, None, DEV)
    ref_logs = [acid.log_to_dict(full.step(ref)) for _ in range(cfg.steps)]
    x = torch.from_numpy(lat).to(DEV)
    part = acid.Loop(model, c, None, DEV)
    logs = [acid.log_to_dict(part.step(x)) for _ in range(6)]
    ckpt = part.checkpoint()
    x_saved = x.clone()
    del part
    torch.cuda.synchronize()
    resumed = acid.Loop.restore(model, c, ckpt, DEV)
    logs += [acid.log_to_dict(resumed.step(x_saved)) for _ in range(cfg.steps - 6)]
    acid.check_device_error()
    np.testing.assert_array_equal(x_saved.cpu().numpy(), ref.cpu().numpy())
    for a, b in zip(logs, ref_logs):
        assert a["computed"] == b["computed"]
        assert (a["signal"] != a["signal"] and b["signal"] != b["signal"]) or a["signal"] == b["signal"]
    assert 0 < sum(l["computed"] for l in logs) < cfg.steps


def test_toy_loop_forced_decisions(acid):
    cfg = S.get_config("toy", steps=6)
    w = S.model_weights(cfg, 3)
    lat = S.latent(cfg, 3)
    forced = [None, False, True, False, None, True]
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg, forced=forced)
    tl = torch.from_numpy(lat).to(DEV)
    logs = acid.acid_denoise_loop(model, c, tl)
    ref = O.denoise_loop(cfg, w, lat, None, forced=forced)
    assert [bool(l["computed"]) for l in logs] == ref.computed
    assert np.abs(tl.cpu().numpy() - ref.latent).max() <= 1e-4 * np.abs(ref.latent).max()


@pytest.mark.parametrize("kind", ["wan", "cog", "hv"])
def test_bf16_loop_teacher_forced_signal_and_replay(acid, kind):
    over = dict(d=256, heads=2, ffn=512, latent_f=3, latent_h=16, latent_w=22, steps=8)
    if kind == "wan":
        cfg = S.get_config("wan", n_blocks=2, n_text=40, d_text=256, **over)
    elif kind == "cog":
        over["heads"] = 4
        cfg = S.get_config("cog", n_blocks=2, n_text=30, d_text=256, **over)
    else:
        cfg = S.get_config("hv", n_blocks=1, n_single=1, n_text=30, d_text=256, **over)
    w = S.model_weights(cfg, 4)
    lat = S.latent(cfg, 4)
    text = S.text(cfg, 4)
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg)
    tt = torch.from_numpy(text).to(DEV, torch.bfloat16)
    loop = acid.Loop(model, c, tt, DEV)
    tl = torch.from_numpy(lat).to(DEV)
    xs, logs = [], []
    for i in range(cfg.steps):
        xs.append(tl.cpu().numpy().astype(np.float64))
        logs.append(acid.log_to_dict(loop.step(tl)))
    acid.check_device_error()
    sig = O.sigmas(cfg.steps)
    W = cfg.warmup
    # teacher-forced signal
    if cfg.method == "teacache":
        temni = [O.block0_temni(cfg, w, O.step_inputs(cfg, w, x, 1000 * sig[i], with_blocks=False).h_in,
                                O.time_embedding(1000 * sig[i], w, cfg.time_freq_dim)) for i, x in enumerate(xs)]
        for i in range(W, cfg.steps):
            ref = O.rel_l1(temni[i - 1], temni[i])
            assert abs(logs[i]["signal"] - ref) <= 1e-3 * ref, (i, logs[i]["signal"], ref)
    # controller replay
    gpu_s = [l["signal"] if i >= W else 0.0 for i, l in enumerate(logs)]
    dec = O.controller_decisions(gpu_s, W, cfg.tau_low, cfg.tau_high, cfg.delta)
    assert dec == [bool(l["computed"]) for l in logs]
    assert all(math.isfinite(l["signal"]) for l in logs[W:])
    assert np.isfinite(tl.cpu().numpy()).all()


@pytest.mark.parametrize("d", [1024, 1152, 1920, 2048, 2560])
def test_teacache_signal_across_row_widths(acid, d):
    """The fused TEMNI + drift kernel keeps the row in registers sized to the
    width (up to 1024, 1536, 2048 or 3072 columns; up to 1536 it also loads
    the previous TEMNI row with the input).  The toy, Wan and HunyuanVideo
    loops cover widths 256, 1536 and 3072.  Here the edges of the ranges and
    the CogVideoX width 1920 (its last vector half filled) run TeaCache, and
    the loop's signal matches the oracle's relative L1 of consecutive TEMNIs,
    teacher-forced on the GPU's own step inputs."""
    cfg = S.get_config("wan", d=d, heads=d // 128, ffn=512, n_blocks=1, n_text=40, d_text=256, latent_f=3,
                       latent_h=16, latent_w=22, steps=4)
    w = S.model_weights(cfg, 6)
    lat = S.latent(cfg, 6)
    text = S.text(cfg, 6)
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg)
    loop = acid.Loop(model, c, torch.from_numpy(text).to(DEV, torch.bfloat16), DEV)
    tl = torch.from_numpy(lat).to(DEV)
    xs, logs = [], []
    for i in range(cfg.steps):
        xs.append(tl.cpu().numpy().astype(np.float64))
        logs.append(acid.log_to_dict(loop.step(tl)))
    acid.check_device_error()
    sig = O.sigmas(cfg.steps)
    temni = [O.block0_temni(cfg, w, O.step_inputs(cfg, w, x, 1000 * sig[i], with_blocks=False).h_in,
                            O.time_embedding(1000 * sig[i], w, cfg.time_freq_dim)) for i, x in enumerate(xs)]
    for i in range(cfg.warmup, cfg.steps):
        ref = O.rel_l1(temni[i - 1], temni[i])
        assert abs(logs[i]["signal"] - ref) <= 1e-3 * ref, (d, i, logs[i]["signal"], ref)


def test_bf16_patch_embedding_keeps_fp32_tokens(acid):
    """bf16 models form the patch embedding H_in on tensor cores from the fp32
    tokens split into bf16 hi and lo parts (hi + lo = x to within 2^-17 |x|).
    The first steps of a 1000-step schedule change the latent by about 0.1%
    per step, so the TeaCache signal is near 2e-3; rounding the tokens to bf16
    alone would move it by about 3% there, the hi + lo split by about 2e-7
    (both computed with the oracle).  The signal must match the oracle's
    (fp32 tokens, fp64 arithmetic) to 1e-4 relative."""
    cfg = S.get_config("wan", d=256, heads=2, ffn=512, n_blocks=1, n_text=40, d_text=256, latent_f=5,
                       latent_h=32, latent_w=46, steps=1000)
    w = S.model_weights(cfg, 8)
    lat = S.latent(cfg, 8)
    text = S.text(cfg, 8)
    model = acid.DeviceModel(cfg, w, DEV)
    c, keep = acid.loop_cfg(cfg)
    loop = acid.Loop(model, c, torch.from_numpy(text).to(DEV, torch.bfloat16), DEV)
    tl = torch.from_numpy(lat).to(DEV)
    xs, logs = [], []
    for i in range(4):
        xs.append(tl.cpu().numpy().astype(np.float64))
        logs.append(acid.log_to_dict(loop.step(tl)))
    acid.check_device_error()
    sig = O.sigmas(cfg.steps)
    temni = [O.block0_temni(cfg, w, O.step_inputs(cfg, w, x, 1000 * sig[i], with_blocks=False).h_in,
                            O.time_embedding(1000 * sig[i], w, cfg.time_freq_dim)) for i, x in enumerate(xs)]
    for i in range(cfg.warmup, len(xs)):
        ref = O.rel_l1(temni[i - 1], temni[i])
        assert ref < 1e-2, ref
        assert abs(logs[i]["signal"] - ref) <= 1e-4 * ref, (i, logs[i]["signal"], ref)
