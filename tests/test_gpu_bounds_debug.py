"""The debug build's memory-index checks (libacid_gb300_debug.so, compiled
with ACID_BOUNDS_CHECK): every hand-computed global-memory index of the
element-wise, LayerNorm, drift, patch, GEMV, GEMM-epilogue and
attention-merge kernels is checked against the extent the host passed, and
an index outside it is recorded (acid_bounds_report) instead of accessed.

The library is loaded in a child process (ACID_LIBRARY=debug), which runs
every kernel family on small, ragged shapes: partial row and column tiles,
single-SM and SM-pair GEMMs with each epilogue, head dims 64 and 128 with a
split tail, odd LayerNorm widths, ragged drift lengths, a bf16 block of each
joint kind, and loop steps of a bf16 and the fp32 model.  Each result is
compared with the oracle, and no index check may have fired.  The self-test
first shows that a check one past the end is recorded (with no access behind
it), so a silent report means the checks ran."""

import os
import subprocess
import sys
import textwrap

import pytest

pytestmark = pytest.mark.gpu
pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = textwrap.dedent(
    r"""
    import numpy as np
    import torch

    import acid_synth as S
    import oracle as O
    from paper_2607_12358_gb300 import acid

    dev = torch.device("cuda")
    rep = acid.bounds_report()
    assert rep["checked"], rep
    acid.selftest_bounds()
    rep = acid.bounds_report()
    assert (rep["site"], rep["index"], rep["extent"]) == (99, 1000, 1000), rep
    assert acid.bounds_report()["site"] == 0

    def bf(a):
        return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev, torch.bfloat16)

    def f32(a):
        return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)

    def close(got, ref, rel_l2, what):
        err = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
        assert err <= rel_l2, (what, err)

    rng = np.random.default_rng(5)
    # GEMMs: single-SM tiles (N <= 2048, K <= 2048) and SM pairs, every epilogue
    for (M, K, N) in [(333, 192, 320), (130, 2176, 2304), (257, 64, 96)]:
        a = S.round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))
        w = S.round_to_bf16((0.05 * rng.normal(size=(N, K))).astype(np.float32))
        b = rng.normal(size=N).astype(np.float32)
        g = rng.normal(size=N).astype(np.float32)
        for epi in ("bias", "gelu", "gated_res", "res"):
            for fp32 in (False, True):
                r = rng.normal(size=(M, N)).astype(np.float32)
                if not fp32:
                    r = S.round_to_bf16(r)
                has_res = epi in ("gated_res", "res")
                out = (f32(r) if fp32 else bf(r))
                acid.acid_linear_forward(bf(a), bf(w), f32(b), epilogue=epi, gate=f32(g),
                                         residual=out if has_res else None, out=out, out_fp32=fp32)
                acc = O.linear(a, w, b)
                ref = {"bias": acc, "gelu": O.gelu_tanh(acc), "gated_res": r + g * acc, "res": r + acc}[epi]
                close(out.float().cpu().numpy(), ref, 1e-2, ("linear", M, K, N, epi, fp32))
    # fp32 GEMM (FP32 pipes)
    a = rng.normal(size=(77, 96)).astype(np.float32)
    w = (0.1 * rng.normal(size=(130, 96))).astype(np.float32)
    out = acid.acid_linear_forward(f32(a), f32(w), None)
    close(out.cpu().numpy(), O.linear(a, w), 1e-5, "linear fp32")
    # attention: bf16 head dims 64 and 128 (long key ranges with the split tail
    # and short ones on persistent CTAs), fp32
    for (nq, nk, H, D) in [(1300, 1300, 2, 128), (700, 1100, 3, 64), (900, 300, 2, 128)]:
        q, k, v = (S.round_to_bf16(rng.normal(size=(n, H * D)).astype(np.float32)) for n in (nq, nk, nk))
        ws = torch.empty(acid.attention_workspace_size(D), dtype=torch.uint8, device=dev)
        out = acid.acid_attention_forward(bf(q), bf(k), bf(v), H, workspace=ws)
        ref = O.attention(q.reshape(nq, H, D), k.reshape(nk, H, D), v.reshape(nk, H, D)).reshape(nq, H * D)
        close(out.float().cpu().numpy(), ref, 1e-2, ("attention", nq, nk, H, D))
    q, k, v = (rng.normal(size=(n, 2 * 64)).astype(np.float32) for n in (50, 70, 70))
    out = acid.acid_attention_forward(f32(q), f32(k), f32(v), 2)
    ref = O.attention(q.reshape(50, 2, 64), k.reshape(70, 2, 64), v.reshape(70, 2, 64)).reshape(50, 128)
    close(out.cpu().numpy(), ref, 1e-5, "attention fp32")
    # LayerNorm-mod, odd widths and row counts, bf16 and fp32 input
    for (rows, d, fp32) in [(37, 1544, False), (5, 3072, True), (129, 264, False)]:
        x = rng.normal(size=(rows, d)).astype(np.float32)
        if not fp32:
            x = S.round_to_bf16(x)
        sh, sc = rng.normal(size=d).astype(np.float32), rng.normal(size=d).astype(np.float32)
        y = acid.acid_layernorm_mod(f32(x) if fp32 else bf(x), f32(sh), f32(sc), out_dtype=torch.float32)
        close(y.cpu().numpy(), O.modulate(O.layer_norm(x), sh, sc), 1e-4, ("layernorm", rows, d, fp32))
    # drift, cache apply, fused drift + apply, ragged lengths
    for n in (37, 4099, 100003):
        p, c = (t.reshape(-1) for t in S.micro_pair(n, 1e-2, seed=n, d=1))
        rel, _ = acid.acid_drift_signal(bf(p), bf(c))
        ref = O.rel_l1(p, c)
        assert abs(rel.item() - ref) <= 1e-3 * ref, ("drift", n)
        p, c = (t.reshape(-1) for t in S.micro_pair(n, 1e-2, seed=n, d=1, bf16=False))
        r = rng.normal(size=n).astype(np.float32)
        o = acid.acid_cache_apply(f32(c), f32(r))
        close(o.cpu().numpy(), c.astype(np.float64) + r, 1e-6, ("apply", n))
        o, rel, _ = acid.acid_drift_apply(f32(p), f32(c), f32(r))
        assert abs(rel.item() - O.rel_l1(p, c)) <= 1e-3 * O.rel_l1(p, c), ("drift apply", n)
        close(o.cpu().numpy(), c.astype(np.float64) + r, 1e-6, ("drift apply", n))
    # TEMNI drift, rows in registers (d <= 1536) and re-read from the ring (d > 1536)
    for (rows, d) in [(301, 1920), (77, 512)]:
        hp = rng.normal(size=(rows, d)).astype(np.float32)
        hc = (hp + 0.05 * rng.normal(size=(rows, d))).astype(np.float32)
        mp = (0.3 * rng.normal(size=2 * d)).astype(np.float32)
        mc = (mp + 0.01 * rng.normal(size=2 * d)).astype(np.float32)
        rel, _ = acid.acid_temni_drift(f32(hp), f32(hc), f32(mp), f32(mc))
        tp = O.modulate(O.layer_norm(hp), mp[:d], mp[d:])
        tc = O.modulate(O.layer_norm(hc), mc[:d], mc[d:])
        assert abs(rel.item() - O.rel_l1(tp, tc)) <= 1e-3 * O.rel_l1(tp, tc), ("temni", rows, d)
    # bf16 blocks: Wan (RoPE QKV, cross-attention) and the joint CogVideoX kind
    for kind in ("wan", "cog"):
        over = dict(d=256, heads=4 if kind == "cog" else 2, ffn=512, latent_f=3, latent_h=16, latent_w=22)
        cfg = S.get_config(kind, n_text=40 if kind == "wan" else 30, d_text=256, **over)
        w = S.block_weights(cfg, 0, seed=9)
        L = 0 if kind == "wan" else cfg.n_text
        x = S.hidden(cfg, cfg.n_video + L, seed=9)
        temb = S.temb_vector(cfg, seed=9)
        ctx = S.round_to_bf16(S.normal(9, (cfg.n_text, cfg.d), 1.0, "bounds", "ctx")) if kind == "wan" else None
        blk = acid.DeviceBlock.upload(w, kind, torch.bfloat16, dev)
        tx = bf(x)
        acid.acid_dit_block_forward(acid.block_desc(cfg, kind), tx, f32(temb), blk, ctx=None if ctx is None else bf(ctx))
        mod = O.block_modulation(temb, w["mod"])
        if kind == "wan":
            ref = O.wan_block(x, mod, w, cfg.grid, cfg.heads, ctx=ctx)
        else:
            ref = O.cog_block(x, mod, w, cfg.grid, cfg.heads, L)
        close(tx.float().cpu().numpy(), ref, 1e-2, ("block", kind))
    # loop steps: bf16 (tensor-core patch embedding, one-launch TEMNI drift) and fp32
    for kind, steps in (("wan", 3), ("toy", 3)):
        if kind == "wan":
            cfg = S.get_config("wan", d=256, heads=2, ffn=512, n_blocks=1, n_text=40, d_text=256, latent_f=3,
                               latent_h=16, latent_w=22, steps=8)
        else:
            cfg = S.get_config("toy", steps=8)
        wts = S.model_weights(cfg, 3)
        model = acid.DeviceModel(cfg, wts, dev)
        c, keep = acid.loop_cfg(cfg)
        text = bf(S.text(cfg, 3)) if cfg.n_text else None
        loop = acid.Loop(model, c, text, dev)
        lat = f32(S.latent(cfg, 3))
        xs, logs = [], []
        for i in range(steps):
            xs.append(lat.cpu().numpy().astype(np.float64))
            logs.append(acid.log_to_dict(loop.step(lat)))
        sig = O.sigmas(cfg.steps)
        tem = [O.block0_temni(cfg, wts, O.step_inputs(cfg, wts, x, 1000 * sig[i], with_blocks=False).h_in,
                              O.time_embedding(1000 * sig[i], wts, cfg.time_freq_dim)) for i, x in enumerate(xs)]
        for i in range(cfg.warmup, steps):
            ref = O.rel_l1(tem[i - 1], tem[i])
            assert abs(logs[i]["signal"] - ref) <= 1e-3 * ref, ("loop", kind, i)
        assert np.isfinite(lat.cpu().numpy()).all()
    acid.check_device_error()
    rep = acid.bounds_report()
    assert rep["site"] == 0, rep
    print("bounds ok")
    """
)


def test_debug_build_index_checks():
    from paper_2607_12358_gb300 import build as b

    b.build(debug=True)
    env = dict(os.environ, ACID_LIBRARY="debug", PYTHONPATH=ROOT + os.pathsep + os.environ.get("PYTHONPATH", ""))
    r = subprocess.run([sys.executable, "-c", CHILD], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0 and "bounds ok" in r.stdout, r.stdout[-3000:] + r.stderr[-3000:]
