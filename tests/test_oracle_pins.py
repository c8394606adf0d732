"""Pins for the oracle's numerical pieces: closed forms, invariants, library
routines and statistical limits, chosen so that a dropped term, a wrong sign
or index or a transposed operand fails at least one of them."""

import math

import numpy as np
import pytest
import torch

import acid_synth as S
import oracle as O

torch.set_default_dtype(torch.float64)


# ---------------------------------------------------------------------------
# Drift signal (TeaCache relative L1, Sec. 2)
# ---------------------------------------------------------------------------

def test_rel_l1_closed_forms():
    rng = np.random.default_rng(0)
    a = rng.normal(size=1000)
    assert O.rel_l1(a, a) == 0.0
    for c in (-0.7, -0.01, 0.3, 2.0):
        assert O.rel_l1(a, (1 + c) * a) == pytest.approx(abs(c), rel=1e-12)
    assert O.rel_l1(a, -a) == pytest.approx(2.0, rel=1e-12)
    assert O.rel_l1(a, np.zeros_like(a)) == pytest.approx(1.0, rel=1e-12)


def test_rel_l1_normaliser_is_previous():
    """Swapping the arguments rescales by sum|a| / sum|b|: the denominator is
    the previous tensor's L1 norm, not the current one's."""
    rng = np.random.default_rng(1)
    a, b = rng.normal(size=500), 3.0 * rng.normal(size=500)
    assert O.rel_l1(a, b) * np.abs(a).sum() == pytest.approx(O.rel_l1(b, a) * np.abs(b).sum())


def test_rel_l1_zero_denominator_reading():
    z = np.zeros(8)
    assert O.rel_l1(z, z) == 0.0
    assert O.rel_l1(z, np.ones(8)) == math.inf


@pytest.mark.parametrize("sigma", [1e-3, 1e-2, 1e-1])
def test_rel_l1_statistical_limit(sigma):
    """prev ~ N(0,1), cur = prev + sigma z: E|sigma z| / E|x| = sigma, so the
    relative L1 tends to sigma (relative standard error ~0.8/sqrt(n))."""
    prev, cur = S.micro_pair(4096, sigma, seed=3, bf16=False)
    n = prev.size
    assert O.rel_l1(prev, cur) == pytest.approx(sigma, rel=6 * 0.8 / math.sqrt(n) + 1e-6)


def test_drift_sums_match_signal():
    rng = np.random.default_rng(2)
    a, b = rng.normal(size=100), rng.normal(size=100)
    num, den = O.drift_sums(a, b)
    assert num / den == pytest.approx(O.rel_l1(a, b))


# ---------------------------------------------------------------------------
# LayerNorm + adaLN, GELU, SiLU
# ---------------------------------------------------------------------------

def test_layernorm_identity_modulation():
    rng = np.random.default_rng(4)
    x = rng.normal(2.0, 3.0, size=(7, 64))
    y = O.modulate(O.layer_norm(x, 1e-6), np.zeros(64), np.zeros(64))
    np.testing.assert_allclose(y.mean(-1), 0, atol=1e-12)
    var = x.var(-1)
    np.testing.assert_allclose(y.var(-1), var / (var + 1e-6), rtol=1e-12)


def test_layernorm_matches_torch():
    rng = np.random.default_rng(5)
    x = rng.normal(size=(5, 48))
    sh, sc = rng.normal(size=48), rng.normal(size=48)
    ref = torch.nn.functional.layer_norm(torch.tensor(x), (48,), eps=1e-6).numpy() * (1 + sc) + sh
    np.testing.assert_allclose(O.modulate(O.layer_norm(x, 1e-6), sh, sc), ref, atol=1e-12)


def test_gelu_tanh_matches_torch_and_erf_bound():
    x = np.linspace(-8, 8, 4001)
    ref = torch.nn.functional.gelu(torch.tensor(x), approximate="tanh").numpy()
    np.testing.assert_allclose(O.gelu_tanh(x), ref, atol=1e-14)
    exact = torch.nn.functional.gelu(torch.tensor(x)).numpy()
    assert np.abs(O.gelu_tanh(x) - exact).max() < 1e-3
    # gelu(x) - gelu(-x) = x (the tanh term is odd)
    np.testing.assert_allclose(O.gelu_tanh(x) - O.gelu_tanh(-x), x, atol=1e-12)


def test_silu_matches_torch():
    x = np.linspace(-20, 20, 101)
    np.testing.assert_allclose(O.silu(x), torch.nn.functional.silu(torch.tensor(x)).numpy(), atol=1e-14)


# ---------------------------------------------------------------------------
# Attention
# ---------------------------------------------------------------------------

def test_attention_one_key_returns_value():
    rng = np.random.default_rng(6)
    q = rng.normal(size=(9, 3, 16))
    k = rng.normal(size=(1, 3, 16))
    v = rng.normal(size=(1, 3, 16))
    np.testing.assert_allclose(O.attention(q, k, v), np.broadcast_to(v, (9, 3, 16)), atol=1e-14)


def test_attention_zero_query_is_mean_value():
    rng = np.random.default_rng(7)
    k = rng.normal(size=(33, 2, 8))
    v = rng.normal(size=(33, 2, 8))
    out = O.attention(np.zeros((4, 2, 8)), k, v)
    np.testing.assert_allclose(out, np.broadcast_to(v.mean(0), (4, 2, 8)), atol=1e-14)


def test_attention_matches_torch_sdpa_and_permutation():
    rng = np.random.default_rng(8)
    q = 3 * rng.normal(size=(70, 4, 32))
    k = rng.normal(size=(130, 4, 32))
    v = rng.normal(size=(130, 4, 32))
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q).transpose(0, 1), torch.tensor(k).transpose(0, 1),
        torch.tensor(v).transpose(0, 1)).transpose(0, 1).numpy()
    out = O.attention(q, k, v, chunk=32)
    np.testing.assert_allclose(out, ref, atol=1e-12)
    perm = rng.permutation(130)
    np.testing.assert_allclose(O.attention(q, k[perm], v[perm]), out, atol=1e-12)


# ---------------------------------------------------------------------------
# 3D RoPE
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("Dh", [64, 128])
def test_rope_split(Dh):
    dt, dh, dw = O.rope_split(Dh)
    assert dt + dh + dw == Dh and dh == dw and dt % 2 == 0 and dh % 2 == 0
    assert (dt, dh) == {64: (24, 20), 128: (44, 42)}[Dh]


def test_rope_identity_at_origin_and_norm():
    rng = np.random.default_rng(9)
    grid = (3, 4, 5)
    x = rng.normal(size=(60, 2, 64))
    y = O.rope_apply(x, O.rope_angles(grid, 64))
    np.testing.assert_allclose(y[0], x[0], atol=1e-15)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-12)


def test_rope_matches_complex_rotation():
    """Pairs (2j, 2j+1) as complex numbers multiplied by exp(i angle)."""
    rng = np.random.default_rng(10)
    grid = (2, 3, 4)
    x = rng.normal(size=(24, 1, 128))
    ang = O.rope_angles(grid, 128)
    z = (x[..., 0::2] + 1j * x[..., 1::2]) * np.exp(1j * ang)[:, None, :]
    y = O.rope_apply(x, ang)
    np.testing.assert_allclose(y[..., 0::2], z.real, atol=1e-12)
    np.testing.assert_allclose(y[..., 1::2], z.imag, atol=1e-12)


def test_rope_relative_position_and_axes():
    """<R_m q, R_n k> depends only on m - n along each axis, and each axis
    owns its own block of pairs (t first, then h, then w)."""
    rng = np.random.default_rng(11)
    grid = (6, 7, 8)
    Dh = 64
    q = rng.normal(size=(1, 1, Dh))
    k = rng.normal(size=(1, 1, Dh))

    def tok(f, h, w):
        return f * 7 * 8 + h * 8 + w

    def dot(m, n):
        am = O.rope_angles(grid, Dh, positions=[m])
        an = O.rope_angles(grid, Dh, positions=[n])
        return float((O.rope_apply(q, am) * O.rope_apply(k, an)).sum())

    assert dot(tok(1, 2, 3), tok(0, 1, 1)) == pytest.approx(dot(tok(3, 4, 5), tok(2, 3, 3)), rel=1e-10)
    assert dot(tok(1, 2, 3), tok(0, 1, 1)) != pytest.approx(dot(tok(1, 2, 3), tok(0, 1, 2)), rel=1e-6)
    dt, dh, dw = O.rope_split(Dh)
    a = O.rope_angles(grid, Dh, positions=[tok(0, 0, 1)])[0]
    assert np.all(a[:dt // 2] == 0) and np.all(a[dt // 2:(dt + dh) // 2] == 0)
    np.testing.assert_allclose(a[(dt + dh) // 2:], 10000.0 ** (-np.arange(0, dw, 2) / dw))
    a = O.rope_angles(grid, Dh, positions=[tok(2, 0, 0)])[0]
    np.testing.assert_allclose(a[:dt // 2], 2 * 10000.0 ** (-np.arange(0, dt, 2) / dt))


# ---------------------------------------------------------------------------
# Timestep embedding, patchify, sampler
# ---------------------------------------------------------------------------

def test_timestep_sinusoid_closed_forms():
    e0 = O.timestep_sinusoid(0.0, 256)
    np.testing.assert_array_equal(e0[:128], 1.0)
    np.testing.assert_array_equal(e0[128:], 0.0)
    e = O.timestep_sinusoid(500.0, 256)
    assert e[0] == pytest.approx(math.cos(500.0)) and e[128] == pytest.approx(math.sin(500.0))
    f127 = math.exp(-math.log(10000.0) * 127 / 128)
    assert e[127] == pytest.approx(math.cos(500.0 * f127)) and e[255] == pytest.approx(math.sin(500.0 * f127))


def test_patchify_index_map_and_roundtrip():
    C, F_, H, W = 3, 2, 4, 6
    c, f, h, w = np.meshgrid(np.arange(C), np.arange(F_), np.arange(H), np.arange(W), indexing="ij")
    lat = c * 1000 + f * 100 + h * 10 + w
    tok = O.patchify(lat, 1, 2, 2)
    assert tok.shape == (2 * 2 * 3, 12)
    # token (f=1, hp=1, wp=2) = 1*6 + 1*3 + 2 = 11; feature (c=2, dh=1, dw=0) = 2*4 + 2 = 10
    assert tok[11, 10] == 2 * 1000 + 1 * 100 + (2 * 1 + 1) * 10 + (2 * 2 + 0)
    np.testing.assert_array_equal(O.unpatchify(tok, lat.shape, 1, 2, 2), lat)


def test_patchify_matches_conv3d_flatten():
    """A Conv3d with kernel = stride = patch equals the linear patch embedding
    over features ordered (c, dt, dh, dw)."""
    rng = np.random.default_rng(12)
    lat = rng.normal(size=(4, 2, 4, 6))
    wconv = rng.normal(size=(5, 4, 1, 2, 2))
    ref = torch.nn.functional.conv3d(torch.tensor(lat)[None], torch.tensor(wconv), stride=(1, 2, 2))
    ref = ref[0].reshape(5, -1).T.numpy()
    out = O.linear(O.patchify(lat, 1, 2, 2), wconv.reshape(5, -1))
    np.testing.assert_allclose(out, ref, atol=1e-12)


def test_time_mlp_and_modulation_silu_closed_forms():
    """SiLU(ln 3) = ln 3 / (1 + 1/3) = 0.75 ln 3.  A time MLP whose first layer
    has zero weights and bias ln 3, followed by an identity layer, returns
    0.75 ln 3 in every unit at any t; the block modulation W SiLU(temb) + b
    with W = I, b = 0 at temb = ln 3 returns the same."""
    d, l3 = 6, math.log(3.0)
    w = {"time1": (np.zeros((d, 256)), np.full(d, l3)), "time2": (np.eye(d), np.zeros(d))}
    for t in (0.0, 417.0, 1000.0):
        np.testing.assert_allclose(O.time_embedding(t, w, 256), 0.75 * l3, rtol=1e-15)
    np.testing.assert_allclose(O.block_modulation(np.full(d, l3), (np.eye(d), np.zeros(d))), 0.75 * l3,
                               rtol=1e-15)


def test_patch_embedding_bias_and_feature_selection():
    """A zero patch weight leaves its bias on every token; a weight that picks
    patch feature j reproduces column j of the patchified latent."""
    cfg = S.get_config("toy")
    w = S.model_weights(cfg, 0, blocks=False)
    lat = S.latent(cfg, 0)
    b = 0.01 * np.arange(cfg.d, dtype=float)
    h = O.step_inputs(cfg, dict(w, patch=(np.zeros((cfg.d, cfg.patch_dim)), b)), lat, 500.0, with_blocks=False).h_in
    assert h.shape == (cfg.n_video, cfg.d)
    np.testing.assert_array_equal(h, np.broadcast_to(b, h.shape))
    sel = np.zeros((cfg.d, cfg.patch_dim))
    sel[:, 5] = 1.0
    h = O.step_inputs(cfg, dict(w, patch=(sel, None)), lat, 500.0, with_blocks=False).h_in
    np.testing.assert_array_equal(h, np.repeat(O.patchify(lat, 1, 2, 2)[:, 5:6], cfg.d, axis=1))


def test_final_layer_on_constant_rows():
    """A constant row normalises to zero, so the final adaLN leaves only the
    shift: with every output unit averaging its input, every latent value is
    mean(shift_f) + bias whatever scale_f is (shift 2, scale 5, bias 0.25
    give 2.25)."""
    cfg = S.get_config("toy")
    d = cfg.d
    w = {"final": (np.full((cfg.patch_dim, d), 1.0 / d), np.full(cfg.patch_dim, 0.25))}
    h = np.repeat(np.arange(cfg.n_video, dtype=float)[:, None] - 7.0, d, axis=1)
    v = O.final_layer(cfg, w, h, np.concatenate([np.full(d, 2.0), np.full(d, 5.0)]))
    assert v.shape == cfg.latent_shape
    np.testing.assert_allclose(v, 2.25, rtol=1e-14)


def test_sigma_shift_closed_form_and_direction():
    """sigma' = s sigma / (1 + (s - 1) sigma) keeps 0 and 1, raises every
    interior level for s > 1 (more of the schedule at high noise) and lowers
    it for s < 1.  s = 3 on a 4-step grid gives 1, 0.9, 0.75, 0.5, 0."""
    np.testing.assert_allclose(O.sigmas(4, 3.0), [1.0, 0.9, 0.75, 0.5, 0.0], rtol=1e-15)
    base = O.sigmas(10)
    for shift in (1.5, 3.0, 7.0):
        sh = O.sigmas(10, shift)
        assert sh[0] == 1.0 and sh[-1] == 0.0 and np.all(sh[1:-1] > base[1:-1])
    assert np.all(O.sigmas(10, 0.5)[1:-1] < base[1:-1])


def test_euler_constant_velocity():
    """Constant v: x_N = x_0 + (sigma_N - sigma_0) v = x_0 - v exactly."""
    rng = np.random.default_rng(13)
    x0, v = rng.normal(size=10), rng.normal(size=10)
    for shift in (1.0, 3.0):
        s = O.sigmas(7, shift)
        assert s[0] == 1.0 and s[-1] == 0.0 and np.all(np.diff(s) < 0)
        x = x0
        for i in range(7):
            x = O.euler_step(x, v, s[i], s[i + 1])
        np.testing.assert_allclose(x, x0 - v, atol=1e-14)


# ---------------------------------------------------------------------------
# Blocks
# ---------------------------------------------------------------------------

def _torch_wan_block(x, mod, w, grid, H, ctx=None, eps=1e-6):
    """Independent composition from torch library routines: layer_norm,
    scaled_dot_product_attention, gelu(tanh) and a complex-number RoPE."""
    T = lambda a: torch.tensor(np.asarray(a, np.float64))
    x = T(x)
    n, d = x.shape
    Dh = d // H
    m = T(mod).reshape(6, d)
    F = torch.nn.functional

    def lin(a, name):
        return F.linear(a, T(w[name][0]), T(w[name][1]))

    def rope(t):
        ang = T(O.rope_angles(grid, Dh))  # angles as data; rotation done in complex form
        z = torch.view_as_complex(t.reshape(n, H, Dh // 2, 2).contiguous())
        z = z * torch.polar(torch.ones_like(ang), ang)[:, None, :]
        return torch.view_as_real(z).reshape(n, H, Dh)

    u = F.layer_norm(x, (d,), eps=eps) * (1 + m[1]) + m[0]
    q, k, v = lin(u, "qkv").split(d, dim=1)
    q, k = rope(q.reshape(n, H, Dh)), rope(k.reshape(n, H, Dh))
    a = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1),
                                       v.reshape(n, H, Dh).transpose(0, 1))
    x = x + m[2] * lin(a.transpose(0, 1).reshape(n, d), "o")
    if ctx is not None:
        c = T(ctx)
        qc = lin(F.layer_norm(x, (d,), eps=eps), "cq").reshape(n, H, Dh).transpose(0, 1)
        kc, vc = lin(c, "ckv").split(d, dim=1)
        L = c.shape[0]
        ac = F.scaled_dot_product_attention(qc, kc.reshape(L, H, Dh).transpose(0, 1),
                                            vc.reshape(L, H, Dh).transpose(0, 1))
        x = x + lin(ac.transpose(0, 1).reshape(n, d), "co")
    h = F.layer_norm(x, (d,), eps=eps) * (1 + m[4]) + m[3]
    return (x + m[5] * lin(F.gelu(lin(h, "ff1"), approximate="tanh"), "ff2")).numpy()


def _small(name="wan", **kw):
    base = dict(d=64, heads=2, ffn=96, latent_f=2, latent_h=6, latent_w=8)
    base.update(kw)
    return S.get_config(name, **base)


@pytest.mark.parametrize("with_ctx", [False, True])
def test_wan_block_matches_torch_composition(with_ctx):
    cfg = _small("wan", n_text=5 if with_ctx else 0, dtype="fp32")
    w = S.block_weights(cfg, 0, 0, q_scale=8.0)
    x = S.hidden(cfg, cfg.n_video)
    rng = np.random.default_rng(14)
    mod = 0.3 * rng.normal(size=6 * cfg.d)
    ctx = rng.normal(size=(5, cfg.d)) if with_ctx else None
    out = O.wan_block(x, mod, w, cfg.grid, cfg.heads, ctx=ctx)
    np.testing.assert_allclose(out, _torch_wan_block(x, mod, w, cfg.grid, cfg.heads, ctx), atol=1e-11)


def test_block_zero_gates_is_identity():
    cfg = _small("wan", n_text=4, dtype="fp32")
    w = S.block_weights(cfg, 0, 0, zero=("co",))
    x = S.hidden(cfg, cfg.n_video)
    rng = np.random.default_rng(15)
    mod = rng.normal(size=6 * cfg.d)
    mod[2 * cfg.d:3 * cfg.d] = 0
    mod[5 * cfg.d:] = 0
    out = O.wan_block(x, mod, w, cfg.grid, cfg.heads, ctx=rng.normal(size=(4, cfg.d)))
    np.testing.assert_array_equal(out, x.astype(np.float64))


@pytest.mark.parametrize("kind", ["wan", "cog", "hv_single"])
def test_sampled_rows_equal_full_block(kind):
    """The row-sampled evaluation (used at full sizes) equals the full one."""
    cfg = _small("cog" if kind == "cog" else "wan", n_text=6, dtype="fp32")
    bt = {"wan": "wan", "cog": "cog", "hv_single": "hv_single"}[kind]
    w = S.block_weights(cfg, 0, 0, block_type=bt)
    rng = np.random.default_rng(16)
    if kind == "wan":
        x = S.hidden(cfg, cfg.n_video)
        mod, ctx = rng.normal(size=6 * cfg.d) * 0.2, rng.normal(size=(6, cfg.d))
        f = lambda rows: O.wan_block(x, mod, w, cfg.grid, cfg.heads, ctx=ctx, rows=rows)
    elif kind == "cog":
        x = S.hidden(cfg, cfg.n_video + 6)
        mod = rng.normal(size=12 * cfg.d) * 0.2
        f = lambda rows: O.cog_block(x, mod, w, cfg.grid, cfg.heads, 6, rows=rows)
    else:
        x = S.hidden(cfg, cfg.n_video + 6)
        mod = rng.normal(size=3 * cfg.d) * 0.2
        f = lambda rows: O.hv_single_block(x, mod, w, cfg.grid, cfg.heads, 6, rows=rows)
    full = f(None)
    rows = np.array([0, 3, 5, 6, 17, x.shape[0] - 1])
    np.testing.assert_allclose(f(rows), full[rows], atol=1e-12)


def test_hv_dual_with_shared_weights_equals_cog_block():
    """A dual-stream block whose text and video streams share weights and
    modulation is the joint single-weight block."""
    cfg = _small("cog", n_text=5, dtype="fp32")
    wc = S.block_weights(cfg, 0, 0, block_type="cog")
    wd = {}
    for k in ("qkv", "o", "ff1", "ff2"):
        wd["vid." + k] = wc[k]
        wd["txt." + k] = wc[k]
    rng = np.random.default_rng(17)
    m6 = rng.normal(size=6 * cfg.d) * 0.3
    x = S.hidden(cfg, cfg.n_video + 5)
    ref = O.cog_block(x, np.concatenate([m6, m6]), wc, cfg.grid, cfg.heads, 5)
    yt, yv = O.hv_dual_block(x[:5], x[5:], m6, m6, wd, cfg.grid, cfg.heads)
    np.testing.assert_allclose(np.concatenate([yt, yv]), ref, atol=1e-12)


@pytest.mark.parametrize("kind", ["cog", "hv"])
def test_joint_stack_of_identity_blocks_returns_the_video_input(kind):
    """Joint sequences hold the text rows first.  With every gate zero each
    block is the identity, so the stack must hand back the video tokens it
    was given; a stack that put the video first would return a shifted mix
    of video and text rows."""
    cfg = _small(kind, n_text=5, dtype="fp32", n_blocks=1, **({"n_single": 1} if kind == "hv" else {}))
    w = S.model_weights(cfg, 2)
    h_in = S.hidden(cfg, cfg.n_video, tag="vid")
    ctx = S.hidden(cfg, 5, tag="txt")
    d = cfg.d
    mods = []
    for wb in w["blocks"]:
        if "vid.mod" in wb:
            m = 0.3 * np.ones(6 * d)
            m[2 * d:3 * d] = m[5 * d:] = 0.0
            mods.append((m, m))
        elif kind == "cog":
            m = 0.3 * np.ones(12 * d)
            for g in (2, 5, 8, 11):
                m[g * d:(g + 1) * d] = 0.0
            mods.append(m)
        else:
            m = 0.3 * np.ones(3 * d)
            m[2 * d:] = 0.0
            mods.append(m)
    np.testing.assert_allclose(O.block_stack(cfg, w, h_in, mods, ctx), h_in, atol=1e-12)


def test_text_context_closed_forms():
    """Wan projects the text once (Linear d_text -> d): a zero weight leaves
    its bias on every text token.  The joint models take the text tokens as
    given."""
    cfg = _small("wan", n_text=5, d_text=12, dtype="fp32")
    w = S.model_weights(cfg, 0, blocks=False)
    text = S.text(cfg, 0)
    b = 0.1 * np.arange(cfg.d, dtype=float)
    ctx = O.text_context(cfg, dict(w, text=(np.zeros((cfg.d, 12)), b)), text)
    np.testing.assert_array_equal(ctx, np.broadcast_to(b, (5, cfg.d)))
    cog = _small("cog", n_text=5, dtype="fp32")
    t = S.hidden(cog, 5, tag="txt")
    np.testing.assert_array_equal(O.text_context(cog, {}, t), t)


def test_dual_stream_step_modulation_reaches_its_own_stream():
    """A dual-stream block whose video gates are zero leaves the video tokens
    unchanged, whatever the text stream's modulation: an HV step's block
    stack must return its video input when only the video modulation's gate
    rows are zeroed, and must not when only the text's are."""
    cfg = _small("hv", n_text=5, dtype="fp32", n_blocks=1)
    w = S.model_weights(cfg, 4)
    lat = S.latent(cfg, 4)
    text = S.hidden(cfg, 5, tag="txt")
    d = cfg.d

    def zero_gates(mod):
        W, b = (np.array(a, dtype=float) for a in mod)
        for g in (2, 5):
            W[g * d:(g + 1) * d] = 0.0
            b[g * d:(g + 1) * d] = 0.0
        return W, b

    for stream, identity in (("vid.mod", True), ("txt.mod", False)):
        blocks = [dict(w["blocks"][0], **{stream: zero_gates(w["blocks"][0][stream])})]
        wz = dict(w, blocks=blocks)
        si = O.step_inputs(cfg, wz, lat, 700.0)
        out = O.block_stack(cfg, wz, si.h_in, si.mods, text)
        assert np.allclose(out, si.h_in, atol=1e-12) == identity, stream


def test_hv_dual_streams_are_interchangeable_without_rope():
    """Without RoPE the dual-stream block treats its two streams alike.
    Swapping the text and video inputs, modulations and per-stream weights
    swaps the outputs, since joint attention does not depend on the order of
    its keys.  A stream that reaches for the other stream's weights, gate or
    modulation breaks the symmetry."""
    cfg = _small("hv", n_text=5, dtype="fp32")
    w = S.block_weights(cfg, 0, 0, block_type="hv_dual")
    ws = {}
    for k, v in w.items():
        if k.startswith("txt."):
            ws["vid." + k[4:]] = v
        elif k.startswith("vid."):
            ws["txt." + k[4:]] = v
        else:
            ws[k] = v
    rng = np.random.default_rng(23)
    mt, mv = 0.3 * rng.normal(size=6 * cfg.d), 0.3 * rng.normal(size=6 * cfg.d)
    xt, xv = S.hidden(cfg, 5, tag="txt"), S.hidden(cfg, 9, tag="vid")
    yt, yv = O.hv_dual_block(xt, xv, mt, mv, w, cfg.grid, cfg.heads, rope=False)
    yv2, yt2 = O.hv_dual_block(xv, xt, mv, mt, ws, cfg.grid, cfg.heads, rope=False)
    np.testing.assert_allclose(yt2, yt, atol=1e-12)
    np.testing.assert_allclose(yv2, yv, atol=1e-12)
    assert np.abs(yt - xt).max() > 1e-3 and np.abs(yv - xv).max() > 1e-3


def test_cog_text_modulation_only_touches_text_rows():
    cfg = _small("cog", n_text=5, dtype="fp32")
    w = S.block_weights(cfg, 0, 0, block_type="cog")
    rng = np.random.default_rng(18)
    m = rng.normal(size=12 * cfg.d) * 0.3
    x = S.hidden(cfg, cfg.n_video + 5)
    base = O.cog_block(x, m, w, cfg.grid, cfg.heads, 5)
    m2 = m.copy()
    m2[6 * cfg.d + 5 * cfg.d:] += 1.0  # text gate2 only
    alt = O.cog_block(x, m2, w, cfg.grid, cfg.heads, 5)
    np.testing.assert_array_equal(alt[5:], base[5:])
    assert np.abs(alt[:5] - base[:5]).max() > 1e-3


def test_hv_single_reduces_to_attention_half_of_wan_block():
    """W2 = [W_o | 0] and no text: the single-stream block is the Wan block's
    attention branch (its FFN branch zeroed)."""
    cfg = _small("wan", n_text=0, dtype="fp32")
    ww = S.block_weights(cfg, 0, 0, block_type="wan", zero=("ff2",))
    ws = S.block_weights(cfg, 0, 0, block_type="hv_single")
    ws["qkv"] = ww["qkv"]
    w2 = np.zeros_like(ws["w2"][0])
    w2[:, :cfg.d] = ww["o"][0]
    ws["w2"] = (w2, ww["o"][1])
    rng = np.random.default_rng(19)
    m3 = rng.normal(size=3 * cfg.d) * 0.3
    m6 = np.concatenate([m3, np.zeros(3 * cfg.d)])
    x = S.hidden(cfg, cfg.n_video)
    np.testing.assert_allclose(O.hv_single_block(x, m3, ws, cfg.grid, cfg.heads, 0),
                               O.wan_block(x, m6, ww, cfg.grid, cfg.heads), atol=1e-12)


def test_hv_single_reduces_to_ffn_half_of_wan_block():
    """W2 = [0 | W_ff2] and no text: the single-stream block is the Wan block's
    feed-forward branch (its attention branch gated off), with W_mlp as the
    first FFN layer and the same shift, scale and gate."""
    cfg = _small("wan", n_text=0, dtype="fp32")
    ww = S.block_weights(cfg, 0, 0, block_type="wan")
    ws = S.block_weights(cfg, 0, 0, block_type="hv_single")
    ws["mlp"] = ww["ff1"]
    w2 = np.zeros_like(ws["w2"][0])
    w2[:, cfg.d:] = ww["ff2"][0]
    ws["w2"] = (w2, ww["ff2"][1])
    rng = np.random.default_rng(21)
    m3 = rng.normal(size=3 * cfg.d) * 0.3
    m6 = np.concatenate([np.zeros(3 * cfg.d), m3])
    x = S.hidden(cfg, cfg.n_video)
    np.testing.assert_allclose(O.hv_single_block(x, m3, ws, cfg.grid, cfg.heads, 0),
                               O.wan_block(x, m6, ww, cfg.grid, cfg.heads), atol=1e-12)


def test_joint_block_token_permutation_without_rope():
    """Without RoPE, joint attention has no notion of order: permuting the
    video tokens permutes the output."""
    cfg = _small("wan", n_text=4, dtype="fp32")
    w = S.block_weights(cfg, 0, 0, block_type="hv_single")
    rng = np.random.default_rng(20)
    m3 = rng.normal(size=3 * cfg.d) * 0.3
    x = S.hidden(cfg, cfg.n_video + 4)
    perm = np.concatenate([np.arange(4), 4 + rng.permutation(cfg.n_video)])
    a = O.hv_single_block(x, m3, w, cfg.grid, cfg.heads, 4, rope=False)
    b = O.hv_single_block(x[perm], m3, w, cfg.grid, cfg.heads, 4, rope=False)
    np.testing.assert_allclose(b, a[perm], atol=1e-12)


def test_temni_is_block0_modulated_input():
    cfg = S.get_config("toy")
    w = S.model_weights(cfg, 0)
    lat = S.latent(cfg, 0)
    si = O.step_inputs(cfg, w, lat, 1000.0)
    temni = O.block0_temni(cfg, w, si.h_in, si.temb)
    d = cfg.d
    m = si.mods[0]
    np.testing.assert_allclose(temni, O.modulate(O.layer_norm(si.h_in), m[:d], m[d:2 * d]), atol=0)
    # shift/scale are the first two d-chunks of block 0's modulation (DiT order)
    assert np.abs(temni.mean(-1) - m[:d].mean() - (O.layer_norm(si.h_in) * m[d:2 * d]).mean(-1)).max() < 1e-12
