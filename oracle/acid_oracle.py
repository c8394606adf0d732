"""Plain float64 restatement of ACID (adaptive dual-threshold step caching)
and of the video-DiT denoising step it wraps.  TEST INFRASTRUCTURE ONLY:
imported by tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py``; never by the product path.

Sections follow the paper:

* drift signals of the wrapped methods (Sec. 2, "TeaCache", "EasyCache");
* the reuse rules of those methods (same paragraphs);
* the adaptive threshold controller (Sec. 3.3, Algorithm 1);
* the reverse-diffusion step loop (Sec. 3.1, Eq. 2), taken as Euler
  flow-matching steps because the workloads specify that sampler;
* the DiT denoiser f_theta(x_t, t, c) (named, not defined, by the paper;
  the paper gives no block definition, so the ones below are readings of
  the workloads' stated architecture).

Parity pins live in ``tests/test_oracle_*.py``.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

F64 = np.float64

# =============================================================================
# Drift signals and reuse rules (Sec. 2)
# =============================================================================


def rel_l1(prev, cur) -> float:
    """TeaCache drift: L1 distance between consecutive modulated inputs,
    relative to the previous one:  sum|cur - prev| / sum|prev|  (Sec. 2,
    "TeaCache"; the relative form is the one the workloads specify).

    Reading for a zero denominator (the paper is silent): 0 when the
    numerator is 0 too, else +inf (which forces a computed step).
    """
    p = np.asarray(prev, dtype=F64).ravel()
    c = np.asarray(cur, dtype=F64).ravel()
    if p.shape != c.shape:
        raise ValueError("shape mismatch")
    num = float(np.abs(c - p).sum())
    den = float(np.abs(p).sum())
    if den == 0.0:
        return 0.0 if num == 0.0 else math.inf
    return num / den


def drift_sums(prev, cur) -> tuple[float, float]:
    """The two sums behind rel_l1: (sum|cur - prev|, sum|prev|)."""
    p = np.asarray(prev, dtype=F64).ravel()
    c = np.asarray(cur, dtype=F64).ravel()
    return float(np.abs(c - p).sum()), float(np.abs(p).sum())


def cache_apply(x, cached_residual) -> np.ndarray:
    """TeaCache reuse on a skipped step: previous block-stack residual added to
    the current block-stack input, H_out = H_in + R (Sec. 2, "TeaCache").
    EasyCache's reuse v_t = x_t + Delta is the same addition (Sec. 2,
    "EasyCache")."""
    return np.asarray(x, dtype=F64) + np.asarray(cached_residual, dtype=F64)


def mean_abs(a) -> float:
    return float(np.abs(np.asarray(a, dtype=F64)).mean())


def easycache_rate(x_c, x_prev, v_c, v_prev) -> float:
    """EasyCache transformation rate k at a computed step c: output change over
    input change between step c-1 and c (Sec. 2, "EasyCache").  Reading: both
    changes measured as mean absolute differences."""
    dx = mean_abs(np.asarray(x_c, F64) - np.asarray(x_prev, F64))
    dv = mean_abs(np.asarray(v_c, F64) - np.asarray(v_prev, F64))
    if dx == 0.0:
        return 0.0 if dv == 0.0 else math.inf
    return dv / dx


def easycache_signal(k: float, x_t, x_prev, v_prev) -> float:
    """EasyCache drift estimate k * Delta_input / ||v_{t-1}|| (Sec. 2,
    "EasyCache"; Sec. 3.3 names it as the signal ACID monitors).  Reading:
    Delta_input = mean|x_t - x_{t-1}|, ||v_{t-1}|| = mean|v_{t-1}|."""
    dx = mean_abs(np.asarray(x_t, F64) - np.asarray(x_prev, F64))
    nv = mean_abs(v_prev)
    num = k * dx
    if nv == 0.0:
        return 0.0 if num == 0.0 else math.inf
    return num / nv


def easycache_reuse(x_t, x_c, v_c) -> np.ndarray:
    """EasyCache reconstruction on a skipped step: current input plus the
    offset output - input of the last computed step (Sec. 2, "EasyCache")."""
    return np.asarray(x_t, F64) + (np.asarray(v_c, F64) - np.asarray(x_c, F64))


def dicache_gamma(p_t, p_c1, p_c2) -> float:
    """Probe-trajectory ratio |P_t - P_c1|_1 / |P_c1 - P_c2|_1 (0 when the
    denominator is 0, i.e. fewer than two distinct computed steps)."""
    den = float(np.abs(np.asarray(p_c1, F64) - np.asarray(p_c2, F64)).sum())
    if den == 0.0:
        return 0.0
    return float(np.abs(np.asarray(p_t, F64) - np.asarray(p_c1, F64)).sum()) / den


def dicache_reuse(p_t, p_c1, p_c2, d_c1, d_c2) -> np.ndarray:
    """DiCache reconstruction on a skipped step (Sec. 2, "DiCache": the deep
    output is estimated from the probe features' trajectory over recent
    steps).  Reading: with D = H_out - P the deep part beyond the probe at
    the last two computed steps c1 (latest) and c2,
        H_out_t = P_t + D_c1 + gamma (D_c1 - D_c2),
        gamma = |P_t - P_c1|_1 / |P_c1 - P_c2|_1,
    i.e. the deep part moves along its last computed direction in proportion
    to how far the probe has moved since."""
    g = dicache_gamma(p_t, p_c1, p_c2)
    d1 = np.asarray(d_c1, F64)
    return np.asarray(p_t, F64) + d1 + g * (d1 - np.asarray(d_c2, F64))


# =============================================================================
# Adaptive threshold controller (Sec. 3.3, Algorithm 1)
# =============================================================================


@dataclass
class StepRecord:
    step: int
    warmup: bool
    signal: float = math.nan       # s_t (nan on warmup steps)
    dsignal: float = math.nan      # |s_t - s_prev| (nan when s_prev is None)
    tau: float = math.nan          # active threshold
    sigma: float = math.nan        # accumulated drift compared against tau
    computed: bool = True          # full model evaluated at this step
    forced: bool = False


class AcidController:
    """Algorithm 1 of Sec. 3.3, stepwise.

    State: accumulated drift Sigma (starts at 0) and previous signal s_prev
    (starts as None).  On a non-warmup step with signal s_t:

    1. Sigma += s_t (before the threshold is chosen);
    2. tau = tau_high if s_prev is not None and |s_t - s_prev| <= delta
       (the closed interval [-delta, delta] of Sec. 3.3), else tau_low;
    3. reuse (skip) if Sigma <= tau, otherwise run the model and set Sigma = 0;
    4. s_prev = s_t, whichever branch was taken.

    Warmup steps run the model and touch neither Sigma nor s_prev.
    ``forced`` overrides the decision of step 3 (used only to continue a
    comparison past an ambiguous step); the state then follows the forced
    branch.  ``tau_fixed`` (a number, not NaN) replaces the threshold of step
    2: the fixed-schedule dual threshold of Sec. 3.2, which switches from a
    low to a high threshold at a chosen step regardless of the signal.
    """

    def __init__(self, tau_low: float, tau_high: float, delta: float):
        self.tau_low = float(tau_low)
        self.tau_high = float(tau_high)
        self.delta = float(delta)
        self.sigma = 0.0
        self.s_prev: float | None = None

    def step(self, s_t: float, forced: bool | None = None,
             tau_fixed: float | None = None) -> tuple[bool, float, float, float]:
        """Returns (skip, tau, sigma_compared, |s_t - s_prev| or nan)."""
        s_t = float(s_t)
        self.sigma = self.sigma + s_t
        if self.s_prev is not None:
            ds = abs(s_t - self.s_prev)
            tau = self.tau_high if ds <= self.delta else self.tau_low
        else:
            ds = math.nan
            tau = self.tau_low
        if tau_fixed is not None and not math.isnan(tau_fixed):
            tau = float(tau_fixed)
        sigma_seen = self.sigma
        skip = sigma_seen <= tau
        if forced is not None:
            skip = not bool(forced)
        if not skip:
            self.sigma = 0.0
        self.s_prev = s_t
        return skip, tau, sigma_seen, ds


def rescale_signal(s: float, coeffs=None) -> float:
    """Optional rescaling of a raw drift value before Algorithm 1,
    s' = sum_j c_j s^j (ascending powers; identity without coefficients).
    TeaCache calibrates such a polynomial per model; the paper's Algorithm 1
    takes the base method's signal as given, so the default is the identity."""
    if not coeffs:
        return float(s)
    return float(sum(c * s ** j for j, c in enumerate(coeffs)))


def controller_decisions(signals, warmup: int, tau_low: float, tau_high: float,
                         delta: float, tau_schedule=None) -> list[bool]:
    """Computed-step mask of Algorithm 1 for a fixed signal sequence
    (``signals[i]`` is ignored for the first ``warmup`` steps)."""
    ctl = AcidController(tau_low, tau_high, delta)
    out = []
    for i, s in enumerate(signals):
        if i < warmup:
            out.append(True)
            continue
        skip, _, _, _ = ctl.step(s, tau_fixed=None if tau_schedule is None else tau_schedule[i])
        out.append(not skip)
    return out


# =============================================================================
# Sampler (Sec. 3.1, Eq. 2 as Euler flow matching)
# =============================================================================


def sigmas(n_steps: int, shift: float = 1.0) -> np.ndarray:
    """Noise levels sigma_i = 1 - i/N, i = 0..N, optionally shifted
    sigma' = s*sigma / (1 + (s-1)*sigma).  Reading: the paper gives the DDPM
    form (Eq. 2); the workloads name Euler flow-matching steps."""
    s = 1.0 - np.arange(n_steps + 1, dtype=F64) / n_steps
    if shift != 1.0:
        s = shift * s / (1.0 + (shift - 1.0) * s)
    return s


def euler_step(x, v, sigma_cur: float, sigma_next: float) -> np.ndarray:
    """x_{i+1} = x_i + (sigma_{i+1} - sigma_i) * v_i."""
    return np.asarray(x, F64) + (sigma_next - sigma_cur) * np.asarray(v, F64)


# =============================================================================
# DiT building blocks (readings; the paper names the models only, Sec. 4.1)
# =============================================================================


def layer_norm(x, eps: float = 1e-6) -> np.ndarray:
    """LayerNorm over the last axis without affine parameters."""
    x = np.asarray(x, F64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def modulate(xn, shift, scale) -> np.ndarray:
    """adaLN modulation xn * (1 + scale) + shift."""
    return np.asarray(xn, F64) * (1.0 + np.asarray(scale, F64)) + np.asarray(shift, F64)


def gelu_tanh(x) -> np.ndarray:
    """GELU, tanh form: 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))."""
    x = np.asarray(x, F64)
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def silu(x) -> np.ndarray:
    x = np.asarray(x, F64)
    return x / (1.0 + np.exp(-x))


def linear(x, w, b=None) -> np.ndarray:
    """y = x W^T + b with W stored [out, in]."""
    y = np.asarray(x, F64) @ np.asarray(w, F64).T
    if b is not None:
        y = y + np.asarray(b, F64)
    return y


def timestep_sinusoid(t: float, dim: int = 256, max_period: float = 10000.0) -> np.ndarray:
    """[cos(t f_j) | sin(t f_j)], f_j = max_period^(-j/(dim/2)), j < dim/2."""
    half = dim // 2
    f = np.exp(-math.log(max_period) * np.arange(half, dtype=F64) / half)
    a = float(t) * f
    return np.concatenate([np.cos(a), np.sin(a)])


def time_embedding(t: float, w: dict, dim: int = 256) -> np.ndarray:
    """temb = W2 SiLU(W1 sinusoid(t) + b1) + b2."""
    h = linear(timestep_sinusoid(t, dim), *w["time1"])
    return linear(silu(h), *w["time2"])


def block_modulation(temb, wb) -> np.ndarray:
    """Per-block adaLN vector W_mod SiLU(temb) + b_mod."""
    return linear(silu(temb), *wb)


def rope_split(head_dim: int) -> tuple[int, int, int]:
    """(d_t, d_h, d_w): d_h = d_w = 2 floor(Dh/6), d_t = Dh - 2 d_h."""
    dh = 2 * (head_dim // 6)
    return head_dim - 2 * dh, dh, dh


def rope_angles(grid, head_dim: int, theta: float = 10000.0, positions=None) -> np.ndarray:
    """Rotation angles [n_tok, Dh/2] of 3D RoPE.  Token n = f*Hp*Wp + h*Wp + w;
    pair j of the head dimension belongs to the t, h or w axis in that order,
    with frequency theta^(-2 j'/d_axis) for its index j' within the axis."""
    F_, Hp, Wp = grid
    if positions is None:
        positions = np.arange(F_ * Hp * Wp)
    positions = np.asarray(positions)
    f = positions // (Hp * Wp)
    h = (positions // Wp) % Hp
    w = positions % Wp
    dt, dh, dw = rope_split(head_dim)
    cols = []
    for pos, da in ((f, dt), (h, dh), (w, dw)):
        inv = theta ** (-np.arange(0, da, 2, dtype=F64) / da)
        cols.append(pos[:, None].astype(F64) * inv[None, :])
    return np.concatenate(cols, axis=1)


def rope_apply(x, angles) -> np.ndarray:
    """Rotate interleaved pairs (2j, 2j+1) of x [n, H, Dh] by angles [n, Dh/2]."""
    x = np.asarray(x, F64)
    c = np.cos(angles)[:, None, :]
    s = np.sin(angles)[:, None, :]
    x0 = x[..., 0::2]
    x1 = x[..., 1::2]
    y = np.empty_like(x)
    y[..., 0::2] = x0 * c - x1 * s
    y[..., 1::2] = x0 * s + x1 * c
    return y


def attention(q, k, v, chunk: int = 1024) -> np.ndarray:
    """softmax(q k^T / sqrt(Dh)) v per head; q [nq, H, Dh], k/v [nk, H, Dh]."""
    q = np.asarray(q, F64)
    k = np.asarray(k, F64)
    v = np.asarray(v, F64)
    nq, H, Dh = q.shape
    out = np.empty((nq, H, v.shape[-1]), dtype=F64)
    scale = 1.0 / math.sqrt(Dh)
    for h in range(H):
        kh = k[:, h, :]
        vh = v[:, h, :]
        for s0 in range(0, nq, chunk):
            s = (q[s0:s0 + chunk, h, :] @ kh.T) * scale
            s = s - s.max(axis=1, keepdims=True)
            p = np.exp(s)
            p /= p.sum(axis=1, keepdims=True)
            out[s0:s0 + chunk, h, :] = p @ vh
    return out


def _heads(a, H):
    return a.reshape(a.shape[0], H, -1)


def _rows(rows, n):
    return np.arange(n) if rows is None else np.asarray(rows)


# ---- blocks ------------------------------------------------------------------
# Every block takes x (all tokens) and returns the updated rows ``rows``
# (default: all).  Per-token operations run only on the returned rows; the
# keys and values of attention are computed for every token.


def wan_block(x, mod, w, grid, heads, ctx=None, eps=1e-6, theta=10000.0, rows=None,
              rope=True) -> np.ndarray:
    """Wan-style block (also the toy block when ctx is None):
      x += g1 * O(Attn_RoPE(QKV(LNmod1(x))))
      x += O_c(Attn(Q_c(LN(x)), K_c/V_c(ctx)))        (only with ctx)
      x += g2 * W2 GELU(W1 LNmod2(x))
    mod = [shift1, scale1, gate1, shift2, scale2, gate2] (6d)."""
    x = np.asarray(x, F64)
    n, d = x.shape
    r = _rows(rows, n)
    sh1, sc1, g1, sh2, sc2, g2 = np.split(np.asarray(mod, F64), 6)
    u = modulate(layer_norm(x, eps), sh1, sc1)
    wq, bq = w["qkv"][0][:d], w["qkv"][1][:d]
    wkv, bkv = w["qkv"][0][d:], w["qkv"][1][d:]
    q = _heads(linear(u[r], wq, bq), heads)
    kv = linear(u, wkv, bkv)
    k = _heads(kv[:, :d], heads)
    v = _heads(kv[:, d:], heads)
    if rope:
        Dh = d // heads
        q = rope_apply(q, rope_angles(grid, Dh, theta, positions=r))
        k = rope_apply(k, rope_angles(grid, Dh, theta))
    a = attention(q, k, v).reshape(len(r), d)
    y = x[r] + g1 * linear(a, *w["o"])
    if ctx is not None:
        c = np.asarray(ctx, F64)
        qc = _heads(linear(layer_norm(y, eps), *w["cq"]), heads)
        kvc = linear(c, *w["ckv"])
        kc = _heads(kvc[:, :d], heads)
        vc = _heads(kvc[:, d:], heads)
        y = y + linear(attention(qc, kc, vc).reshape(len(r), d), *w["co"])
    h = modulate(layer_norm(y, eps), sh2, sc2)
    return y + g2 * linear(gelu_tanh(linear(h, *w["ff1"])), *w["ff2"])


def _stream_mod(mods_by_stream, n_text, idx, part):
    """Per-row modulation vector: rows < n_text use the text stream."""
    mv, mt = mods_by_stream
    a = np.where((idx < n_text)[:, None], mt[part][None, :], mv[part][None, :])
    return a


def cog_block(x, mod, w, grid, heads, n_text, eps=1e-6, theta=10000.0, rows=None,
              rope=True) -> np.ndarray:
    """CogVideoX-style joint block over [text (n_text) ; video] tokens with one
    set of weights and separate modulation per stream; mod = video 6d then
    text 6d.  RoPE on video tokens only (video position = row - n_text)."""
    x = np.asarray(x, F64)
    n, d = x.shape
    r = _rows(rows, n)
    m = np.asarray(mod, F64)
    mv = np.split(m[:6 * d], 6)
    mt = np.split(m[6 * d:], 6)
    allr = np.arange(n)

    def lnmod(z, idx, base):
        return modulate(layer_norm(z, eps), _stream_mod((mv, mt), n_text, idx, base),
                        _stream_mod((mv, mt), n_text, idx, base + 1))

    u = lnmod(x, allr, 0)
    qkv_all = linear(u, *w["qkv"])
    q = _heads(qkv_all[r, :d], heads)
    k = _heads(qkv_all[:, d:2 * d], heads)
    v = _heads(qkv_all[:, 2 * d:], heads)
    if rope:
        q = _rope_video(q, r, n_text, grid, d // heads, theta)
        k = _rope_video(k, allr, n_text, grid, d // heads, theta)
    a = attention(q, k, v).reshape(len(r), d)
    g1 = _stream_mod((mv, mt), n_text, r, 2)
    y = x[r] + g1 * linear(a, *w["o"])
    h = lnmod(y, r, 3)
    g2 = _stream_mod((mv, mt), n_text, r, 5)
    return y + g2 * linear(gelu_tanh(linear(h, *w["ff1"])), *w["ff2"])


def _rope_video(t, idx, n_text, grid, Dh, theta):
    """Apply 3D RoPE to rows whose token index is >= n_text."""
    idx = np.asarray(idx)
    out = t.copy()
    vid = idx >= n_text
    if vid.any():
        out[vid] = rope_apply(t[vid], rope_angles(grid, Dh, theta, positions=idx[vid] - n_text))
    return out


def hv_dual_block(x_txt, x_vid, mod_txt, mod_vid, w, grid, heads, eps=1e-6, theta=10000.0,
                  rows_vid=None, rows_txt=None, rope=True):
    """HunyuanVideo-style dual-stream block: per-stream weights (mod, qkv, o,
    ff1, ff2), joint attention over [text ; video], RoPE on video tokens.
    Returns (x_txt[rows_txt], x_vid[rows_vid])."""
    xt = np.asarray(x_txt, F64)
    xv = np.asarray(x_vid, F64)
    L, d = xt.shape
    N = xv.shape[0]
    rv = _rows(rows_vid, N)
    rt = _rows(rows_txt, L)
    mt = np.split(np.asarray(mod_txt, F64), 6)
    mv = np.split(np.asarray(mod_vid, F64), 6)
    ut = modulate(layer_norm(xt, eps), mt[0], mt[1])
    uv = modulate(layer_norm(xv, eps), mv[0], mv[1])
    qkv_t = linear(ut, *w["txt.qkv"])
    qkv_v = linear(uv, *w["vid.qkv"])
    Dh = d // heads
    qv = _heads(qkv_v[rv, :d], heads)
    kv_ = _heads(qkv_v[:, d:2 * d], heads)
    if rope:
        qv = rope_apply(qv, rope_angles(grid, Dh, theta, positions=rv))
        kv_ = rope_apply(kv_, rope_angles(grid, Dh, theta))
    k = np.concatenate([_heads(qkv_t[:, d:2 * d], heads), kv_], axis=0)
    v = np.concatenate([_heads(qkv_t[:, 2 * d:], heads), _heads(qkv_v[:, 2 * d:], heads)], axis=0)
    q = np.concatenate([_heads(qkv_t[rt, :d], heads), qv], axis=0)
    a = attention(q, k, v).reshape(len(rt) + len(rv), d)
    at, av = a[:len(rt)], a[len(rt):]
    yt = xt[rt] + mt[2] * linear(at, *w["txt.o"])
    yv = xv[rv] + mv[2] * linear(av, *w["vid.o"])
    ht = modulate(layer_norm(yt, eps), mt[3], mt[4])
    hv = modulate(layer_norm(yv, eps), mv[3], mv[4])
    yt = yt + mt[5] * linear(gelu_tanh(linear(ht, *w["txt.ff1"])), *w["txt.ff2"])
    yv = yv + mv[5] * linear(gelu_tanh(linear(hv, *w["vid.ff1"])), *w["vid.ff2"])
    return yt, yv


def hv_single_block(x, mod, w, grid, heads, n_text, eps=1e-6, theta=10000.0, rows=None,
                    rope=True) -> np.ndarray:
    """HunyuanVideo-style single-stream block over [text ; video]:
      h = LNmod(x);  qkv = h W_qkv;  m = GELU(h W_mlp)
      x += g * W2 [Attn_RoPE(qkv) | m]      (W2: d x (d + ffn))
    mod = [shift, scale, gate] (3d)."""
    x = np.asarray(x, F64)
    n, d = x.shape
    r = _rows(rows, n)
    sh, sc, g = np.split(np.asarray(mod, F64), 3)
    h = modulate(layer_norm(x, eps), sh, sc)
    qkv_all = linear(h, *w["qkv"])
    allr = np.arange(n)
    Dh = d // heads
    q = _heads(qkv_all[r, :d], heads)
    k = _heads(qkv_all[:, d:2 * d], heads)
    v = _heads(qkv_all[:, 2 * d:], heads)
    if rope:
        q = _rope_video(q, r, n_text, grid, Dh, theta)
        k = _rope_video(k, allr, n_text, grid, Dh, theta)
    a = attention(q, k, v).reshape(len(r), d)
    m = gelu_tanh(linear(h[r], *w["mlp"]))
    return x[r] + g * linear(np.concatenate([a, m], axis=1), *w["w2"])


# =============================================================================
# Whole denoiser f_theta and the step loop (Algorithm 1 wrapped around it)
# =============================================================================


def patchify(latent, pt, ph, pw) -> np.ndarray:
    """[C, F, H, W] -> tokens [N, C*pt*ph*pw]; token n = f*Hp*Wp + h*Wp + w,
    feature index c*(pt*ph*pw) + dt*(ph*pw) + dh*pw + dw."""
    a = np.asarray(latent, F64)
    C, F_, H, W = a.shape
    a = a.reshape(C, F_ // pt, pt, H // ph, ph, W // pw, pw)
    a = a.transpose(1, 3, 5, 0, 2, 4, 6)
    return a.reshape((F_ // pt) * (H // ph) * (W // pw), C * pt * ph * pw)


def unpatchify(tokens, latent_shape, pt, ph, pw) -> np.ndarray:
    C, F_, H, W = latent_shape
    a = np.asarray(tokens, F64).reshape(F_ // pt, H // ph, W // pw, C, pt, ph, pw)
    a = a.transpose(3, 0, 4, 1, 5, 2, 6)
    return a.reshape(C, F_, H, W)


@dataclass
class StepInputs:
    """Quantities of one step that do not depend on the block stack."""
    temb: np.ndarray
    h_in: np.ndarray          # video tokens after patch embedding [N, d]
    mods: list                # per-block modulation vectors
    final_mod: np.ndarray     # [2d]


def step_inputs(cfg, w, x_latent, t: float, with_blocks: bool = True) -> StepInputs:
    temb = time_embedding(t, w, cfg.time_freq_dim)
    h_in = linear(patchify(x_latent, cfg.pt, cfg.ph, cfg.pw), *w["patch"])
    mods = []
    for wb in (w["blocks"] if with_blocks else []):
        if "vid.mod" in wb:  # dual-stream block: (video, text)
            mods.append((block_modulation(temb, wb["vid.mod"]), block_modulation(temb, wb["txt.mod"])))
        else:
            mods.append(block_modulation(temb, wb["mod"]))
    fm = block_modulation(temb, w["final_mod"])
    return StepInputs(temb=temb, h_in=h_in, mods=mods, final_mod=fm)


def block0_temni(cfg, w, h_in, temb) -> np.ndarray:
    """TeaCache's timestep-embedding-modulated noisy input (Sec. 2,
    "TeaCache"): the first block's attention-branch adaLN applied to the
    video tokens, LN(h) (1 + scale1) + shift1, with block 0's video-stream
    modulation at this step's timestep embedding."""
    wb = w["blocks"][0]
    m = block_modulation(temb, wb["vid.mod"] if "vid.mod" in wb else wb["mod"])
    d = cfg.d
    return modulate(layer_norm(h_in, cfg.ln_eps), m[:d], m[d:2 * d])


def text_context(cfg, w, text):
    """Wan: ctx = Linear(d_text -> d)(text); Cog/HV: the text tokens as given."""
    if text is None:
        return None
    if cfg.kind == "wan":
        return linear(text, *w["text"])
    return np.asarray(text, F64)


def stack_state(cfg, h_in, ctx) -> np.ndarray:
    """Hidden state entering the block stack: the video tokens (Wan) or
    [text ; video] (joint models)."""
    if cfg.kind == "wan":
        return np.asarray(h_in, F64)
    return np.concatenate([np.asarray(ctx, F64), np.asarray(h_in, F64)], axis=0)


def state_video(cfg, state, ctx) -> np.ndarray:
    return state if cfg.kind == "wan" else state[ctx.shape[0]:]


def run_block_range(cfg, w, state, mods, ctx, b0, b1) -> np.ndarray:
    """Blocks b0 <= i < b1 applied to a stack state (see stack_state)."""
    grid = cfg.grid
    H = cfg.heads
    x = np.asarray(state, F64)
    L = 0 if cfg.kind == "wan" else ctx.shape[0]
    for i in range(b0, b1):
        wb, m = w["blocks"][i], mods[i]
        if cfg.kind == "wan":
            x = wan_block(x, m, wb, grid, H, ctx=ctx, eps=cfg.ln_eps, theta=cfg.rope_theta)
        elif cfg.kind == "cog":
            x = cog_block(x, m, wb, grid, H, L, eps=cfg.ln_eps, theta=cfg.rope_theta)
        elif i < cfg.n_blocks:  # hv dual-stream
            mv, mt = m
            xt, xv = hv_dual_block(x[:L], x[L:], mt, mv, wb, grid, H, eps=cfg.ln_eps, theta=cfg.rope_theta)
            x = np.concatenate([xt, xv], axis=0)
        else:  # hv single-stream
            x = hv_single_block(x, m, wb, grid, H, L, eps=cfg.ln_eps, theta=cfg.rope_theta)
    return x


def block_stack(cfg, w, h_in, mods, ctx) -> np.ndarray:
    """Run every block on the video tokens h_in (and the text stream for joint
    models); returns the video tokens after the last block."""
    state = run_block_range(cfg, w, stack_state(cfg, h_in, ctx), mods, ctx, 0, len(w["blocks"]))
    return state_video(cfg, state, ctx)


def final_layer(cfg, w, h_out, final_mod) -> np.ndarray:
    """v = unpatchify(W_f LNmod(h_out; shift_f, scale_f) + b_f)."""
    d = cfg.d
    y = modulate(layer_norm(h_out, cfg.ln_eps), final_mod[:d], final_mod[d:])
    return unpatchify(linear(y, *w["final"]), cfg.latent_shape, cfg.pt, cfg.ph, cfg.pw)


def denoiser(cfg, w, x_latent, t, ctx) -> np.ndarray:
    """f_theta(x_t, t, c): the full model evaluation."""
    si = step_inputs(cfg, w, x_latent, t)
    h_out = block_stack(cfg, w, si.h_in, si.mods, ctx)
    return final_layer(cfg, w, h_out, si.final_mod)


@dataclass
class LoopResult:
    latent: np.ndarray
    records: list = field(default_factory=list)

    @property
    def computed(self) -> list[bool]:
        return [r.computed for r in self.records]


class SamplerBranch:
    """One stream of model evaluations inside the sampler, with its own
    Algorithm 1 controller and its own cache of the base method M.  A plain
    generation has one branch; classifier-free guidance has two (conditional
    and unconditional text), which decide and cache independently.

    TeaCache (Sec. 2): s_t = rel_l1(TEMNI_{t-1}, TEMNI_t) between consecutive
    steps (computed or not); M.update stores R = H_out - H_in of the block
    stack; M.reuse gives H_out = H_in + R.
    EasyCache (Sec. 2): s_t = k * mean|x_t - x_{t-1}| / mean|v_{t-1}|;
    M.update refreshes k and the offset v_c - x_c; M.reuse gives
    v_t = x_t + (v_c - x_c).
    DiCache (Sec. 2): the first ``probe_blocks`` blocks run on every step;
    s_t = rel_l1(P_{t-1}, P_t) of the probe features; M.update keeps the probe
    features and deep parts D = H_out - P of the last two computed steps;
    M.reuse is dicache_reuse.
    """

    def __init__(self, cfg, w, text, tau_low, tau_high, delta, warmup, method, probe_blocks=1,
                 signal_poly=None):
        self.cfg, self.w = cfg, w
        self.ctx = text_context(cfg, w, text)
        self.ctl = AcidController(tau_low, tau_high, delta)
        self.warmup, self.method = warmup, method
        self.probe_blocks, self.signal_poly = probe_blocks, signal_poly
        self.temni_prev = self.resid = None
        self.x_prev = self.v_prev = self.x_c = self.v_c = self.k_rate = None
        self.probe_prev = self.p_c1 = self.p_c2 = self.d_c1 = self.d_c2 = None

    def _decide(self, rec, s, f, tf):
        skip, tau, sg, ds = self.ctl.step(s, forced=f, tau_fixed=tf)
        rec.signal, rec.tau, rec.sigma, rec.dsignal = s, tau, sg, ds
        rec.forced = f is not None
        return not skip

    def velocity(self, i, x, si, f=None, tf=None):
        """The model output v at step i for latent x (si = step_inputs of x):
        Algorithm 1 decides compute or reuse; returns (v, StepRecord).
        f: forced decision (None, True, False); tf: fixed threshold or None."""
        cfg, w, ctx, poly = self.cfg, self.w, self.ctx, self.signal_poly
        rec = StepRecord(step=i, warmup=i < self.warmup)
        if self.method == "teacache":
            temni = block0_temni(cfg, w, si.h_in, si.temb)
            compute = True if rec.warmup else \
                self._decide(rec, rescale_signal(rel_l1(self.temni_prev, temni), poly), f, tf)
            self.temni_prev = temni
            if compute:
                h_out = block_stack(cfg, w, si.h_in, si.mods, ctx)
                self.resid = h_out - si.h_in
            else:
                h_out = cache_apply(si.h_in, self.resid)
            v = final_layer(cfg, w, h_out, si.final_mod)
        elif self.method == "easycache":
            compute = True if rec.warmup else \
                self._decide(rec, rescale_signal(easycache_signal(self.k_rate, x, self.x_prev, self.v_prev), poly),
                             f, tf)
            if compute:
                h_out = block_stack(cfg, w, si.h_in, si.mods, ctx)
                v = final_layer(cfg, w, h_out, si.final_mod)
                if self.x_prev is not None:
                    self.k_rate = easycache_rate(x, self.x_prev, v, self.v_prev)
                self.x_c, self.v_c = x, v
            else:
                v = easycache_reuse(x, self.x_c, self.v_c)
            self.x_prev, self.v_prev = x, v
        elif self.method == "dicache":
            # probe: the first probe_blocks blocks, run on every step
            pb = self.probe_blocks
            state = run_block_range(cfg, w, stack_state(cfg, si.h_in, ctx), si.mods, ctx, 0, pb)
            probe = state_video(cfg, state, ctx)
            compute = True if rec.warmup else \
                self._decide(rec, rescale_signal(rel_l1(self.probe_prev, probe), poly), f, tf)
            self.probe_prev = probe
            if compute:
                state = run_block_range(cfg, w, state, si.mods, ctx, pb, len(w["blocks"]))
                h_out = state_video(cfg, state, ctx)
                d_new = h_out - probe
                if self.p_c1 is None:
                    self.p_c2, self.d_c2 = probe, d_new
                else:
                    self.p_c2, self.d_c2 = self.p_c1, self.d_c1
                self.p_c1, self.d_c1 = probe, d_new
            else:
                h_out = dicache_reuse(probe, self.p_c1, self.p_c2, self.d_c1, self.d_c2)
            v = final_layer(cfg, w, h_out, si.final_mod)
        else:
            raise ValueError(self.method)
        rec.computed = compute
        return v, rec


def _loop_args(cfg, n_steps, tau_low, tau_high, delta, warmup, method):
    return (cfg.steps if n_steps is None else n_steps,
            cfg.tau_low if tau_low is None else tau_low,
            cfg.tau_high if tau_high is None else tau_high,
            cfg.delta if delta is None else delta,
            cfg.warmup if warmup is None else warmup,
            cfg.method if method is None else method)


def _step_override(seq, i):
    return None if seq is None else seq[i]


def denoise_loop(cfg, w, latent, text, n_steps=None, tau_low=None, tau_high=None, delta=None,
                 warmup=None, method=None, forced=None, force_last=False, shift=1.0,
                 probe_blocks=1, signal_poly=None, tau_schedule=None) -> LoopResult:
    """The sampling loop of Algorithm 1 (Sec. 3.3) around an Euler
    flow-matching sampler, with TeaCache, EasyCache or DiCache as the base
    method M (one SamplerBranch).

    ``forced``: optional per-step list of None/True/False; True or False
    replaces the controller's decision at that step (compute / skip).
    ``tau_schedule``: optional per-step thresholds (None or NaN: the delta
    rule), see AcidController.
    """
    n_steps, tau_low, tau_high, delta, warmup, method = _loop_args(cfg, n_steps, tau_low, tau_high, delta, warmup,
                                                                   method)
    sig = sigmas(n_steps, shift)
    br = SamplerBranch(cfg, w, text, tau_low, tau_high, delta, warmup, method, probe_blocks, signal_poly)
    x = np.asarray(latent, F64)
    res = LoopResult(latent=x)
    for i in range(n_steps):
        si = step_inputs(cfg, w, x, 1000.0 * sig[i])
        f = _step_override(forced, i)
        if force_last and i == n_steps - 1 and f is None:
            f = True
        v, rec = br.velocity(i, x, si, f, _step_override(tau_schedule, i))
        res.records.append(rec)
        x = euler_step(x, v, sig[i], sig[i + 1])
    res.latent = x
    return res


@dataclass
class GuidedResult:
    latent: np.ndarray
    cond: list = field(default_factory=list)     # StepRecord per step, conditional branch
    uncond: list = field(default_factory=list)   # StepRecord per step, unconditional branch


def guided_velocity(v_cond, v_uncond, scale: float):
    """Classifier-free guidance: v = v_u + g (v_c - v_u)."""
    return v_uncond + scale * (v_cond - v_uncond)


def denoise_loop_guided(cfg, w, latent, text_cond, text_uncond, scale, n_steps=None, tau_low=None, tau_high=None,
                        delta=None, warmup=None, method=None, forced_cond=None, forced_uncond=None,
                        force_last=False, shift=1.0, probe_blocks=1, signal_poly=None,
                        tau_schedule=None) -> GuidedResult:
    """Algorithm 1 with classifier-free guidance: the conditional and the
    unconditional model evaluations are two SamplerBranches, each with its
    own Sigma, s_prev and cache (the paper is silent on guidance; caching
    the branches independently is the reading).  Both branches see the same
    latent x_i and thresholds; the Euler step uses the guided velocity."""
    n_steps, tau_low, tau_high, delta, warmup, method = _loop_args(cfg, n_steps, tau_low, tau_high, delta, warmup,
                                                                   method)
    sig = sigmas(n_steps, shift)
    bc = SamplerBranch(cfg, w, text_cond, tau_low, tau_high, delta, warmup, method, probe_blocks, signal_poly)
    bu = SamplerBranch(cfg, w, text_uncond, tau_low, tau_high, delta, warmup, method, probe_blocks, signal_poly)
    x = np.asarray(latent, F64)
    res = GuidedResult(latent=x)
    for i in range(n_steps):
        si = step_inputs(cfg, w, x, 1000.0 * sig[i])
        tf = _step_override(tau_schedule, i)
        fc, fu = _step_override(forced_cond, i), _step_override(forced_uncond, i)
        if force_last and i == n_steps - 1:
            fc = True if fc is None else fc
            fu = True if fu is None else fu
        vc, rc = bc.velocity(i, x, si, fc, tf)
        vu, ru = bu.velocity(i, x, si, fu, tf)
        res.cond.append(rc)
        res.uncond.append(ru)
        x = euler_step(x, guided_velocity(vc, vu, scale), sig[i], sig[i + 1])
    res.latent = x
    return res

