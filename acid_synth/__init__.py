"""Seeded synthetic inputs shared by the CPU oracle and the CUDA path.

This module holds shapes and random draws only.  It contains none of the
method's arithmetic (no LayerNorm, attention, drift, controller or sampler
step): both sides call it to obtain identical weights, latents, text features
and micro-benchmark tensors, and then compute independently.

Recipe (all draws from ``numpy.random.default_rng``):

* every weight matrix and bias ~ N(0, 0.02^2), one independent stream per
  tensor, keyed by (seed, config, tensor name);
* latents and text features ~ N(0, 1);
* drift micro-benchmark: ``prev ~ N(0, 1)`` of shape [T, 3072] and
  ``cur = prev + sigma * z`` with ``z ~ N(0, 1)``.

The workload shapes are those of the five workloads the method is measured
on: a 2-block fp32 toy DiT, and Wan-2.1-1.3B-, CogVideoX-2B- and
HunyuanVideo-shaped stacks at 480p/720p-class token counts, plus the
[T, 3072] drift micro-benchmark.  The paper evaluates trained checkpoints on
VBench prompts; neither is available, so these seeded stand-ins with the same
shapes and N(0, .) value distributions replace them.
"""

from __future__ import annotations

import zlib
from dataclasses import dataclass, field, replace

import numpy as np

WEIGHT_STD = 0.02


@dataclass(frozen=True)
class DiTConfig:
    """Shape description of one DiT workload."""

    name: str
    kind: str  # "wan" (incl. toy), "cog" (joint, shared weights), "hv" (dual + single)
    dtype: str  # "fp32" or "bf16"
    d: int
    heads: int
    ffn: int
    n_blocks: int  # wan / cog: block count; hv: dual-stream blocks
    n_single: int = 0  # hv: single-stream blocks
    latent_c: int = 16
    latent_f: int = 4
    latent_h: int = 16
    latent_w: int = 16
    pt: int = 1
    ph: int = 2
    pw: int = 2
    n_text: int = 0  # wan: cross-attention context tokens; cog/hv: joint text tokens
    d_text: int = 0  # width of the raw text features
    steps: int = 10
    method: str = "teacache"  # "teacache" or "easycache"
    tau_low: float = 0.05
    tau_high: float = 0.2
    delta: float = 0.01
    time_freq_dim: int = 256
    rope_theta: float = 10000.0
    ln_eps: float = 1e-6

    @property
    def head_dim(self) -> int:
        return self.d // self.heads

    @property
    def grid(self) -> tuple[int, int, int]:
        return (self.latent_f // self.pt, self.latent_h // self.ph, self.latent_w // self.pw)

    @property
    def n_video(self) -> int:
        f, h, w = self.grid
        return f * h * w

    @property
    def patch_dim(self) -> int:
        return self.latent_c * self.pt * self.ph * self.pw

    @property
    def latent_shape(self) -> tuple[int, int, int, int]:
        return (self.latent_c, self.latent_f, self.latent_h, self.latent_w)

    @property
    def warmup(self) -> int:
        # TeaCache needs one computed step to define the previous modulated
        # input; EasyCache needs two to define its transformation rate k.
        return 2 if self.method == "easycache" else 1


CONFIGS: dict[str, DiTConfig] = {
    # 2 blocks, d=256, 4 heads of 64, MLP 1024; latent 16 x 4 x 16 x 16 -> 4 x 8 x 8 = 256 tokens.
    "toy": DiTConfig(name="toy", kind="wan", dtype="fp32", d=256, heads=4, ffn=1024, n_blocks=2,
                     latent_f=4, latent_h=16, latent_w=16, n_text=0, d_text=0, steps=10,
                     method="teacache", tau_low=0.05, tau_high=0.2),
    # 480x832, 81 frames, VAE 4x8x8 -> latent 16 x 21 x 60 x 104 -> 21 x 30 x 52 = 32760 tokens.
    "wan": DiTConfig(name="wan", kind="wan", dtype="bf16", d=1536, heads=12, ffn=8960, n_blocks=30,
                     latent_f=21, latent_h=60, latent_w=104, n_text=512, d_text=4096, steps=50,
                     method="teacache", tau_low=0.05, tau_high=0.2),
    # 480x720, 49 frames -> latent 16 x 13 x 60 x 90 -> 13 x 30 x 45 = 17550 video + 226 text tokens.
    "cog": DiTConfig(name="cog", kind="cog", dtype="bf16", d=1920, heads=30, ffn=7680, n_blocks=30,
                     latent_f=13, latent_h=60, latent_w=90, n_text=226, d_text=1920, steps=50,
                     method="easycache", tau_low=0.02, tau_high=0.04),
    # 544x960, 129 frames -> latent 16 x 33 x 68 x 120 -> 33 x 34 x 60 = 67320 video + 256 text tokens.
    "hv": DiTConfig(name="hv", kind="hv", dtype="bf16", d=3072, heads=24, ffn=12288, n_blocks=20,
                    n_single=40, latent_f=33, latent_h=68, latent_w=120, n_text=256, d_text=3072,
                    steps=50, method="teacache", tau_low=0.1, tau_high=0.3),
}

MICRO_T = (4096, 32760, 67320, 118800)
MICRO_D = 3072
MICRO_SIGMA = (1e-3, 1e-2, 1e-1)


def get_config(name: str, **overrides) -> DiTConfig:
    cfg = CONFIGS[name]
    return replace(cfg, **overrides) if overrides else cfg


def _rng(seed: int, *key) -> np.random.Generator:
    tag = zlib.crc32("/".join(str(k) for k in key).encode())
    return np.random.default_rng([int(seed), tag])


def normal(seed: int, shape, std: float = 1.0, *key) -> np.ndarray:
    """fp32 array ~ N(0, std^2) from an independent stream keyed by ``key``."""
    a = _rng(seed, *key).standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        a *= np.float32(std)
    return a


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even), returned as fp32.

    Used so that both sides consume exactly the values stored on the device
    in bf16 mode; it is an input conversion, not part of the method.
    """
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).reshape(a.shape)


# ----------------------------------------------------------------------------
# Weight tensors.  Layout: every matrix is [out, in] (row-major, the
# nn.Linear convention); every bias is [out].
# ----------------------------------------------------------------------------

def _lin(seed, cfg_name, name, n_out, n_in, prepare):
    w = prepare(normal(seed, (n_out, n_in), WEIGHT_STD, cfg_name, name, "w"))
    b = normal(seed, (n_out,), WEIGHT_STD, cfg_name, name, "b")
    return w, b


def stream_weight_shapes(cfg: DiTConfig) -> dict[str, tuple[int, int]]:
    """[out, in] of every linear layer of one stream of one block."""
    d, f = cfg.d, cfg.ffn
    return {"mod": (6 * d, d), "qkv": (3 * d, d), "o": (d, d), "ff1": (f, d), "ff2": (d, f)}


def block_weights(cfg: DiTConfig, index: int, seed: int = 0, block_type: str | None = None,
                  bf16: bool | None = None, q_scale: float = 1.0, zero: tuple[str, ...] = ()) -> dict:
    """Weights of one block.

    ``block_type``: "wan" | "cog" | "hv_dual" | "hv_single" (defaults from cfg.kind).
    ``q_scale`` multiplies the query rows of the QKV matrix (a "peaky" attention
    variant used by the tests so that softmax is far from flat).
    ``zero`` lists layer names whose weight and bias are set to zero.
    Returns {name: (w, b)}; w is fp32, already bf16-rounded in bf16 mode.
    """
    d = cfg.d
    bt = block_type or ("hv_dual" if cfg.kind == "hv" else cfg.kind)
    use_bf16 = (cfg.dtype == "bf16") if bf16 is None else bf16
    prep = round_to_bf16 if use_bf16 else (lambda x: x)
    tag = f"{cfg.name}/{bt}{index}"
    out: dict[str, tuple[np.ndarray, np.ndarray]] = {}

    def lin(name, n_out, n_in):
        w, b = _lin(seed, tag, name, n_out, n_in, lambda x: x)
        if name in zero or name.split(".")[-1] in zero:
            w = np.zeros_like(w)
            b = np.zeros_like(b)
        out[name] = (w, b)

    if bt == "wan":
        for k, (o, i) in stream_weight_shapes(cfg).items():
            lin(k, o, i)
        if cfg.n_text > 0:
            lin("cq", d, d)
            lin("ckv", 2 * d, d)
            lin("co", d, d)
    elif bt == "cog":
        shapes = stream_weight_shapes(cfg)
        shapes["mod"] = (12 * d, d)  # video 6d followed by text 6d
        for k, (o, i) in shapes.items():
            lin(k, o, i)
    elif bt == "hv_dual":
        for stream in ("vid", "txt"):
            for k, (o, i) in stream_weight_shapes(cfg).items():
                lin(f"{stream}.{k}", o, i)
    elif bt == "hv_single":
        lin("mod", 3 * d, d)
        lin("qkv", 3 * d, d)
        lin("mlp", cfg.ffn, d)
        lin("w2", d, d + cfg.ffn)
    else:
        raise ValueError(bt)

    if q_scale != 1.0:
        for name in list(out):
            if name.endswith("qkv"):
                w, b = out[name]
                w = w.copy()
                b = b.copy()
                w[:d] *= np.float32(q_scale)
                b[:d] *= np.float32(q_scale)
                out[name] = (w, b)
    return {k: (prep(w), b) for k, (w, b) in out.items()}


def model_weights(cfg: DiTConfig, seed: int = 0, blocks: bool = True) -> dict:
    """All weights of a DiT: patch embedding, time MLP, text projection,
    blocks and final layer."""
    d = cfg.d
    prep = round_to_bf16 if cfg.dtype == "bf16" else (lambda x: x)
    m: dict = {}

    def lin(name, n_out, n_in):
        w, b = _lin(seed, cfg.name, name, n_out, n_in, prep)
        m[name] = (w, b)

    lin("patch", d, cfg.patch_dim)
    lin("time1", d, cfg.time_freq_dim)
    lin("time2", d, d)
    if cfg.kind == "wan" and cfg.n_text > 0:
        lin("text", d, cfg.d_text)
    lin("final_mod", 2 * d, d)
    lin("final", cfg.patch_dim, d)
    if blocks:
        if cfg.kind == "hv":
            m["blocks"] = [block_weights(cfg, i, seed, "hv_dual") for i in range(cfg.n_blocks)]
            m["blocks"] += [block_weights(cfg, i, seed, "hv_single") for i in range(cfg.n_single)]
        else:
            m["blocks"] = [block_weights(cfg, i, seed) for i in range(cfg.n_blocks)]
    return m


# ----------------------------------------------------------------------------
# Activations and inputs.
# ----------------------------------------------------------------------------

def latent(cfg: DiTConfig, seed: int = 0) -> np.ndarray:
    """Initial noise latent [C, F, H, W] ~ N(0, 1)."""
    a = normal(seed, cfg.latent_shape, 1.0, cfg.name, "latent")
    return round_to_bf16(a) if cfg.dtype == "bf16" else a


def text(cfg: DiTConfig, seed: int = 0) -> np.ndarray | None:
    """Raw text features [n_text, d_text] ~ N(0, 1) (None without text)."""
    if cfg.n_text == 0:
        return None
    a = normal(seed, (cfg.n_text, cfg.d_text), 1.0, cfg.name, "text")
    return round_to_bf16(a) if cfg.dtype == "bf16" else a


def hidden(cfg: DiTConfig, n_rows: int, seed: int = 0, tag: str = "hidden") -> np.ndarray:
    """A block input [n_rows, d] ~ N(0, 1)."""
    a = normal(seed, (n_rows, cfg.d), 1.0, cfg.name, tag)
    return round_to_bf16(a) if cfg.dtype == "bf16" else a


def temb_vector(cfg: DiTConfig, seed: int = 0) -> np.ndarray:
    """A stand-in timestep embedding [d] ~ N(0, 1), fp32 (block-level tests)."""
    return normal(seed, (cfg.d,), 1.0, cfg.name, "temb")


def micro_pair(t_rows: int, sigma: float, seed: int = 0, d: int = MICRO_D,
               bf16: bool = True) -> tuple[np.ndarray, np.ndarray]:
    """Drift micro-benchmark pair: prev ~ N(0,1) [T, d]; cur = prev + sigma * z."""
    prev = normal(seed, (t_rows, d), 1.0, "micro", t_rows, "prev")
    z = normal(seed, (t_rows, d), 1.0, "micro", t_rows, sigma, "z")
    cur = prev + np.float32(sigma) * z
    if bf16:
        return round_to_bf16(prev), round_to_bf16(cur)
    return prev, cur


def micro_residual(t_rows: int, seed: int = 0, d: int = MICRO_D, bf16: bool = True) -> np.ndarray:
    r = normal(seed, (t_rows, d), 0.1, "micro", t_rows, "residual")
    return round_to_bf16(r) if bf16 else r
