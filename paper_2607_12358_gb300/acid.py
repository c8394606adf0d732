"""Python binding of the ACID C ABI (include/acid.h).

Argument marshalling only: every function below turns torch tensors into
device pointers, sizes and the current CUDA stream, calls the entry point of
the same name in libacid_gb300.so and raises on a non-zero status.  Device
memory (outputs, workspaces, weights) is allocated with torch, as the C ABI
leaves all allocation to the caller.
"""

from __future__ import annotations

import ctypes as C
import math
from dataclasses import dataclass, field

import numpy as np
import torch

from . import _capi as A
from ._capi import check, load

_DT = {torch.bfloat16: A.ACID_BF16, torch.float32: A.ACID_FP32}
_TORCH_DT = {A.ACID_BF16: torch.bfloat16, A.ACID_FP32: torch.float32}
_KIND = {"wan": A.ACID_BLOCK_WAN, "cog": A.ACID_BLOCK_COG, "hv_dual": A.ACID_BLOCK_HV_DUAL,
         "hv_single": A.ACID_BLOCK_HV_SINGLE}


def _dtype(t: torch.Tensor) -> int:
    if t.dtype not in _DT:
        raise TypeError(f"unsupported dtype {t.dtype}")
    return _DT[t.dtype]


def _stream(stream=None) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def _need_cuda(*ts):
    for t in ts:
        if t is not None and not t.is_cuda:
            raise ValueError("tensor must be on a CUDA device")


def version() -> str:
    return load().acid_version().decode()


def check_device_error() -> None:
    check(load().acid_check_device_error())


def selftest_wait_timeout(budget_cycles: int, stream=None) -> None:
    """Runs the failure-path diagnostic (a bounded wait that runs out); the next
    check_device_error() raises with ACID_ERR_TIMEOUT."""
    check(load().acid_selftest_wait_timeout(int(budget_cycles), _stream(stream)))


def bounds_report() -> dict:
    """The first kernel memory-index violation recorded since the last report
    (debug build only; ``checked`` is False in the release build)."""
    c, site, idx, ext = C.c_int32(), C.c_int64(), C.c_int64(), C.c_int64()
    check(load().acid_bounds_report(C.byref(c), C.byref(site), C.byref(idx), C.byref(ext)))
    return {"checked": bool(c.value), "site": site.value, "index": idx.value, "extent": ext.value}


def selftest_bounds(stream=None) -> None:
    """Evaluates one index check one past the end (no access behind it); the
    debug build's next bounds_report() shows site 99."""
    check(load().acid_selftest_bounds(_stream(stream)))


def launch_count() -> int:
    return int(load().acid_launch_count())


PROF_ATTENTION, PROF_LINEAR, PROF_DRIFT = 0, 1, 2


def profile_enable(on: bool = True) -> None:
    check(load().acid_profile_enable(int(bool(on))))


def profile_read(kind: int) -> tuple[int, float, float]:
    """(launches, total device ms, total algorithmic work) of one launch kind."""
    n, ms, wk = C.c_int64(), C.c_double(), C.c_double()
    check(load().acid_profile_read(int(kind), C.byref(n), C.byref(ms), C.byref(wk)))
    return n.value, ms.value, wk.value


# ---------------------------------------------------------------------------
# drift signal and cache apply
# ---------------------------------------------------------------------------

def drift_workspace_size(n: int) -> int:
    b = C.c_size_t()
    check(load().acid_drift_workspace_size(int(n), C.byref(b)))
    return b.value


def acid_drift_signal(prev: torch.Tensor, cur: torch.Tensor, out_rel: torch.Tensor | None = None,
                      out_sums: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                      stream=None):
    """rel_l1 = sum|cur - prev| / sum|prev| (device fp64 tensors [1] and [2])."""
    _need_cuda(prev, cur)
    if prev.dtype != cur.dtype or prev.numel() != cur.numel():
        raise ValueError("prev and cur must have the same dtype and size")
    n = prev.numel()
    dev = prev.device
    out_rel = torch.empty(1, dtype=torch.float64, device=dev) if out_rel is None else out_rel
    out_sums = torch.empty(2, dtype=torch.float64, device=dev) if out_sums is None else out_sums
    ws = torch.empty(drift_workspace_size(n), dtype=torch.uint8, device=dev) if workspace is None else workspace
    check(load().acid_drift_signal(prev.data_ptr(), cur.data_ptr(), n, _dtype(prev), out_rel.data_ptr(),
                                   out_sums.data_ptr(), ws.data_ptr(), ws.numel(), _stream(stream)))
    return out_rel, out_sums


def acid_temni_drift(h_prev: torch.Tensor, h_cur: torch.Tensor, mod_prev: torch.Tensor, mod_cur: torch.Tensor,
                     eps: float = 1e-6, out_rel: torch.Tensor | None = None, out_sums: torch.Tensor | None = None,
                     workspace: torch.Tensor | None = None, stream=None):
    """rel_l1(TEMNI_prev, TEMNI_cur) with TEMNI = LN(h) (1 + scale) + shift from
    fp32 h [rows, d] and mod = [shift | scale] fp32 [2d] of each step."""
    _need_cuda(h_prev, h_cur, mod_prev, mod_cur)
    for t in (h_prev, h_cur, mod_prev, mod_cur):
        if t.dtype != torch.float32 or not t.is_contiguous():
            raise ValueError("temni_drift inputs must be contiguous fp32")
    rows, d = h_cur.shape
    if h_prev.shape != h_cur.shape or mod_prev.numel() != 2 * d or mod_cur.numel() != 2 * d:
        raise ValueError("temni_drift: shape mismatch")
    dev = h_cur.device
    out_rel = torch.empty(1, dtype=torch.float64, device=dev) if out_rel is None else out_rel
    out_sums = torch.empty(2, dtype=torch.float64, device=dev) if out_sums is None else out_sums
    ws = torch.empty(drift_workspace_size(rows * d), dtype=torch.uint8, device=dev) if workspace is None else workspace
    check(load().acid_temni_drift(h_prev.data_ptr(), h_cur.data_ptr(), mod_prev.data_ptr(), mod_cur.data_ptr(), rows,
                                  d, float(eps), out_rel.data_ptr(), out_sums.data_ptr(), ws.data_ptr(), ws.numel(),
                                  _stream(stream)))
    return out_rel, out_sums


def acid_cache_apply(x: torch.Tensor, cached_residual: torch.Tensor, out: torch.Tensor | None = None,
                     stream=None) -> torch.Tensor:
    """out = x + cached_residual."""
    _need_cuda(x, cached_residual)
    out = torch.empty_like(x) if out is None else out
    check(load().acid_cache_apply(x.data_ptr(), cached_residual.data_ptr(), out.data_ptr(), x.numel(),
                                  _dtype(x), _stream(stream)))
    return out


def acid_drift_apply(prev, cur, cached_residual, out=None, out_rel=None, out_sums=None, workspace=None,
                     stream=None):
    """Fused: rel_l1(prev, cur) and out = cur + cached_residual in one pass."""
    _need_cuda(prev, cur, cached_residual)
    n = prev.numel()
    dev = prev.device
    out = torch.empty_like(cur) if out is None else out
    out_rel = torch.empty(1, dtype=torch.float64, device=dev) if out_rel is None else out_rel
    out_sums = torch.empty(2, dtype=torch.float64, device=dev) if out_sums is None else out_sums
    ws = torch.empty(drift_workspace_size(n), dtype=torch.uint8, device=dev) if workspace is None else workspace
    check(load().acid_drift_apply(prev.data_ptr(), cur.data_ptr(), cached_residual.data_ptr(), out.data_ptr(), n,
                                  _dtype(prev), out_rel.data_ptr(), out_sums.data_ptr(), ws.data_ptr(),
                                  ws.numel(), _stream(stream)))
    return out, out_rel, out_sums


# ---------------------------------------------------------------------------
# kernel-level entry points
# ---------------------------------------------------------------------------

_EPI = {"bias": A.ACID_EPI_BIAS, "gelu": A.ACID_EPI_GELU, "gated_res": A.ACID_EPI_GATED_RES, "res": A.ACID_EPI_RES}


def acid_linear_forward(a: torch.Tensor, w: torch.Tensor, bias: torch.Tensor | None = None, epilogue: str = "bias",
                        gate: torch.Tensor | None = None, residual: torch.Tensor | None = None,
                        out: torch.Tensor | None = None, out_fp32: bool = False, stream=None) -> torch.Tensor:
    """out = epilogue(a @ w.T + bias); a [M, K] (row stride a.stride(0)), w [N, K]."""
    _need_cuda(a, w, bias, gate, residual, out)
    M, K = a.shape
    N = w.shape[0]
    if out is None:
        odt = torch.float32 if (out_fp32 or a.dtype == torch.float32) else a.dtype
        out = torch.empty(M, N, dtype=odt, device=a.device)
    check(load().acid_linear_forward(_dtype(a), a.data_ptr(), a.stride(0), M, K, w.data_ptr(), _ptr(bias), N,
                                     out.data_ptr(), out.stride(0), _EPI[epilogue], _ptr(gate), _ptr(residual),
                                     0 if residual is None else residual.stride(0), int(out_fp32), _stream(stream)))
    return out


def attention_workspace_size(head_dim: int) -> int:
    b = C.c_size_t()
    check(load().acid_attention_workspace_size(int(head_dim), C.byref(b)))
    return b.value


def acid_attention_forward(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, heads: int,
                           out: torch.Tensor | None = None, workspace: torch.Tensor | None = None,
                           stream=None) -> torch.Tensor:
    """softmax(q k^T / sqrt(Dh)) v per head; q [nq, H*Dh], k/v [nk, H*Dh] (row strides taken from the tensors).
    ``workspace`` (optional, attention_workspace_size bytes) enables the split of a partial last wave for key
    ranges of more than 8 key tiles; shorter ones run on persistent CTAs and leave it unused."""
    _need_cuda(q, k, v, out, workspace)
    nq, nk = q.shape[0], k.shape[0]
    hd = q.shape[1] // heads
    out = torch.empty(nq, heads * hd, dtype=q.dtype, device=q.device) if out is None else out
    check(load().acid_attention_forward(_dtype(q), q.data_ptr(), q.stride(0), k.data_ptr(), k.stride(0),
                                        v.data_ptr(), v.stride(0), out.data_ptr(), out.stride(0), nq, nk, heads, hd,
                                        _ptr(workspace), 0 if workspace is None else workspace.numel(),
                                        _stream(stream)))
    return out


def acid_layernorm_mod(x: torch.Tensor, shift: torch.Tensor | None = None, scale: torch.Tensor | None = None,
                       eps: float = 1e-6, out_dtype=None, stream=None, out: torch.Tensor | None = None) -> torch.Tensor:
    """y = LN(x) * (1 + scale) + shift over the last axis of x [rows, d]
    (written into `out` when given: same shape, dtype out_dtype or x's)."""
    _need_cuda(x, shift, scale, out)
    y = torch.empty(x.shape, dtype=out_dtype or x.dtype, device=x.device) if out is None else out
    if y.shape != x.shape or not y.is_contiguous():
        raise ValueError("out must be contiguous with the shape of x")
    check(load().acid_layernorm_mod(_dtype(x), x.data_ptr(), _dtype(y), y.data_ptr(), x.shape[0], x.shape[1],
                                    _ptr(shift), _ptr(scale), eps, _stream(stream)))
    return y


# ---------------------------------------------------------------------------
# blocks
# ---------------------------------------------------------------------------

def block_desc(cfg, block_type: str) -> A.acid_block_desc:
    """C descriptor of one block of a workload (cfg: acid_synth.DiTConfig-like)."""
    f, h, w = cfg.grid
    return A.acid_block_desc(kind=_KIND[block_type], dtype=A.ACID_BF16 if cfg.dtype == "bf16" else A.ACID_FP32,
                             d=cfg.d, heads=cfg.heads, ffn=cfg.ffn, grid_f=f, grid_h=h, grid_w=w,
                             n_text=cfg.n_text, rope_theta=cfg.rope_theta, ln_eps=cfg.ln_eps)


def block_rows(desc: A.acid_block_desc) -> int:
    r = C.c_int64()
    check(load().acid_block_rows(C.byref(desc), C.byref(r)))
    return r.value


def block_workspace_size(desc: A.acid_block_desc) -> int:
    b = C.c_size_t()
    check(load().acid_block_workspace_size(C.byref(desc), C.byref(b)))
    return b.value


_FIELD_MAP = {
    "wan": {"mod": "mod", "qkv": "qkv", "o": "o", "ff1": "ff1", "ff2": "ff2", "cq": "cq", "ckv": "ckv", "co": "co"},
    "cog": {"mod": "mod", "qkv": "qkv", "o": "o", "ff1": "ff1", "ff2": "ff2"},
    "hv_dual": {"vid.mod": "mod", "vid.qkv": "qkv", "vid.o": "o", "vid.ff1": "ff1", "vid.ff2": "ff2",
                "txt.mod": "t_mod", "txt.qkv": "t_qkv", "txt.o": "t_o", "txt.ff1": "t_ff1", "txt.ff2": "t_ff2"},
    "hv_single": {"mod": "mod", "qkv": "qkv", "mlp": "ff1", "w2": "ff2"},
}


def _upload_linear(w: np.ndarray, b: np.ndarray | None, wdtype, device):
    tw = torch.from_numpy(np.ascontiguousarray(w)).to(device=device, dtype=wdtype)
    tb = None if b is None else torch.from_numpy(np.ascontiguousarray(b, dtype=np.float32)).to(device)
    return tw, tb


@dataclass
class DeviceBlock:
    """Device copies of one block's weights and the C struct pointing at them."""
    block_type: str
    tensors: dict = field(default_factory=dict)
    struct: A.acid_block_weights = field(default_factory=A.acid_block_weights)

    @classmethod
    def upload(cls, weights: dict, block_type: str, wdtype, device="cuda") -> "DeviceBlock":
        blk = cls(block_type)
        for src, dst in _FIELD_MAP[block_type].items():
            if src not in weights:
                continue
            tw, tb = _upload_linear(*weights[src], wdtype, device)
            blk.tensors[dst] = (tw, tb)
            setattr(blk.struct, dst, A.acid_linear(tw.data_ptr(), _ptr(tb)))
        return blk


def acid_dit_block_forward(desc: A.acid_block_desc, x: torch.Tensor, temb: torch.Tensor,
                           block: DeviceBlock, ctx: torch.Tensor | None = None,
                           workspace: torch.Tensor | None = None, stream=None,
                           ctx_kv: torch.Tensor | None = None) -> torch.Tensor:
    """One block in place on x [rows, d]; temb fp32 [d]; ctx [n_text, d] (WAN);
    ctx_kv [n_text, 2d] (WAN, optional): the block's cross-attention keys and
    values computed ahead, used instead of projecting ctx."""
    _need_cuda(x, temb, ctx, ctx_kv)
    if workspace is None:
        workspace = torch.empty(block_workspace_size(desc) + 1024, dtype=torch.uint8, device=x.device)
    base = workspace.data_ptr()
    aligned = (base + 1023) // 1024 * 1024
    cond = A.acid_cond(temb.data_ptr(), _ptr(ctx), _ptr(ctx_kv))
    check(load().acid_dit_block_forward(C.byref(desc), x.data_ptr(), C.byref(cond), C.byref(block.struct),
                                        aligned, workspace.numel() - (aligned - base), _stream(stream)))
    return x


# ---------------------------------------------------------------------------
# whole model and the step loop
# ---------------------------------------------------------------------------

class DeviceModel:
    """Device weights of a DiT (from acid_synth.model_weights) and its acid_model struct."""

    def __init__(self, cfg, weights: dict, device="cuda"):
        self.cfg = cfg
        self.device = torch.device(device)
        wdtype = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
        self.wdtype = wdtype
        types = (["hv_dual"] * cfg.n_blocks + ["hv_single"] * cfg.n_single) if cfg.kind == "hv" \
            else [cfg.kind] * cfg.n_blocks
        self.blocks = [DeviceBlock.upload(wb, bt, wdtype, device) for wb, bt in zip(weights["blocks"], types)]
        self._block_array = (A.acid_block_weights * len(self.blocks))(*[b.struct for b in self.blocks])
        self.tensors = {}
        m = A.acid_model()
        m.block = block_desc(cfg, types[0])
        m.n_blocks = cfg.n_blocks
        m.n_single = cfg.n_single
        m.blocks = C.cast(self._block_array, C.POINTER(A.acid_block_weights))
        m.latent_c, m.latent_f, m.latent_h, m.latent_w = cfg.latent_shape
        m.pt, m.ph, m.pw = cfg.pt, cfg.ph, cfg.pw
        m.time_freq_dim = cfg.time_freq_dim
        m.d_text = cfg.d_text if cfg.kind == "wan" else cfg.d
        for name, fld in (("patch", "patch"), ("time1", "time1"), ("time2", "time2"), ("text", "text"),
                          ("final_mod", "final_mod"), ("final", "final_out")):
            if name in weights:
                tw, tb = _upload_linear(*weights[name], wdtype, device)
                self.tensors[name] = (tw, tb)
                setattr(m, fld, A.acid_linear(tw.data_ptr(), _ptr(tb)))
        self.struct = m

    def workspace_size(self) -> int:
        b = C.c_size_t()
        check(load().acid_loop_workspace_size(C.byref(self.struct), C.byref(b)))
        return b.value


_METHOD = {"teacache": A.ACID_METHOD_TEACACHE, "easycache": A.ACID_METHOD_EASYCACHE, "dicache": A.ACID_METHOD_DICACHE}


def loop_cfg(cfg, n_steps=None, tau_low=None, tau_high=None, delta=None, warmup=None, method=None,
             force_last=False, shift=1.0, forced=None, probe_blocks=1, signal_poly=None, tau_schedule=None):
    """acid_loop_cfg from a workload config; returns (struct, keepalive)."""
    method = cfg.method if method is None else method
    c = A.acid_loop_cfg()
    c.n_steps = cfg.steps if n_steps is None else n_steps
    c.warmup = (2 if method == "easycache" else 1) if warmup is None else warmup
    c.method = _METHOD[method]
    c.probe_blocks = probe_blocks
    c.force_last = int(bool(force_last))
    c.tau_low = cfg.tau_low if tau_low is None else tau_low
    c.tau_high = cfg.tau_high if tau_high is None else tau_high
    c.delta = cfg.delta if delta is None else delta
    c.shift = shift
    keep = []
    if forced is not None:
        fk = (C.c_int8 * c.n_steps)(*[-1 if f is None else int(bool(f)) for f in forced])
        c.forced = C.cast(fk, C.POINTER(C.c_int8))
        keep.append(fk)
    if signal_poly is not None:
        pk = (C.c_double * len(signal_poly))(*[float(x) for x in signal_poly])
        c.signal_poly_n = len(signal_poly)
        c.signal_poly = C.cast(pk, C.POINTER(C.c_double))
        keep.append(pk)
    if tau_schedule is not None:
        if len(tau_schedule) != c.n_steps:
            raise ValueError("tau_schedule needs one entry per step")
        tk = (C.c_double * c.n_steps)(*[math.nan if x is None else float(x) for x in tau_schedule])
        c.tau_schedule = C.cast(tk, C.POINTER(C.c_double))
        keep.append(tk)
    return c, keep


def _aligned_ws(nbytes: int, device) -> tuple[torch.Tensor, int, int]:
    ws = torch.empty(nbytes + 1024, dtype=torch.uint8, device=device)
    base = ws.data_ptr()
    a = (base + 1023) // 1024 * 1024
    return ws, a, ws.numel() - (a - base)


class Loop:
    """A generation driven step by step: acid_loop_begin + acid_denoise_step."""

    def __init__(self, model: DeviceModel, cfg_struct, text: torch.Tensor | None, device="cuda", stream=None):
        self.model = model
        self.cfg = cfg_struct
        self.ws, self.ws_ptr, self.ws_bytes = _aligned_ws(model.workspace_size(), device)
        self.state = A.acid_loop_state()
        self.text = text
        self.stream = stream
        check(load().acid_loop_begin(C.byref(model.struct), C.byref(cfg_struct), _ptr(text), C.byref(self.state),
                                     self.ws_ptr, self.ws_bytes, _stream(stream)))

    def step(self, latent: torch.Tensor, log: bool = True):
        lg = A.acid_step_log()
        check(load().acid_denoise_step(C.byref(self.model.struct), C.byref(self.cfg), C.byref(self.state),
                                       latent.data_ptr(), C.byref(lg) if log else None, self.ws_ptr, self.ws_bytes,
                                       _stream(self.stream)))
        return lg if log else None

    def checkpoint(self) -> dict:
        """The generation's resumable state: a copy of the controller struct and
        of the loop workspace (caches, text context, RoPE table).  Together with
        the latent it restores the generation exactly (Loop.restore)."""
        st = A.acid_loop_state()
        C.memmove(C.byref(st), C.byref(self.state), C.sizeof(st))
        n = self.model.workspace_size()
        off = self.ws_ptr - self.ws.data_ptr()
        return {"state": st, "workspace": self.ws[off:off + n].clone()}

    @classmethod
    def restore(cls, model: DeviceModel, cfg_struct, ckpt: dict, device="cuda", stream=None) -> "Loop":
        """A Loop that continues a checkpointed generation in a fresh workspace."""
        obj = cls.__new__(cls)
        obj.model, obj.cfg, obj.text, obj.stream = model, cfg_struct, None, stream
        obj.ws, obj.ws_ptr, obj.ws_bytes = _aligned_ws(model.workspace_size(), device)
        n = ckpt["workspace"].numel()
        off = obj.ws_ptr - obj.ws.data_ptr()
        obj.ws[off:off + n].copy_(ckpt["workspace"])
        obj.state = A.acid_loop_state()
        C.memmove(C.byref(obj.state), C.byref(ckpt["state"]), C.sizeof(obj.state))
        return obj


def log_to_dict(lg: A.acid_step_log) -> dict:
    return {k: getattr(lg, k) for k, _ in A.acid_step_log._fields_}


def acid_denoise_loop(model: DeviceModel, cfg_struct, latent: torch.Tensor, text: torch.Tensor | None = None,
                      log: bool = True, workspace=None, stream=None, graph: bool = False) -> list[dict]:
    """Runs all steps in place on latent (fp32 [C, F, H, W]); returns the step log.
    ``graph=True`` calls acid_denoise_loop_graph (the whole generation as one CUDA graph)."""
    _need_cuda(latent, text)
    if latent.dtype != torch.float32:
        raise TypeError("latent must be fp32")
    n = cfg_struct.n_steps
    logs = (A.acid_step_log * n)()
    ws, ptr, nbytes = _aligned_ws(model.workspace_size(), latent.device) if workspace is None else workspace
    fn = load().acid_denoise_loop_graph if graph else load().acid_denoise_loop
    check(fn(C.byref(model.struct), C.byref(cfg_struct), latent.data_ptr(), _ptr(text), logs if log else None, ptr,
             nbytes, _stream(stream)))
    return [log_to_dict(x) for x in logs] if log else []


# ---------------------------------------------------------------------------
# classifier-free guidance: two independently cached branches
# ---------------------------------------------------------------------------

def guided_workspace_size(model: DeviceModel) -> int:
    b = C.c_size_t()
    check(load().acid_guided_workspace_size(C.byref(model.struct), C.byref(b)))
    return b.value


class GuidedLoop:
    """A guided generation driven step by step: acid_guided_begin + acid_guided_step."""

    def __init__(self, model: DeviceModel, cfg_cond, cfg_uncond, scale: float, text_cond, text_uncond,
                 device="cuda", stream=None):
        self.model, self.cfg_c, self.cfg_u, self.scale = model, cfg_cond, cfg_uncond, float(scale)
        self.ws, self.ws_ptr, self.ws_bytes = _aligned_ws(guided_workspace_size(model), device)
        self.st_c, self.st_u = A.acid_loop_state(), A.acid_loop_state()
        self.texts = (text_cond, text_uncond)
        self.stream = stream
        check(load().acid_guided_begin(C.byref(model.struct), C.byref(cfg_cond), C.byref(cfg_uncond),
                                       _ptr(text_cond), _ptr(text_uncond), C.byref(self.st_c), C.byref(self.st_u),
                                       self.ws_ptr, self.ws_bytes, _stream(stream)))

    def step(self, latent: torch.Tensor, log: bool = True):
        lc, lu = A.acid_step_log(), A.acid_step_log()
        check(load().acid_guided_step(C.byref(self.model.struct), C.byref(self.cfg_c), C.byref(self.cfg_u),
                                      self.scale, C.byref(self.st_c), C.byref(self.st_u), latent.data_ptr(),
                                      C.byref(lc) if log else None, C.byref(lu) if log else None, self.ws_ptr,
                                      self.ws_bytes, _stream(self.stream)))
        return (lc, lu) if log else None


def acid_denoise_loop_guided(model: DeviceModel, cfg_cond, cfg_uncond, scale: float, latent: torch.Tensor,
                             text_cond: torch.Tensor | None = None, text_uncond: torch.Tensor | None = None,
                             log: bool = True, stream=None, graph: bool = False) -> tuple[list[dict], list[dict]]:
    """Runs a guided generation in place on latent; returns the two branches' step logs.
    ``graph=True`` calls acid_denoise_loop_guided_graph (one CUDA graph, decisions on the device)."""
    _need_cuda(latent, text_cond, text_uncond)
    if latent.dtype != torch.float32:
        raise TypeError("latent must be fp32")
    n = cfg_cond.n_steps
    lc, lu = (A.acid_step_log * n)(), (A.acid_step_log * n)()
    ws, ptr, nbytes = _aligned_ws(guided_workspace_size(model), latent.device)
    fn = load().acid_denoise_loop_guided_graph if graph else load().acid_denoise_loop_guided
    check(fn(C.byref(model.struct), C.byref(cfg_cond), C.byref(cfg_uncond), float(scale), latent.data_ptr(),
             _ptr(text_cond), _ptr(text_uncond), lc if log else None, lu if log else None, ptr, nbytes,
             _stream(stream)))
    return ([log_to_dict(x) for x in lc], [log_to_dict(x) for x in lu]) if log else ([], [])
