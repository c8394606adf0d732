"""Times one kernel of the library at a chosen shape (CUDA events, after
warm-up), for tuning and for profiler captures of a single launch.

    python -m paper_2607_12358_gb300.kernel_bench attention --n 32760 --heads 12 --head-dim 128
    python -m paper_2607_12358_gb300.kernel_bench linear --m 32760 --k 1536 --n 8960 --epi gelu
    python -m paper_2607_12358_gb300.kernel_bench drift --rows 118800 --cols 3072 [--apply]
    python -m paper_2607_12358_gb300.kernel_bench temni --rows 32760 --cols 1536
    python -m paper_2607_12358_gb300.kernel_bench layernorm --rows 32760 --cols 1536 --in-dtype fp32
    python -m paper_2607_12358_gb300.kernel_bench block --workload wan [--block-type wan]

Inputs are random bf16 tensors created on the device (block: the synthetic
full-size weights of one block of the named workload, a N(0,1) input and a
N(0,1) stand-in time embedding).  Prints one JSON line.
"""

from __future__ import annotations

import argparse
import json
import os
import sys

import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def _time(fn, warmup, iters):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(iters):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / iters


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("kernel", choices=["attention", "linear", "drift", "temni", "layernorm", "block"])
    ap.add_argument("--workload", default="wan", help="block: wan | cog | hv")
    ap.add_argument("--block-type", default=None, help="block: wan | cog | hv_dual | hv_single")
    ap.add_argument("--n", type=int, default=32760)
    ap.add_argument("--nk", type=int, default=0, help="keys (attention); default = --n")
    ap.add_argument("--heads", type=int, default=12)
    ap.add_argument("--head-dim", type=int, default=128)
    ap.add_argument("--m", type=int, default=32760)
    ap.add_argument("--k", type=int, default=1536)
    ap.add_argument("--epi", default="bias", choices=["bias", "gelu", "gated_res", "res"])
    ap.add_argument("--rows", type=int, default=118800)
    ap.add_argument("--cols", type=int, default=3072)
    ap.add_argument("--apply", action="store_true")
    ap.add_argument("--in-dtype", default="bf16", choices=["bf16", "fp32"], help="layernorm: input dtype")
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--iters", type=int, default=5)
    a = ap.parse_args()

    import __graft_entry__ as g

    g.build()
    from paper_2607_12358_gb300 import acid

    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(0)
    out = {"kernel": a.kernel}
    if a.kernel == "attention":
        nk = a.nk or a.n
        w = a.heads * a.head_dim
        qkv = torch.randn(max(a.n, nk), 3 * w, device=dev, generator=gen).to(torch.bfloat16)
        q, k, v = qkv[:a.n, :w], qkv[:nk, w:2 * w], qkv[:nk, 2 * w:]
        o = torch.empty(a.n, w, device=dev, dtype=torch.bfloat16)
        ws = torch.empty(acid.attention_workspace_size(a.head_dim), dtype=torch.uint8, device=dev)
        ms = _time(lambda: acid.acid_attention_forward(q, k, v, a.heads, out=o, workspace=ws), a.warmup, a.iters)
        flop = 4.0 * a.n * nk * a.head_dim * a.heads
        out.update(shape=[a.n, nk, a.heads, a.head_dim], ms=ms, tflops=flop / ms / 1e9)
    elif a.kernel == "linear":
        x = torch.randn(a.m, a.k, device=dev, generator=gen).to(torch.bfloat16)
        wt = (0.02 * torch.randn(a.n, a.k, device=dev, generator=gen)).to(torch.bfloat16)
        b = torch.randn(a.n, device=dev, generator=gen)
        gate = torch.randn(a.n, device=dev, generator=gen)
        y = torch.randn(a.m, a.n, device=dev, generator=gen).to(torch.bfloat16)
        res = y if a.epi in ("gated_res", "res") else None
        ms = _time(lambda: acid.acid_linear_forward(x, wt, b, epilogue=a.epi, gate=gate, residual=res, out=y),
                   a.warmup, a.iters)
        flop = 2.0 * a.m * a.n * a.k
        out.update(shape=[a.m, a.k, a.n], epi=a.epi, ms=ms, tflops=flop / ms / 1e9)
    elif a.kernel == "layernorm":
        # adaLN LayerNorm of the residual stream into the bf16 GEMM operand:
        # reads x once, writes y once (the shift / scale vectors stay in L2)
        dt = torch.float32 if a.in_dtype == "fp32" else torch.bfloat16
        x = torch.randn(a.rows, a.cols, device=dev, generator=gen).to(dt)
        shift = torch.randn(a.cols, device=dev, generator=gen)
        scale = torch.randn(a.cols, device=dev, generator=gen)
        y = torch.empty(a.rows, a.cols, device=dev, dtype=torch.bfloat16)
        ms = _time(lambda: acid.acid_layernorm_mod(x, shift, scale, out_dtype=torch.bfloat16, out=y),
                   a.warmup, a.iters)
        nbytes = float(a.rows) * a.cols * (x.element_size() + 2)
        out.update(shape=[a.rows, a.cols], in_dtype=a.in_dtype, ms=ms, gbs=nbytes / ms / 1e6)
    elif a.kernel == "temni":
        # TeaCache signal from two steps' fp32 patch embeddings: reads 8 B/elem
        hp = torch.randn(a.rows, a.cols, device=dev, generator=gen)
        hc = hp + 0.05 * torch.randn(a.rows, a.cols, device=dev, generator=gen)
        mp = 0.3 * torch.randn(2 * a.cols, device=dev, generator=gen)
        mc = mp + 0.01 * torch.randn(2 * a.cols, device=dev, generator=gen)
        ws = torch.empty(acid.drift_workspace_size(a.rows * a.cols), dtype=torch.uint8, device=dev)
        rel = torch.empty(1, dtype=torch.float64, device=dev)
        sums = torch.empty(2, dtype=torch.float64, device=dev)
        ms = _time(lambda: acid.acid_temni_drift(hp, hc, mp, mc, out_rel=rel, out_sums=sums, workspace=ws),
                   a.warmup, a.iters)
        nbytes = 8.0 * a.rows * a.cols
        out.update(shape=[a.rows, a.cols], ms=ms, gbs=nbytes / ms / 1e6, rel_l1=rel.item())
    elif a.kernel == "block":
        import acid_synth as S

        cfg = S.get_config(a.workload)
        bt = a.block_type or {"wan": "wan", "cog": "cog", "hv": "hv_dual"}[a.workload]
        w = S.block_weights(cfg, 0, seed=0, block_type=bt)
        rows = cfg.n_video + (0 if bt == "wan" else cfg.n_text)
        desc = acid.block_desc(cfg, bt)
        blk = acid.DeviceBlock.upload(w, bt, torch.bfloat16, dev)
        temb = torch.from_numpy(S.temb_vector(cfg, 0)).to(dev)
        x0 = torch.randn(rows, cfg.d, device=dev, generator=gen).to(torch.bfloat16)
        x = x0.clone()
        ctx = None
        if bt == "wan" and cfg.n_text:
            ctx = torch.randn(cfg.n_text, cfg.d, device=dev, generator=gen).to(torch.bfloat16)
        ws = torch.empty(acid.block_workspace_size(desc) + 1024, dtype=torch.uint8, device=dev)
        ms = _time(lambda: acid.acid_dit_block_forward(desc, x.copy_(x0), temb, blk, ctx=ctx, workspace=ws),
                   a.warmup, a.iters)
        out.update(workload=a.workload, block_type=bt, rows=rows, ms=ms)
    else:
        n = a.rows * a.cols
        p = torch.randn(n, device=dev, generator=gen).to(torch.bfloat16)
        c = (p.float() + 0.01 * torch.randn(n, device=dev, generator=gen)).to(torch.bfloat16)
        ws = torch.empty(acid.drift_workspace_size(n), dtype=torch.uint8, device=dev)
        rel = torch.empty(1, dtype=torch.float64, device=dev)
        sums = torch.empty(2, dtype=torch.float64, device=dev)
        if a.apply:
            r = torch.randn(n, device=dev, generator=gen).to(torch.bfloat16)
            o = torch.empty_like(p)
            ms = _time(lambda: acid.acid_drift_apply(p, c, r, out=o, out_rel=rel, out_sums=sums, workspace=ws),
                       a.warmup, a.iters)
            nbytes = 8.0 * n
        else:
            ms = _time(lambda: acid.acid_drift_signal(p, c, out_rel=rel, out_sums=sums, workspace=ws),
                       a.warmup, a.iters)
            nbytes = 4.0 * n
        out.update(shape=[a.rows, a.cols], apply=a.apply, ms=ms, gbs=nbytes / ms / 1e6)
    acid.check_device_error()
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
