#!/usr/bin/env python3
"""Benchmark of the ACID hot path on the Wan-2.1-1.3B-shaped 480p workload.

One step = one sampler step of the whole path: timestep embedding and
modulation, patch embedding, block-0 modulated input and its relative-L1
drift, the dual-threshold decision (Algorithm 1), the 30-block DiT stack
(computed), the TeaCache residual update, the final layer and the Euler
update.  The timed schedule computes every step (thresholds -1), so the
number is the cost of a computed step with the drift machinery included; a
second pass with the workload's thresholds reports the effective rate under
caching.  Weights are random N(0, 0.02), latents and text N(0, 1).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  Under torchrun every rank runs an independent
replica (the path has no data-parallel exchange) and the value is the total
steps/s over all ranks.
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "DiT steps/s and attention TFLOP/s (% bf16 peak), Wan-1.3B-shaped 480p"
UNIT = "steps/s"
WORKLOAD = ("Wan-2.1-1.3B-shaped 480p step: 30 blocks, d=1536, 12 heads x 128, FFN 8960, "
            "32760 video tokens (21x30x52, 3D RoPE), cross-attention to 512 text tokens (4096 -> 1536)")
# Query rows of the oracle sample, the same for the GPU arm's cpu_baseline and
# for the reference arm (about 7 s of fp64 numpy work per sample on 16 cores).
SAMPLE_ROWS = 2048
MICRO_T = (32760, 67320, 118800)  # drift micro-benchmark rows (x 3072 bf16)
MICRO_SIGMA = 1e-2

# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum, ncu captures of
# a self-attention call (main launch, split tail launch and merge) and a
# cross-attention call (one persistent launch) at this shape, each the mean of
# two calls) per attention call of the step's 1:1 self/cross mix: 436.9 MB and
# 159.2 MB.  Valid only for the kernel source it was measured on; any other
# source reports null.
ATTN_TRAFFIC = {"source_sha256_16": "c918258b40c85349", "bytes_per_launch": (436.88e6 + 159.20e6) / 2}


def _attn_traffic():
    import hashlib

    src = os.path.join(ROOT, "paper_2607_12358_gb300", "csrc", "attention.cu")
    with open(src, "rb") as f:
        h = hashlib.sha256(f.read()).hexdigest()[:16]
    return ATTN_TRAFFIC["bytes_per_launch"] if h == ATTN_TRAFFIC["source_sha256_16"] else None


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(value: float, world: int) -> float:
    """The largest `value` over all ranks: the job takes as long as its slowest
    rank (the process group must be initialised when world > 1)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(value)], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.item()


def job_rate(steps: int, seconds: float, world: int) -> float:
    """Whole-job steps/s: each of the `world` replicas runs `steps` steps in at
    most `seconds` (the max over ranks)."""
    return world * steps / seconds


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines: list[str] = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self._t = threading.Thread(target=self._read, daemon=True)
            self._t.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self) -> dict:
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU oracle sample (baseline and reference arm)
# ---------------------------------------------------------------------------

def _step_flops(cfg) -> float:
    N, L, d, F = cfg.n_video, cfg.n_text, cfg.d, cfg.ffn
    blk = (2 * N * d * 3 * d + 4 * N * N * d + 2 * N * d * d       # self-attention branch
           + 2 * N * d * d + 2 * L * d * 2 * d + 4 * N * L * d + 2 * N * d * d  # cross-attention
           + 4 * N * d * F)                                          # FFN
    return cfg.n_blocks * blk


def _sample_flops(cfg, R) -> float:
    N, L, d, F = cfg.n_video, cfg.n_text, cfg.d, cfg.ffn
    return (2 * N * d * 2 * d + 2 * R * d * d + 4 * R * N * d + 2 * R * d * d
            + 2 * R * d * d + 2 * L * d * 2 * d + 4 * R * L * d + 2 * R * d * d + 4 * R * d * F)


class OracleSample:
    """One Wan-shaped block in the fp64 oracle: keys and values for all 32760
    tokens and every per-token operation for R query rows.  Scaled by
    algorithmic FLOPs to one 30-block step."""

    def __init__(self, rows: int, seed: int = 0):
        import numpy as np

        import acid_synth as S
        import oracle as O

        self.O = O
        self.cfg = S.get_config("wan")
        self.w = S.block_weights(self.cfg, 0, seed)
        self.x = S.hidden(self.cfg, self.cfg.n_video, seed).astype(np.float64)
        self.mod = O.block_modulation(S.temb_vector(self.cfg, seed), self.w["mod"])
        self.ctx = S.round_to_bf16(S.normal(seed, (self.cfg.n_text, self.cfg.d), 1.0, "bench", "ctx"))
        self.rows = np.arange(rows)
        self.R = rows

    def run(self) -> float:
        t0 = time.perf_counter()
        self.O.wan_block(self.x, self.mod, self.w, self.cfg.grid, self.cfg.heads, ctx=self.ctx, rows=self.rows)
        return time.perf_counter() - t0

    def steps_per_s(self, seconds: float) -> float:
        return _sample_flops(self.cfg, self.R) / (seconds * _step_flops(self.cfg))

    def describe(self) -> str:
        return (f"fp64 numpy oracle: one Wan-shaped block, K/V for all {self.cfg.n_video} tokens and every "
                f"per-token op for {self.R} query rows ({_sample_flops(self.cfg, self.R) / 1e12:.2f} TFLOP), "
                f"scaled by algorithmic FLOPs to a 30-block step ({_step_flops(self.cfg) / 1e12:.1f} TFLOP)")


def _cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def _config(seq_len: int) -> dict:
    """The workload description both arms print (identical keys and values)."""
    return {"workload": WORKLOAD, "global_batch": 1, "seq_len": seq_len, "parallelism": "replicas",
            "schedule": "every step computed (tau_low = tau_high = -1); drift and decision still run",
            "l2": "no flush: per-step working set (3.4 GB of bf16 weights read once per step, >0.5 GB "
                  "activations) exceeds the 129 MB L2"}


def baseline_record(sample: "OracleSample", seconds: list[float]) -> dict:
    """cpu_baseline object of a timed oracle sample: the step rate is the
    sample's FLOP-scaled rate (extrapolated, not timed as a whole step)."""
    mean = sum(seconds) / len(seconds)
    return {"value": sample.steps_per_s(mean), "unit": UNIT, "cores": _cores(), "kind": "oracle",
            "sample": sample.describe(), "extrapolated_from_rows": sample.R,
            "sample_seconds": mean, "samples_timed": len(seconds),
            "scaled_by": "algorithmic FLOPs of one 30-block step / FLOPs of the sample"}


def run_reference(args) -> None:
    ws, rank, _ = _dist()
    if rank != 0:
        return
    s = OracleSample(SAMPLE_ROWS)
    for _ in range(args.warmup):
        s.run()
    times = [s.run() for _ in range(args.steps)]
    base = baseline_record(s, times)
    value = base["value"]
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 / value,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (random N(0,0.02) weights, N(0,1) latent and text)",
            "config": _config(32760),
            "cpu_baseline": base,
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "note": "each timed step is one oracle sample of %d query rows (%.1f s); ms_per_step is the "
                    "FLOP-scaled time of a whole 30-block step, not a timed step" % (s.R, base["sample_seconds"])}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

def _launch_ms(fn, iters: int) -> float:
    """Mean device time of one call of fn over `iters` back-to-back calls
    (CUDA events on the current stream around the whole run)."""
    import torch

    st = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(iters):
        fn()
    e1.record(st)
    e1.synchronize()
    return e0.elapsed_time(e1) / iters


def micro_bench(acid, dev, peaks: dict, iters: int = 20) -> dict:
    """Drift reduction, stand-alone cache apply and the fused drift + apply on
    [T, 3072] bf16 (prev ~ N(0,1), cur = prev + 0.01 z).  Every input set is
    at least 403 MB, three times the 129 MB L2, so launches run back to back
    without a flush (a flush by writing leaves dirty lines whose write-back
    would land inside the next timed launch).  Algorithmic bytes per element:
    drift 4 (reads prev, cur), apply 6 (reads x, residual, writes out), fused 8
    (reads prev, cur, residual, writes out)."""
    import torch

    gen = torch.Generator(device=dev).manual_seed(7)
    hbm = peaks["hbm_gbs"]
    out = {"d": 3072, "sigma": MICRO_SIGMA, "l2": "inputs >= 403 MB (3x L2), back-to-back launches, no flush",
           "rows": {}}
    worst = {"drift": 1.0, "apply": 1.0, "fused": 1.0}
    for T in MICRO_T:
        n = T * 3072
        p = torch.randn(n, device=dev, generator=gen).to(torch.bfloat16)
        c = (p.float() + MICRO_SIGMA * torch.randn(n, device=dev, generator=gen)).to(torch.bfloat16)
        r = torch.randn(n, device=dev, generator=gen).to(torch.bfloat16)
        o = torch.empty_like(p)
        ws = torch.empty(acid.drift_workspace_size(n), dtype=torch.uint8, device=dev)
        rel = torch.empty(1, dtype=torch.float64, device=dev)
        sums = torch.empty(2, dtype=torch.float64, device=dev)
        runs = {
            "drift": (lambda: acid.acid_drift_signal(p, c, out_rel=rel, out_sums=sums, workspace=ws), 4.0,
                      "drift_partials_kernel + drift_final_kernel"),
            "apply": (lambda: acid.acid_cache_apply(c, r, out=o), 6.0, "add_vec_kernel"),
            "fused": (lambda: acid.acid_drift_apply(p, c, r, out=o, out_rel=rel, out_sums=sums, workspace=ws), 8.0,
                      "drift_partials_kernel<apply> + drift_final_kernel"),
        }
        row = {}
        for name, (fn, bpe, kern) in runs.items():
            fn()
            fn()
            ms = _launch_ms(fn, iters)
            gbs = bpe * n / ms / 1e6
            row[name] = {"ms": ms, "gbs": gbs, "frac_of_hbm": gbs / hbm, "bytes_per_elem": bpe, "kernel": kern}
            worst[name] = min(worst[name], gbs / hbm)
        torch.cuda.synchronize()
        row["rel_l1"] = rel.item()
        out["rows"][str(T)] = row
        del p, c, r, o, ws
    out["min_frac_of_hbm"] = worst
    out["hbm_peak"] = hbm
    # the TeaCache signal from two steps' fp32 patch embeddings
    # (acid_temni_drift: reads 8 B/elem, the call includes the final
    # reduction), at the Wan step's shape and at a 720p-class row count
    out["temni"] = {}
    for rows, d in ((32760, 1536), (118800, 1536)):
        hp = torch.randn(rows, d, device=dev, generator=gen)
        hc = hp + 0.05 * torch.randn(rows, d, device=dev, generator=gen)
        mp = 0.3 * torch.randn(2 * d, device=dev, generator=gen)
        mc = mp + 0.01 * torch.randn(2 * d, device=dev, generator=gen)
        ws = torch.empty(acid.drift_workspace_size(rows * d), dtype=torch.uint8, device=dev)
        rel = torch.empty(1, dtype=torch.float64, device=dev)
        sums = torch.empty(2, dtype=torch.float64, device=dev)
        fn = lambda: acid.acid_temni_drift(hp, hc, mp, mc, out_rel=rel, out_sums=sums, workspace=ws)
        fn()
        fn()
        ms = _launch_ms(fn, iters)
        gbs = 8.0 * rows * d / ms / 1e6
        out["temni"][f"{rows}x{d}"] = {"ms": ms, "gbs": gbs, "frac_of_hbm": gbs / hbm, "bytes_per_elem": 8.0,
                                       "kernel": "temni_drift_kernel + drift_final_kernel"}
        del hp, hc, ws
    torch.cuda.empty_cache()
    return out


def block_bench(acid, dev, peaks: dict, iters: int = 3) -> dict:
    """One block of each other workload at full length (random N(0, 0.02)
    weights of that block, N(0, 1) input): block ms, and the attention and
    GEMM rates inside it from the library's per-launch CUDA events."""
    import torch

    import acid_synth as S

    res = {}
    for wl, bt in (("cog", "cog"), ("hv", "hv_dual"), ("hv", "hv_single")):
        cfg = S.get_config(wl)
        w = S.block_weights(cfg, 0, seed=0, block_type=bt)
        blk = acid.DeviceBlock.upload(w, bt, torch.bfloat16, dev)
        del w
        rows = cfg.n_video + cfg.n_text
        desc = acid.block_desc(cfg, bt)
        gen = torch.Generator(device=dev).manual_seed(11)
        temb = torch.from_numpy(S.temb_vector(cfg, 0)).to(dev)
        x0 = torch.randn(rows, cfg.d, device=dev, generator=gen).to(torch.bfloat16)
        x = x0.clone()
        ws = torch.empty(acid.block_workspace_size(desc) + 1024, dtype=torch.uint8, device=dev)

        def run():
            acid.acid_dit_block_forward(desc, x, temb, blk, workspace=ws)

        for _ in range(2):
            x.copy_(x0)
            run()
        torch.cuda.synchronize()
        ms_total = 0.0
        acid.profile_enable(True)
        for _ in range(iters):
            x.copy_(x0)
            ms_total += _launch_ms(run, 1)
        a_n, a_ms, a_flop = acid.profile_read(acid.PROF_ATTENTION)
        l_n, l_ms, l_flop = acid.profile_read(acid.PROF_LINEAR)
        acid.profile_enable(False)
        acid.check_device_error()
        att = a_flop / (a_ms / 1000.0) / 1e12 if a_ms > 0 else None
        lin = l_flop / (l_ms / 1000.0) / 1e12 if l_ms > 0 else None
        res[f"{wl}/{bt}"] = {
            "rows": rows, "d": cfg.d, "heads": cfg.heads, "head_dim": cfg.head_dim, "block_ms": ms_total / iters,
            "attention_tflops": att, "attention_frac_of_burst_peak": att / peaks["bf16_tflops"] if att else None,
            "attention_ms": a_ms / iters, "linear_tflops": lin, "linear_ms": l_ms / iters,
            "step_ms_estimate": ms_total / iters * (cfg.n_blocks if bt != "hv_single" else cfg.n_single),
        }
        del blk, x, x0, ws
        torch.cuda.empty_cache()
    res["note"] = ("one block timed alone, CUDA events; step_ms_estimate = block_ms x blocks of that kind; "
                   "working sets exceed L2 (no flush)")
    return res


def toy_bench(acid, dev, steps: int = 10) -> dict:
    """The fp32 toy DiT (2 blocks, d 256, 256 tokens): every step of a 10-step
    generation computed, device time per step."""
    import torch

    import acid_synth as S

    cfg = S.get_config("toy")
    model = acid.DeviceModel(cfg, S.model_weights(cfg, 0), dev)
    lat0 = torch.from_numpy(S.latent(cfg, 0)).to(dev)
    c, keep = acid.loop_cfg(cfg, n_steps=steps, tau_low=-1.0, tau_high=-1.0)
    loop = acid.Loop(model, c, None, dev)
    lat = lat0.clone()
    loop.step(lat, log=False)
    ms = _launch_ms(lambda: [loop.step(lat, log=False) for _ in range(steps - 1)], 1) / (steps - 1)
    return {"step_ms": ms, "steps_per_s": 1000.0 / ms, "dtype": "f32", "tokens": cfg.n_video, "blocks": cfg.n_blocks}


def run_ours(args) -> None:
    import numpy as np
    import torch

    import acid_synth as S
    import __graft_entry__ as g

    world, rank, local = _dist()
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("gloo")
    g.build()
    from paper_2607_12358_gb300 import acid

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    cfg = S.get_config("wan")
    weights = S.model_weights(cfg, seed=rank)
    model = acid.DeviceModel(cfg, weights, dev)
    del weights
    text = torch.from_numpy(S.text(cfg, rank)).to(dev, torch.bfloat16)
    lat0 = S.latent(cfg, rank)
    K, W = args.steps, args.warmup
    n_total = W + K + 1

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()

    # ---- device-resident pass: every step computed
    c, keep = acid.loop_cfg(cfg, n_steps=n_total, tau_low=-1.0, tau_high=-1.0)
    loop = acid.Loop(model, c, text, dev)
    lat = torch.from_numpy(lat0).to(dev)
    for _ in range(W):
        loop.step(lat, log=False)
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    acid.profile_enable(True)
    n_launch0 = acid.launch_count()
    with ClockSampler(local) as clk:
        e0.record()
        for _ in range(K):
            loop.step(lat, log=False)
        e1.record()
        barrier()
    ms = e0.elapsed_time(e1)
    launches = acid.launch_count() - n_launch0
    a_n, a_ms, a_flop = acid.profile_read(acid.PROF_ATTENTION)
    l_n, l_ms, l_flop = acid.profile_read(acid.PROF_LINEAR)
    d_n, d_ms, d_bytes = acid.profile_read(acid.PROF_DRIFT)
    acid.profile_enable(False)
    acid.check_device_error()
    assert torch.isfinite(lat).all().item()
    t_max = max_over_ranks(ms, world)
    value = job_rate(K, t_max / 1000.0, world)

    # ---- end to end: latent from pinned host memory each step, result read back
    c2, keep2 = acid.loop_cfg(cfg, n_steps=W + K + 1, tau_low=-1.0, tau_high=-1.0)
    loop2 = acid.Loop(model, c2, text, dev)
    host_in = torch.from_numpy(lat0).pin_memory()
    host_out = torch.empty_like(host_in).pin_memory()
    dlat = torch.empty(host_in.shape, dtype=torch.float32, device=dev)
    for _ in range(W):
        dlat.copy_(host_in, non_blocking=True)
        loop2.step(dlat, log=False)
        host_out.copy_(dlat, non_blocking=True)
    barrier()
    t0 = time.perf_counter()
    for _ in range(K):
        dlat.copy_(host_in, non_blocking=True)
        loop2.step(dlat, log=False)
        host_out.copy_(dlat, non_blocking=True)
    barrier()
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)
    lat_bytes = host_in.numel() * 4

    # ---- the workload's own thresholds (effective rate under caching)
    c3, keep3 = acid.loop_cfg(cfg, n_steps=K + 1)
    loop3 = acid.Loop(model, c3, text, dev)
    lat3 = torch.from_numpy(lat0).to(dev)
    barrier()
    e0.record()
    logs = [loop3.step(lat3) for _ in range(K)]
    e1.record()
    barrier()
    acid_ms = e0.elapsed_time(e1)
    computed = sum(int(x.computed) for x in logs)

    # ---- a step that reuses the cache: time embedding, patch embedding, the
    # TEMNI drift and the host decision, the cached residual, the final layer
    # and the Euler update (the method's whole per-step cost when it skips)
    c5, keep5 = acid.loop_cfg(cfg, n_steps=W + K + 2, forced=[True] + [False] * (W + K + 1))
    loop5 = acid.Loop(model, c5, text, dev)
    lat5 = torch.from_numpy(lat0).to(dev)
    for _ in range(W + 1):
        loop5.step(lat5, log=False)
    barrier()
    e0.record()
    for _ in range(K):
        loop5.step(lat5, log=False)
    e1.record()
    barrier()
    skip_ms = max_over_ranks(e0.elapsed_time(e1) / K, world)

    # ---- the same every-step-computed generation as one CUDA graph (signal and
    # decision on the device); the wall time includes building and
    # instantiating the graph
    c4, keep4 = acid.loop_cfg(cfg, n_steps=K, tau_low=-1.0, tau_high=-1.0)
    lat4 = torch.from_numpy(lat0).to(dev)
    barrier()
    t0 = time.perf_counter()
    acid.acid_denoise_loop(model, c4, lat4, text, log=False, graph=True)
    barrier()
    graph_s = max_over_ranks(time.perf_counter() - t0, world)
    acid.check_device_error()

    if rank != 0:
        return
    peaks, src = _peaks()
    peak = peaks["bf16_tflops_sustained"]
    att_tflops = a_flop / (a_ms / 1000.0) / 1e12 if a_ms > 0 else 0.0
    lin_tflops = l_flop / (l_ms / 1000.0) / 1e12 if l_ms > 0 else 0.0
    d_gbs = d_bytes / (d_ms / 1000.0) / 1e9 if d_ms > 0 else None
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": t_max / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic (random N(0,0.02) weights, N(0,1) latent and text)",
        "config": _config(cfg.n_video),
        "roofline": {"bound": "tensor", "kernel": "attn_tc_kernel<128> (self) + attn_persist_kernel<128> (cross attention)",
                     "achieved": att_tflops, "peak": peak, "unit": "TFLOP/s", "frac": att_tflops / peak,
                     "peak_source": f"bf16_tflops_sustained, {src}", "traffic": _attn_traffic(),
                     "frac_of_burst_peak": att_tflops / peaks["bf16_tflops"],
                     "launches": a_n, "avg_launch_ms": a_ms / max(a_n, 1)},
        "attention_tflops": att_tflops,
        "attention_pct_bf16_peak": 100.0 * att_tflops / peaks["bf16_tflops"],
        "linear": {"tflops": lin_tflops, "launches": l_n, "ms": l_ms},
        "drift": {"kernel": "temni_drift_kernel (TEMNI of this and the previous step formed from both steps' fp32 H_in in one read-only pass, 8 B/elem; its last CTA reduces the partials)",
                  "gbs": d_gbs, "frac_of_hbm": d_gbs / peaks["hbm_gbs"] if d_gbs else None,
                  "hbm_peak_source": f"hbm_gbs, {src}", "launches": d_n, "ms": d_ms},
        "block_ms": t_max / K / cfg.n_blocks,
        "acid_mode": {"steps_per_s": K / (acid_ms / 1000.0), "computed_steps": computed, "of": K,
                      "tau_low": cfg.tau_low, "tau_high": cfg.tau_high, "delta": cfg.delta,
                      "note": "random weights: the skip rate says nothing about a trained model"},
        "skip_step": {"ms": skip_ms, "frac_of_computed_step": skip_ms / (t_max / K),
                      "note": "a step whose decision is to reuse: time and patch embedding, TEMNI drift, host "
                              "decision, cached residual, final layer, Euler update"},
        "graph_mode": {"steps_per_s": job_rate(K, graph_s, world),
                       "note": "the same K steps, every step computed, as one CUDA graph (WHILE over steps, "
                               "IF/ELSE per decision); wall time including graph build and instantiation"},
        "e2e": {"value": job_rate(K, e2e_s, world), "unit": UNIT, "h2d_bytes_per_step": lat_bytes,
                "d2h_bytes_per_step": lat_bytes},
        "gpu_launches": launches,
        "clocks": clk.summary(),
    }
    if not args.no_extras:
        line["micro"] = micro_bench(acid, dev, peaks)
        line["blocks"] = block_bench(acid, dev, peaks)
        line["toy"] = toy_bench(acid, dev)
    if not args.no_cpu_baseline and world == 1:
        s = OracleSample(SAMPLE_ROWS)
        line["cpu_baseline"] = baseline_record(s, [s.run()])
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the per-workload blocks, the drift micro-benchmark and the toy step")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)  # at least three untimed warm-up steps
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
