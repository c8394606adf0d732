"""Threshold sweeps over whole generations (Sec. 3.2 and Sec. 3.3).

Sec. 3.2 motivates the dual threshold with an experiment: a low fixed
threshold, a high fixed threshold, and two-threshold runs that switch from
low to high at a chosen step, compared on speed (steps computed) and quality
(distance to the uncached output), next to the trace of the caching signal
and of its rate of change.  This module runs that experiment, plus Algorithm
1's adaptive switch over a grid of delta, on the GPU loop:

    python -m paper_2607_12358_gb300.sweep --workload wan --blocks 30 \
        --transitions 5,10,15,20,25 --deltas 0.002,0.005,0.01,0.02 --out sweep.json

Every run is one call of the graph-launched generation (or the host-driven
loop with ``--host-loop``).  Per run the output records the decisions, the
signal s_t, |s_t - s_prev| and tau of every step, the compute count, the
generation time and the relative L2 distance of the final latent to the
every-step-computed latent.  With random weights the distances say nothing
about video quality; the sweep exercises the mechanics and records the
signal traces.

The analysis helpers (first and second differences of a trace, the step from
which |s_t - s_{t-1}| stays within delta, and which runs beat the straight
line between the two fixed-threshold runs) are plain host arithmetic on the
logs and are usable without a GPU.
"""

from __future__ import annotations

import argparse
import json
import math
import time


# ---------------------------------------------------------------------------
# host-side analysis of logged traces
# ---------------------------------------------------------------------------

def differences(trace):
    """First and second differences of a signal trace (NaN where undefined:
    warmup steps carry NaN and propagate)."""
    d1 = [math.nan] + [b - a for a, b in zip(trace[:-1], trace[1:])]
    d2 = [math.nan] + [b - a for a, b in zip(d1[:-1], d1[1:])]
    return d1, d2


def stable_from(trace, delta):
    """First step k from which |s_t - s_{t-1}| <= delta holds at every later
    step where the difference is defined (Sec. 3.2 finds the best switch
    points where the signal's rate of change settles).  None if the last
    defined difference exceeds delta; len(trace) if none is defined."""
    d1, _ = differences(trace)
    defined = [t for t in range(len(trace)) if not math.isnan(d1[t])]
    if not defined:
        return len(trace)
    k = None
    for t in reversed(defined):
        if abs(d1[t]) > delta:
            break
        k = t
    return k


def beats_fixed_line(run, lo, hi):
    """True if (computed, err) of ``run`` lies strictly below the straight
    line through the fixed-low and fixed-high runs in the (steps computed,
    error) plane, i.e. at equal cost it is more accurate than mixing the two
    fixed thresholds.  The paper states the criterion only in words; this is
    the reading used here."""
    c_lo, e_lo = lo["computed"], lo["rel_l2"]
    c_hi, e_hi = hi["computed"], hi["rel_l2"]
    c, e = run["computed"], run["rel_l2"]
    if c_lo == c_hi:
        return c <= c_lo and e < min(e_lo, e_hi)
    line = e_hi + (e_lo - e_hi) * (c - c_hi) / (c_lo - c_hi)
    return e < line


def transition_schedule(n_steps, k, tau_low, tau_high):
    """tau_low before step k, tau_high from step k on."""
    return [tau_low] * k + [tau_high] * (n_steps - k)


# ---------------------------------------------------------------------------
# GPU runs
# ---------------------------------------------------------------------------

def _run(acid, torch, model, cfg, lat0, text, n_steps, graph, **kw):
    c, keep = acid.loop_cfg(cfg, n_steps=n_steps, **kw)
    lat = torch.from_numpy(lat0).to(model.device)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    logs = acid.acid_denoise_loop(model, c, lat, text, graph=graph)
    torch.cuda.synchronize()
    secs = time.perf_counter() - t0
    acid.check_device_error()
    del keep
    return lat, logs, secs


def _record(name, lat, ref, logs, secs, **extra):
    err = ((lat - ref).norm() / ref.norm()).item()
    rec = {
        "name": name,
        "computed": sum(int(l["computed"]) for l in logs),
        "steps": len(logs),
        "rel_l2": err,
        "seconds": secs,
        "decisions": [int(l["computed"]) for l in logs],
        "signal": [l["signal"] for l in logs],
        "dsignal": [l["dsignal"] for l in logs],
        "tau": [l["tau"] for l in logs],
    }
    rec.update(extra)
    return rec


def sweep(cfg, weights, latent, text=None, n_steps=None, tau_low=None, tau_high=None, transitions=(),
          deltas=(), method=None, graph=True, device="cuda", model=None):
    """Runs the sweep on one GPU and returns a JSON-ready dict.

    cfg, weights, latent, text: a workload config and its numpy inputs (the
    shapes of acid_synth's generators); ``model`` may pass an already
    uploaded DeviceModel.  transitions: switch steps k of the fixed low-to-high
    schedule; deltas: delta values for Algorithm 1's adaptive switch."""
    import numpy as np
    import torch

    from . import acid

    n_steps = cfg.steps if n_steps is None else n_steps
    tau_low = cfg.tau_low if tau_low is None else tau_low
    tau_high = cfg.tau_high if tau_high is None else tau_high
    method = cfg.method if method is None else method
    if model is None:
        model = acid.DeviceModel(cfg, weights, device)
    tt = None if text is None else torch.from_numpy(np.asarray(text)).to(model.device, model.wdtype)
    common = dict(method=method, graph=graph)

    ref, logs, secs = _run(acid, torch, model, cfg, latent, tt, n_steps, tau_low=-1.0, tau_high=-1.0, **common)
    full = _record("every step computed", ref, ref, logs, secs)
    d1, d2 = differences(full["signal"])
    full["d1"], full["d2"] = d1, d2

    runs = []
    lat, logs, secs = _run(acid, torch, model, cfg, latent, tt, n_steps, tau_low=tau_low, tau_high=tau_low, **common)
    lo = _record("fixed tau_low", lat, ref, logs, secs, tau_value=tau_low)
    lat, logs, secs = _run(acid, torch, model, cfg, latent, tt, n_steps, tau_low=tau_high, tau_high=tau_high,
                           **common)
    hi = _record("fixed tau_high", lat, ref, logs, secs, tau_value=tau_high)
    for k in transitions:
        sched = transition_schedule(n_steps, int(k), tau_low, tau_high)
        lat, logs, secs = _run(acid, torch, model, cfg, latent, tt, n_steps, tau_low=tau_low, tau_high=tau_high,
                               tau_schedule=sched, **common)
        runs.append(_record(f"switch at step {k}", lat, ref, logs, secs, kind="transition", k=int(k)))
    for dl in deltas:
        lat, logs, secs = _run(acid, torch, model, cfg, latent, tt, n_steps, tau_low=tau_low, tau_high=tau_high,
                               delta=float(dl), **common)
        runs.append(_record(f"adaptive delta={dl}", lat, ref, logs, secs, kind="adaptive", delta=float(dl),
                            stable_from=stable_from(full["signal"], float(dl))))
    for r in runs:
        r["beats_fixed_line"] = beats_fixed_line(r, lo, hi)
    del ref
    return {
        "workload": cfg.name, "method": method, "n_steps": n_steps, "tau_low": tau_low, "tau_high": tau_high,
        "launch": "graph" if graph else "host loop",
        "full": full, "fixed_low": lo, "fixed_high": hi, "runs": runs,
    }


def _ints(s):
    return [int(x) for x in s.split(",") if x]


def _floats(s):
    return [float(x) for x in s.split(",") if x]


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workload", default="wan", help="toy | wan | cog | hv (synthetic inputs of that shape)")
    ap.add_argument("--blocks", type=int, default=None, help="override the block count (HV: dual blocks)")
    ap.add_argument("--single", type=int, default=None, help="HV: override the single-stream block count")
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--method", default=None, help="teacache | easycache | dicache")
    ap.add_argument("--tau-low", type=float, default=None)
    ap.add_argument("--tau-high", type=float, default=None)
    ap.add_argument("--transitions", type=_ints, default=[])
    ap.add_argument("--deltas", type=_floats, default=[])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--host-loop", action="store_true", help="host-driven loop instead of the CUDA graph")
    ap.add_argument("--out", default=None, help="write the JSON here (default: stdout)")
    ap.add_argument("--jsonl", default=None,
                    help="also write one JSON line per run and step (run, step, t, signal, dsignal, tau, sigma, "
                         "computed)")
    a = ap.parse_args(argv)

    import acid_synth as S

    over = {}
    if a.blocks is not None:
        over["n_blocks"] = a.blocks
    if a.single is not None:
        over["n_single"] = a.single
    if a.steps is not None:
        over["steps"] = a.steps
    cfg = S.get_config(a.workload, **over)
    weights = S.model_weights(cfg, a.seed)
    text = S.text(cfg, a.seed) if cfg.n_text > 0 else None
    res = sweep(cfg, weights, S.latent(cfg, a.seed), text, tau_low=a.tau_low, tau_high=a.tau_high,
                transitions=a.transitions, deltas=a.deltas, method=a.method, graph=not a.host_loop)
    out = json.dumps(res)
    if a.jsonl:
        with open(a.jsonl, "w") as f:
            for r in [res["full"], res["fixed_low"], res["fixed_high"]] + res["runs"]:
                for i in range(r["steps"]):
                    f.write(json.dumps({"run": r["name"], "step": i, "signal": r["signal"][i],
                                        "dsignal": r["dsignal"][i], "tau": r["tau"][i],
                                        "computed": r["decisions"][i]}) + "\n")
    if a.out:
        with open(a.out, "w") as f:
            f.write(out + "\n")
    else:
        print(out)
    for r in [res["fixed_low"], res["fixed_high"]] + res["runs"]:
        print(f"{r['name']:>28}: computed {r['computed']:3d}/{r['steps']}  rel_l2 {r['rel_l2']:.3e}  "
              f"{r['seconds']:.2f} s" + ("  *" if r.get("beats_fixed_line") else ""), flush=True)


if __name__ == "__main__":
    main()
