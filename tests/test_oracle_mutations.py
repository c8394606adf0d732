"""The oracle's pins catch plausible mistakes.

Each mutant plants one mistake in a copy of the oracle: a dropped term, a
flipped sign, a swapped operand, axis or argument, an off-by-one, or a step of
Algorithm 1 done in the wrong order or under the wrong condition.  It then
runs the pin tests of that part against the copy, in a subprocess, and
expects them to fail.  A control run of the same selections against an
unmodified copy must pass, so that a failure is the planted mistake's doing.
The real oracle is never touched; every copy lives in a temporary directory.
"""

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE_SRC = os.path.join(ROOT, "oracle", "acid_oracle.py")

P = "tests/test_oracle_pins.py"
C = "tests/test_oracle_controller.py"
G = "tests/test_oracle_guidance.py"

# (name, [(text in the oracle, replacement), ...], pin files, -k selection)
MUTANTS = [
    ("rel_l1 normalised by the current value",
     [("    den = float(np.abs(p).sum())\n    if den == 0.0:\n        return 0.0 if num == 0.0 else math.inf\n"
       "    return num / den",
       "    den = float(np.abs(c).sum())\n    if den == 0.0:\n        return 0.0 if num == 0.0 else math.inf\n"
       "    return num / den")], [P], "rel_l1"),
    ("rel_l1 with the sign kept inside the sum",
     [("    num = float(np.abs(c - p).sum())\n    den",
       "    num = float(abs((c - p).sum()))\n    den")], [P], "rel_l1"),
    ("drift sums returned in swapped order",
     [("return float(np.abs(c - p).sum()), float(np.abs(p).sum())",
       "return float(np.abs(p).sum()), float(np.abs(c - p).sum())")], [P], "drift_sums"),
    ("cache apply subtracts the residual",
     [("+ np.asarray(cached_residual, dtype=F64)", "- np.asarray(cached_residual, dtype=F64)")],
     [C], "loop"),
    ("EasyCache rate inverted",
     [("        return 0.0 if dv == 0.0 else math.inf\n    return dv / dx",
       "        return 0.0 if dv == 0.0 else math.inf\n    return dx / max(dv, 1e-300)")], [C], "easycache"),
    ("EasyCache reuse offset reversed",
     [("(np.asarray(v_c, F64) - np.asarray(x_c, F64))", "(np.asarray(x_c, F64) - np.asarray(v_c, F64))")],
     [C], "easycache"),
    ("DiCache ratio against the older computed step",
     [("float(np.abs(np.asarray(p_t, F64) - np.asarray(p_c1, F64)).sum()) / den",
       "float(np.abs(np.asarray(p_t, F64) - np.asarray(p_c2, F64)).sum()) / den")], [C], "dicache"),
    ("DiCache extrapolation with the wrong sign",
     [("d1 + g * (d1 - np.asarray(d_c2, F64))", "d1 - g * (d1 - np.asarray(d_c2, F64))")], [C], "dicache"),
    ("a tie computes instead of skipping",
     [("skip = sigma_seen <= tau", "skip = sigma_seen < tau")], [C], "golden or schedule"),
    ("open interval for |s_t - s_prev| <= delta",
     [("tau = self.tau_high if ds <= self.delta else self.tau_low",
       "tau = self.tau_high if ds < self.delta else self.tau_low")], [C], "golden"),
    ("signal accumulated after the comparison",
     [("        s_t = float(s_t)\n        self.sigma = self.sigma + s_t\n", "        s_t = float(s_t)\n"),
      ("        sigma_seen = self.sigma\n        skip = sigma_seen <= tau\n",
       "        sigma_seen = self.sigma\n        skip = sigma_seen <= tau\n        self.sigma = self.sigma + s_t\n")],
     [C], "golden"),
    ("accumulator not reset on a computed step",
     [("        if not skip:\n            self.sigma = 0.0\n", "        if not skip:\n            pass\n")],
     [C], "golden"),
    ("s_prev updated on computed steps only",
     [("        self.s_prev = s_t\n        return skip", "        if not skip:\n            self.s_prev = s_t\n"
       "        return skip")], [C], "golden"),
    ("first non-warmup step uses the high threshold",
     [("            ds = math.nan\n            tau = self.tau_low", "            ds = math.nan\n"
       "            tau = self.tau_high")], [C], "golden"),
    ("Euler step with the wrong sign",
     [("(sigma_next - sigma_cur) * np.asarray(v, F64)", "(sigma_cur - sigma_next) * np.asarray(v, F64)")],
     [P], "euler"),
    ("noise levels off by one",
     [("s = 1.0 - np.arange(n_steps + 1, dtype=F64) / n_steps",
       "s = 1.0 - np.arange(n_steps + 1, dtype=F64) / (n_steps + 1)")], [P], "euler"),
    ("LayerNorm with the unbiased variance",
     [("var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)",
       "var = ((x - mu) ** 2).sum(axis=-1, keepdims=True) / (x.shape[-1] - 1)")], [P], "layernorm"),
    ("modulation without the 1 in (1 + scale)",
     [("np.asarray(xn, F64) * (1.0 + np.asarray(scale, F64))", "np.asarray(xn, F64) * np.asarray(scale, F64)")],
     [P], "layernorm or wan_block or temni"),
    ("GELU without the cubic term",
     [("(x + 0.044715 * x ** 3)", "(x)")], [P], "gelu"),
    ("attention scaled by 1/Dh",
     [("scale = 1.0 / math.sqrt(Dh)", "scale = 1.0 / Dh")], [P], "attention"),
    ("attention weights applied to the keys",
     [("out[s0:s0 + chunk, h, :] = p @ vh", "out[s0:s0 + chunk, h, :] = p @ kh")], [P], "attention"),
    ("RoPE rotation with the wrong sign",
     [("y[..., 0::2] = x0 * c - x1 * s", "y[..., 0::2] = x0 * c + x1 * s")], [P], "rope"),
    ("RoPE height and width positions swapped",
     [("for pos, da in ((f, dt), (h, dh), (w, dw)):", "for pos, da in ((f, dt), (w, dh), (h, dw)):")],
     [P], "rope"),
    ("RoPE frequency exponent over half the axis width",
     [("inv = theta ** (-np.arange(0, da, 2, dtype=F64) / da)",
       "inv = theta ** (-np.arange(0, da, 2, dtype=F64) / (da // 2))")], [P], "rope"),
    ("timestep sinusoid laid out [sin | cos]",
     [("np.concatenate([np.cos(a), np.sin(a)])", "np.concatenate([np.sin(a), np.cos(a)])")], [P], "sinusoid"),
    ("patchify with the channel index last",
     [("a = a.transpose(1, 3, 5, 0, 2, 4, 6)", "a = a.transpose(1, 3, 5, 2, 4, 6, 0)")], [P], "patchify"),
    ("self-attention residual without its gate",
     [('y = x[r] + g1 * linear(a, *w["o"])\n    if ctx is not None:',
       'y = x[r] + linear(a, *w["o"])\n    if ctx is not None:')], [P], "wan_block or zero_gates"),
    ("cross-attention query from the unnormalised residual",
     [('qc = _heads(linear(layer_norm(y, eps), *w["cq"]), heads)', 'qc = _heads(linear(y, *w["cq"]), heads)')],
     [P], "wan_block"),
    ("TeaCache caches the block-stack output instead of its residual",
     [("self.resid = h_out - si.h_in", "self.resid = h_out")], [C], "loop"),
    ("joint blocks give text rows the video modulation",
     [("np.where((idx < n_text)[:, None], mt[part][None, :], mv[part][None, :])",
       "np.where((idx < n_text)[:, None], mv[part][None, :], mt[part][None, :])")], [P], "cog_text or hv_dual"),
    ("single-stream block applies GELU before the MLP weights",
     [('m = gelu_tanh(linear(h[r], *w["mlp"]))', 'm = linear(gelu_tanh(h[r]), *w["mlp"])')], [P], "hv_single"),
    ("cross-attention keys from the video tokens",
     [('kvc = linear(c, *w["ckv"])', 'kvc = linear(y, *w["ckv"])')], [P], "wan_block"),
    ("feed-forward on the residual before attention",
     [("h = modulate(layer_norm(y, eps), sh2, sc2)", "h = modulate(layer_norm(x[r], eps), sh2, sc2)")],
     [P], "wan_block"),
    ("TEMNI from the feed-forward branch's modulation",
     [("return modulate(layer_norm(h_in, cfg.ln_eps), m[:d], m[d:2 * d])",
       "return modulate(layer_norm(h_in, cfg.ln_eps), m[3 * d:4 * d], m[4 * d:5 * d])")], [P, C],
     "temni"),
    ("signal polynomial in descending powers",
     [("return float(sum(c * s ** j for j, c in enumerate(coeffs)))",
       "return float(sum(c * s ** (len(coeffs) - 1 - j) for j, c in enumerate(coeffs)))")], [C], "polynomial"),
    ("fixed threshold schedule ignored",
     [("if tau_fixed is not None and not math.isnan(tau_fixed):", "if False:")], [C], "schedule"),
    ("controller replay with one warmup step too many",
     [("        if i < warmup:\n            out.append(True)", "        if i <= warmup:\n            out.append(True)")],
     [C], "equal_thresholds or negative_delta or zero_signal"),
    ("loop's timestep embedding at sigma instead of 1000 sigma",
     [("        si = step_inputs(cfg, w, x, 1000.0 * sig[i])\n        f = _step_override(forced, i)",
       "        si = step_inputs(cfg, w, x, sig[i])\n        f = _step_override(forced, i)")], [C], "loop"),
    ("force_last ignored",
     [("if force_last and i == n_steps - 1 and f is None:", "if False:")], [C], "force_last"),
    ("time MLP without its SiLU",
     [('    return linear(silu(h), *w["time2"])', '    return linear(h, *w["time2"])')], [P], "silu_closed"),
    ("block modulation without its SiLU",
     [("    return linear(silu(temb), *wb)", "    return linear(temb, *wb)")], [P], "silu_closed"),
    ("final layer with shift and scale swapped",
     [("final_mod[:d], final_mod[d:])", "final_mod[d:], final_mod[:d])")], [P], "final_layer_on_constant"),
    ("patch embedding without its bias",
     [('cfg.pw), *w["patch"])', 'cfg.pw), w["patch"][0])')], [P], "patch_embedding_bias"),
    ("noise-level shift inverted",
     [("        s = shift * s / (1.0 + (shift - 1.0) * s)", "        s = s / (shift - (shift - 1.0) * s)")],
     [P], "sigma_shift"),
    ("dual-stream text QKV from the video weights",
     [('    qkv_t = linear(ut, *w["txt.qkv"])', '    qkv_t = linear(ut, *w["vid.qkv"])')], [P], "interchangeable"),
    ("dual-stream text residual gated by the video gate",
     [('    yt = xt[rt] + mt[2] * linear(at, *w["txt.o"])', '    yt = xt[rt] + mv[2] * linear(at, *w["txt.o"])')],
     [P], "interchangeable"),
    ("dual-stream video FFN input on the text modulation",
     [("    hv = modulate(layer_norm(yv, eps), mv[3], mv[4])", "    hv = modulate(layer_norm(yv, eps), mt[3], mt[4])")],
     [P], "interchangeable"),
    ("TeaCache signal against the last computed step's TEMNI",
     [("            self.temni_prev = temni\n            if compute:\n",
       "            if compute:\n                self.temni_prev = temni\n")], [C], "consecutive_steps_through"),
    ("EasyCache rate against the last computed step",
     [("self.k_rate = easycache_rate(x, self.x_prev, v, self.v_prev)",
       "self.k_rate = easycache_rate(x, self.x_c, v, self.v_c)")], [C], "skip_then_compute"),
    ("EasyCache previous input and output kept from computed steps only",
     [("                v = easycache_reuse(x, self.x_c, self.v_c)\n            self.x_prev, self.v_prev = x, v",
       "                v = easycache_reuse(x, self.x_c, self.v_c)\n            if compute:\n"
       "                self.x_prev, self.v_prev = x, v")], [C], "skip_then_compute"),
    ("EasyCache rate 0 for an unchanged input",
     [("        return 0.0 if dv == 0.0 else math.inf\n    return dv / dx", "        return 0.0\n    return dv / dx")],
     [C], "unchanged_input"),
    ("force_last overrides an explicit skip",
     [("        if force_last and i == n_steps - 1 and f is None:", "        if force_last and i == n_steps - 1:")],
     [C], "explicit_decision"),
    ("DiCache keeps only the latest computed step",
     [("                    self.p_c2, self.d_c2 = self.p_c1, self.d_c1", "                    self.p_c2, self.d_c2 = probe, d_new")],
     [C], "last_two_computed"),
    ("joint stack with the video rows first",
     [("    return np.concatenate([np.asarray(ctx, F64), np.asarray(h_in, F64)], axis=0)",
       "    return np.concatenate([np.asarray(h_in, F64), np.asarray(ctx, F64)], axis=0)")],
     [P], "identity_blocks_returns"),
    ("guided branches share one branch state",
     [("    bu = SamplerBranch(cfg, w, text_uncond, tau_low, tau_high, delta, warmup, method, probe_blocks, signal_poly)",
       "    bu = bc")], [G], "branch_state"),
    ("text projection without its bias",
     [('        return linear(text, *w["text"])', '        return linear(text, w["text"][0])')], [P], "text_context_closed"),
    ("dual-stream modulations handed over in swapped order",
     [('            mods.append((block_modulation(temb, wb["vid.mod"]), block_modulation(temb, wb["txt.mod"])))',
       '            mods.append((block_modulation(temb, wb["txt.mod"]), block_modulation(temb, wb["vid.mod"])))')],
     [P], "reaches_its_own_stream"),
    ("guidance extrapolates from the conditional branch",
     [("return v_uncond + scale * (v_cond - v_uncond)", "return v_cond + scale * (v_uncond - v_cond)")],
     [G], "guidance or unit_and_zero"),
]


def _tree(base, name, source):
    """A directory with tests/ and acid_synth/ linked from the repository and
    oracle/ holding `source` as its module."""
    d = os.path.join(base, name)
    os.makedirs(os.path.join(d, "oracle"))
    shutil.copy(os.path.join(ROOT, "oracle", "__init__.py"), os.path.join(d, "oracle", "__init__.py"))
    with open(os.path.join(d, "oracle", "acid_oracle.py"), "w") as f:
        f.write(source)
    for sub in ("tests", "acid_synth"):
        os.symlink(os.path.join(ROOT, sub), os.path.join(d, sub))
    return d


def _pytest(d, files, kexpr):
    env = {k: v for k, v in os.environ.items() if k != "PYTHONPATH"}
    env["PYTHONDONTWRITEBYTECODE"] = "1"
    cmd = [sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", "-m", "not gpu",
           "--rootdir", d, "-c", os.devnull, "-k", kexpr, *files]
    r = subprocess.run(cmd, cwd=d, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode, r.stdout[-2000:]


@pytest.fixture(scope="module")
def outcomes(tmp_path_factory):
    base = str(tmp_path_factory.mktemp("oracle_mutants"))
    with open(ORACLE_SRC) as f:
        src = f.read()
    jobs = {}
    for i, (name, edits, files, kexpr) in enumerate(MUTANTS):
        mutated = src
        for old, new in edits:
            assert src.count(old) == 1, f"{name}: the text to mutate must occur exactly once"
            mutated = mutated.replace(old, new)
        jobs[("mutant", name)] = (_tree(base, f"m{i:02d}", mutated), files, kexpr)
    for j, sel in enumerate(sorted({(tuple(f), k) for _, _, f, k in MUTANTS})):
        jobs[("control", sel)] = (_tree(base, f"c{j:02d}", src), list(sel[0]), sel[1])
    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        futs = {key: ex.submit(_pytest, *job) for key, job in jobs.items()}
        return {key: fut.result() for key, fut in futs.items()}


@pytest.mark.parametrize("sel", sorted({(tuple(f), k) for _, _, f, k in MUTANTS}), ids=lambda s: s[1])
def test_selection_passes_on_the_oracle(outcomes, sel):
    rc, out = outcomes[("control", sel)]
    assert rc == 0, out


@pytest.mark.parametrize("name", [m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(outcomes, name):
    rc, out = outcomes[("mutant", name)]
    assert rc == 1, f"no pin caught: {name}\n{out}"
