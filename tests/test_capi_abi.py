"""CPU checks of the C ABI: the library loads, exports every function
include/acid.h declares, the ctypes mirror matches the C struct layouts, and
argument validation rejects bad calls before touching a GPU."""

import ctypes
import os
import re
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "acid.h")


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g

    g.build()
    from paper_2607_12358_gb300 import _capi

    return _capi.load()


def _declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(acid_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared_functions()
    for required in ("acid_dit_block_forward", "acid_drift_signal", "acid_cache_apply", "acid_denoise_loop"):
        assert required in names


def test_every_declared_function_is_exported(lib):
    so = os.path.join(ROOT, "paper_2607_12358_gb300", "libacid_gb300.so")
    out = subprocess.run(["nm", "-D", "--defined-only", so], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\sT\s(acid_[a-z0-9_]+)$", out, flags=re.M))
    missing = [n for n in _declared_functions() if n not in exported]
    assert not missing, missing
    for n in _declared_functions():
        assert hasattr(lib, n)


def test_debug_build_exports_the_same_boundary():
    """The debug build (kernel memory-index checks compiled in) builds from
    the same sources without a GPU and exports every declared function."""
    from paper_2607_12358_gb300 import build as b

    so = b.build(debug=True)
    out = subprocess.run(["nm", "-D", "--defined-only", so], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\sT\s(acid_[a-z0-9_]+)$", out, flags=re.M))
    missing = [n for n in _declared_functions() if n not in exported]
    assert not missing, missing


def test_version_and_clean_error(lib):
    assert b"sm_103a" in lib.acid_version()
    assert lib.acid_last_error() == b""


_PROBE = r"""
#include <stdio.h>
#include <stddef.h>
#include "acid.h"
#define P(T) printf(#T " %zu\n", sizeof(T));
#define O(T, f) printf(#T "." #f " %zu\n", offsetof(T, f));
int main(void) {
  P(acid_block_desc) O(acid_block_desc, n_text) O(acid_block_desc, ln_eps)
  P(acid_linear) P(acid_block_weights) O(acid_block_weights, t_ff2)
  P(acid_cond) O(acid_cond, ctx_kv) P(acid_model) O(acid_model, blocks) O(acid_model, d_text) O(acid_model, final_out)
  P(acid_loop_cfg) O(acid_loop_cfg, tau_low) O(acid_loop_cfg, forced) O(acid_loop_cfg, probe_blocks) O(acid_loop_cfg, signal_poly)
  O(acid_loop_cfg, tau_schedule)
  P(acid_step_log) O(acid_step_log, ms) P(acid_loop_state) O(acid_loop_state, k_rate)
  return 0;
}
"""


def test_ctypes_layout_matches_c(tmp_path):
    from paper_2607_12358_gb300 import _capi as A

    c = tmp_path / "probe.c"
    c.write_text(_PROBE)
    exe = tmp_path / "probe"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.dirname(HEADER), str(c), "-o", str(exe)], check=True)
    lines = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    for line in filter(None, lines):
        key, val = line.split()
        val = int(val)
        if "." in key:
            t, f = key.split(".")
            assert getattr(getattr(A, t), f).offset == val, key
        else:
            assert ctypes.sizeof(getattr(A, key)) == val, key


def test_host_validation_without_gpu(lib):
    from paper_2607_12358_gb300 import _capi as A

    d = A.acid_block_desc(kind=A.ACID_BLOCK_WAN, dtype=A.ACID_BF16, d=1536, heads=12, ffn=8960, grid_f=21,
                          grid_h=30, grid_w=52, n_text=512, rope_theta=1e4, ln_eps=1e-6)
    b = ctypes.c_size_t()
    assert lib.acid_block_workspace_size(ctypes.byref(d), ctypes.byref(b)) == A.ACID_OK
    assert b.value > 32760 * 1536 * 2 * 7
    rows = ctypes.c_int64()
    assert lib.acid_block_rows(ctypes.byref(d), ctypes.byref(rows)) == A.ACID_OK and rows.value == 32760
    d.heads = 7  # 1536 / 7 is not an integer
    assert lib.acid_block_workspace_size(ctypes.byref(d), ctypes.byref(b)) == A.ACID_ERR_INVALID_ARG
    assert b"heads" in lib.acid_last_error()
    d.heads = 48  # head_dim 32: not a tcgen05 attention shape
    assert lib.acid_block_workspace_size(ctypes.byref(d), ctypes.byref(b)) == A.ACID_ERR_UNSUPPORTED
    d.heads, d.d = 12, 1000
    assert lib.acid_block_workspace_size(ctypes.byref(d), ctypes.byref(b)) != A.ACID_OK
    # null output of the drift signal is rejected before any device work
    assert lib.acid_drift_signal(None, None, 10, A.ACID_BF16, None, None, None, 0, None) == A.ACID_ERR_INVALID_ARG
    assert lib.acid_drift_signal(None, None, 10, 7, None, None, None, 0, None) == A.ACID_ERR_INVALID_ARG
    assert lib.acid_cache_apply(None, None, None, 10, A.ACID_BF16, None) == A.ACID_ERR_INVALID_ARG
    assert lib.acid_cache_apply(None, None, None, 0, A.ACID_BF16, None) == A.ACID_OK
    # the failure-path diagnostic validates its budget before launching anything
    assert lib.acid_selftest_wait_timeout(10, None) == A.ACID_ERR_INVALID_ARG
    assert lib.acid_linear_forward(A.ACID_BF16, None, 64, 10, 64, None, None, 64, None, 64, 9, None, None, 0, 0,
                                   None) == A.ACID_ERR_INVALID_ARG
    # zero rows are a valid empty call (no launch, null pointers allowed);
    # negative rows or an empty key set are not
    for nq, nk, want in ((0, 4, A.ACID_OK), (-1, 4, A.ACID_ERR_INVALID_ARG), (0, 0, A.ACID_ERR_INVALID_ARG)):
        assert lib.acid_attention_forward(A.ACID_BF16, None, 64, None, 64, None, 64, None, 64, nq, nk, 1, 64,
                                          None, 0, None) == want
    for M, want in ((0, A.ACID_OK), (-1, A.ACID_ERR_INVALID_ARG), (4, A.ACID_ERR_INVALID_ARG)):
        assert lib.acid_linear_forward(A.ACID_BF16, None, 64, M, 64, None, None, 64, None, 64, A.ACID_EPI_BIAS,
                                       None, None, 0, 0, None) == want
    n = ctypes.c_size_t()
    assert lib.acid_attention_workspace_size(128, ctypes.byref(n)) == A.ACID_OK and n.value > 0
    # TEMNI drift: shapes, pointers, alignment and workspace are checked before
    # any device work (the pointer values below are never dereferenced)
    f = lib.acid_temni_drift
    out = ctypes.c_double()
    po = ctypes.byref(out)
    assert f(None, None, None, None, 10, 1004, 1e-6, po, None, None, 0, None) == A.ACID_ERR_UNSUPPORTED  # d % 8
    assert f(None, None, None, None, 10, 4096, 1e-6, po, None, None, 0, None) == A.ACID_ERR_UNSUPPORTED  # d > 3072
    assert f(None, None, None, None, -1, 1536, 1e-6, po, None, None, 0, None) == A.ACID_ERR_INVALID_ARG
    assert f(None, None, None, None, 10, 1536, 1e-6, None, None, None, 0, None) == A.ACID_ERR_INVALID_ARG
    assert f(None, None, None, None, 10, 1536, 1e-6, po, None, None, 0, None) == A.ACID_ERR_INVALID_ARG
    assert f(8, 16, 16, 16, 10, 1536, 1e-6, po, None, 256, 1 << 20, None) == A.ACID_ERR_UNSUPPORTED  # misaligned
    assert f(16, 16, 16, 16, 10, 1536, 1e-6, po, None, None, 0, None) == A.ACID_ERR_WORKSPACE
    assert f(16, 16, 16, 16, 10, 1536, 1e-6, po, None, 256, 100, None) == A.ACID_ERR_WORKSPACE
    assert b"workspace too small" in lib.acid_last_error()


def test_loop_workspace_size_without_gpu(lib):
    """The model validation and workspace query are host-only."""
    import acid_synth as S
    from paper_2607_12358_gb300 import _capi as A
    from paper_2607_12358_gb300.acid import block_desc

    cfg = S.get_config("wan")
    m = A.acid_model()
    m.block = block_desc(cfg, "wan")
    m.n_blocks = 30
    blocks = (A.acid_block_weights * 30)()
    for b in blocks:
        for f in ("mod", "qkv", "o", "ff1", "ff2", "cq", "ckv", "co"):
            setattr(b, f, A.acid_linear(16, None))  # dummy non-null pointers; never dereferenced
    m.blocks = ctypes.cast(blocks, ctypes.POINTER(A.acid_block_weights))
    m.latent_c, m.latent_f, m.latent_h, m.latent_w = cfg.latent_shape
    m.pt, m.ph, m.pw = 1, 2, 2
    m.time_freq_dim = 256
    m.d_text = 4096
    for f in ("patch", "time1", "time2", "text", "final_mod", "final_out"):
        setattr(m, f, A.acid_linear(16, None))
    n = ctypes.c_size_t()
    assert lib.acid_loop_workspace_size(ctypes.byref(m), ctypes.byref(n)) == A.ACID_OK, lib.acid_last_error()
    assert n.value > 32760 * 1536 * 4 * 4
    m.latent_w = 103  # not divisible by the patch
    assert lib.acid_loop_workspace_size(ctypes.byref(m), ctypes.byref(n)) == A.ACID_ERR_INVALID_ARG
