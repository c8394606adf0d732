"""ctypes mirror of include/acid.h and the loader of libacid_gb300.so.

Loading fails loudly (ImportError) when the library has not been built:
there is no other implementation behind these names.
"""

from __future__ import annotations

import ctypes as C
import os

# ACID_LIBRARY=debug selects the debug build (kernel memory-index checks, see
# acid_bounds_report in include/acid.h), built by `build.py --debug`.
_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)),
                         "libacid_gb300_debug.so" if os.environ.get("ACID_LIBRARY") == "debug" else "libacid_gb300.so")

ACID_OK, ACID_ERR_INVALID_ARG, ACID_ERR_UNSUPPORTED, ACID_ERR_WORKSPACE, ACID_ERR_CUDA, ACID_ERR_TIMEOUT = range(6)
ACID_BF16, ACID_FP32 = 0, 1
ACID_BLOCK_WAN, ACID_BLOCK_COG, ACID_BLOCK_HV_DUAL, ACID_BLOCK_HV_SINGLE = range(4)
ACID_METHOD_TEACACHE, ACID_METHOD_EASYCACHE, ACID_METHOD_DICACHE = 0, 1, 2
ACID_EPI_BIAS, ACID_EPI_GELU, ACID_EPI_GATED_RES, ACID_EPI_RES = 0, 1, 3, 4

STATUS_NAMES = {0: "ACID_OK", 1: "ACID_ERR_INVALID_ARG", 2: "ACID_ERR_UNSUPPORTED", 3: "ACID_ERR_WORKSPACE",
                4: "ACID_ERR_CUDA", 5: "ACID_ERR_TIMEOUT"}


class acid_block_desc(C.Structure):
    _fields_ = [("kind", C.c_int32), ("dtype", C.c_int32), ("d", C.c_int32), ("heads", C.c_int32),
                ("ffn", C.c_int32), ("grid_f", C.c_int32), ("grid_h", C.c_int32), ("grid_w", C.c_int32),
                ("n_text", C.c_int64), ("rope_theta", C.c_float), ("ln_eps", C.c_float)]


class acid_linear(C.Structure):
    _fields_ = [("w", C.c_void_p), ("b", C.c_void_p)]


_BW_FIELDS = ["mod", "qkv", "o", "ff1", "ff2", "cq", "ckv", "co", "t_mod", "t_qkv", "t_o", "t_ff1", "t_ff2"]


class acid_block_weights(C.Structure):
    _fields_ = [(n, acid_linear) for n in _BW_FIELDS]


class acid_cond(C.Structure):
    _fields_ = [("temb", C.c_void_p), ("ctx", C.c_void_p), ("ctx_kv", C.c_void_p)]


class acid_model(C.Structure):
    _fields_ = [("block", acid_block_desc), ("n_blocks", C.c_int32), ("n_single", C.c_int32),
                ("blocks", C.POINTER(acid_block_weights)),
                ("latent_c", C.c_int32), ("latent_f", C.c_int32), ("latent_h", C.c_int32), ("latent_w", C.c_int32),
                ("pt", C.c_int32), ("ph", C.c_int32), ("pw", C.c_int32), ("time_freq_dim", C.c_int32),
                ("d_text", C.c_int32),
                ("patch", acid_linear), ("time1", acid_linear), ("time2", acid_linear), ("text", acid_linear),
                ("final_mod", acid_linear), ("final_out", acid_linear)]


class acid_loop_cfg(C.Structure):
    _fields_ = [("n_steps", C.c_int32), ("warmup", C.c_int32), ("method", C.c_int32), ("force_last", C.c_int32),
                ("tau_low", C.c_double), ("tau_high", C.c_double), ("delta", C.c_double), ("shift", C.c_double),
                ("forced", C.POINTER(C.c_int8)), ("probe_blocks", C.c_int32), ("signal_poly_n", C.c_int32),
                ("signal_poly", C.POINTER(C.c_double)), ("tau_schedule", C.POINTER(C.c_double))]


class acid_step_log(C.Structure):
    _fields_ = [("step", C.c_int32), ("warmup", C.c_int32), ("computed", C.c_int32), ("forced", C.c_int32),
                ("t", C.c_double), ("signal", C.c_double), ("dsignal", C.c_double), ("tau", C.c_double),
                ("sigma", C.c_double), ("ms", C.c_double)]


class acid_loop_state(C.Structure):
    _fields_ = [("step", C.c_int32), ("have_prev_signal", C.c_int32), ("have_cache", C.c_int32),
                ("have_rate", C.c_int32), ("sigma_acc", C.c_double), ("s_prev", C.c_double),
                ("k_rate", C.c_double)]


_P = C.c_void_p
_PROTOS = {
    "acid_last_error": (C.c_char_p, []),
    "acid_version": (C.c_char_p, []),
    "acid_check_device_error": (C.c_int, []),
    "acid_selftest_wait_timeout": (C.c_int, [C.c_int64, _P]),
    "acid_bounds_report": (C.c_int, [C.POINTER(C.c_int32), C.POINTER(C.c_int64), C.POINTER(C.c_int64),
                                     C.POINTER(C.c_int64)]),
    "acid_selftest_bounds": (C.c_int, [_P]),
    "acid_launch_count": (C.c_int64, []),
    "acid_profile_enable": (C.c_int, [C.c_int32]),
    "acid_profile_read": (C.c_int, [C.c_int32, C.POINTER(C.c_int64), C.POINTER(C.c_double),
                                    C.POINTER(C.c_double)]),
    "acid_drift_workspace_size": (C.c_int, [C.c_int64, C.POINTER(C.c_size_t)]),
    "acid_drift_signal": (C.c_int, [_P, _P, C.c_int64, C.c_int32, _P, _P, _P, C.c_size_t, _P]),
    "acid_cache_apply": (C.c_int, [_P, _P, _P, C.c_int64, C.c_int32, _P]),
    "acid_temni_drift": (C.c_int, [_P, _P, _P, _P, C.c_int64, C.c_int32, C.c_float, _P, _P, _P, C.c_size_t, _P]),
    "acid_drift_signal_noalloc": (C.c_int, [_P, _P, C.c_int64, C.c_int32, _P, _P, _P]),
    "acid_drift_apply": (C.c_int, [_P, _P, _P, _P, C.c_int64, C.c_int32, _P, _P, _P, C.c_size_t, _P]),
    "acid_linear_forward": (C.c_int, [C.c_int32, _P, C.c_int64, C.c_int64, C.c_int32, _P, _P, C.c_int32, _P,
                                      C.c_int64, C.c_int32, _P, _P, C.c_int64, C.c_int32, _P]),
    "acid_attention_forward": (C.c_int, [C.c_int32, _P, C.c_int64, _P, C.c_int64, _P, C.c_int64, _P, C.c_int64,
                                         C.c_int64, C.c_int64, C.c_int32, C.c_int32, _P, C.c_size_t, _P]),
    "acid_attention_workspace_size": (C.c_int, [C.c_int32, C.POINTER(C.c_size_t)]),
    "acid_layernorm_mod": (C.c_int, [C.c_int32, _P, C.c_int32, _P, C.c_int64, C.c_int32, _P, _P, C.c_float, _P]),
    "acid_block_rows": (C.c_int, [C.POINTER(acid_block_desc), C.POINTER(C.c_int64)]),
    "acid_block_workspace_size": (C.c_int, [C.POINTER(acid_block_desc), C.POINTER(C.c_size_t)]),
    "acid_dit_block_forward": (C.c_int, [C.POINTER(acid_block_desc), _P, C.POINTER(acid_cond),
                                         C.POINTER(acid_block_weights), _P, C.c_size_t, _P]),
    "acid_loop_workspace_size": (C.c_int, [C.POINTER(acid_model), C.POINTER(C.c_size_t)]),
    "acid_loop_begin": (C.c_int, [C.POINTER(acid_model), C.POINTER(acid_loop_cfg), _P, C.POINTER(acid_loop_state),
                                  _P, C.c_size_t, _P]),
    "acid_denoise_step": (C.c_int, [C.POINTER(acid_model), C.POINTER(acid_loop_cfg), C.POINTER(acid_loop_state), _P,
                                    C.POINTER(acid_step_log), _P, C.c_size_t, _P]),
    "acid_denoise_loop": (C.c_int, [C.POINTER(acid_model), C.POINTER(acid_loop_cfg), _P, _P,
                                    C.POINTER(acid_step_log), _P, C.c_size_t, _P]),
    "acid_denoise_loop_graph": (C.c_int, [C.POINTER(acid_model), C.POINTER(acid_loop_cfg), _P, _P,
                                          C.POINTER(acid_step_log), _P, C.c_size_t, _P]),
    "acid_guided_workspace_size": (C.c_int, [C.POINTER(acid_model), C.POINTER(C.c_size_t)]),
    "acid_guided_begin": (C.c_int, [C.POINTER(acid_model), C.POINTER(acid_loop_cfg), C.POINTER(acid_loop_cfg), _P, _P,
                                    C.POINTER(acid_loop_state), C.POINTER(acid_loop_state), _P, C.c_size_t, _P]),
    "acid_guided_step": (C.c_int, [C.POINTER(acid_model), C.POINTER(acid_loop_cfg), C.POINTER(acid_loop_cfg),
                                   C.c_double, C.POINTER(acid_loop_state), C.POINTER(acid_loop_state), _P,
                                   C.POINTER(acid_step_log), C.POINTER(acid_step_log), _P, C.c_size_t, _P]),
    "acid_denoise_loop_guided": (C.c_int, [C.POINTER(acid_model), C.POINTER(acid_loop_cfg), C.POINTER(acid_loop_cfg),
                                           C.c_double, _P, _P, _P, C.POINTER(acid_step_log),
                                           C.POINTER(acid_step_log), _P, C.c_size_t, _P]),
    "acid_denoise_loop_guided_graph": (C.c_int, [C.POINTER(acid_model), C.POINTER(acid_loop_cfg),
                                                 C.POINTER(acid_loop_cfg), C.c_double, _P, _P, _P,
                                                 C.POINTER(acid_step_log), C.POINTER(acid_step_log), _P, C.c_size_t,
                                                 _P]),
}

_lib = None


def lib_path() -> str:
    return _LIB_PATH


def load() -> C.CDLL:
    """The loaded library (raises ImportError if it is not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise ImportError(f"{_LIB_PATH} is missing: build it with "
                              "`python -c 'import __graft_entry__ as g; g.build()'`")
        lib = C.CDLL(_LIB_PATH)
        for name, (res, args) in _PROTOS.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


class AcidError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def check(status: int) -> None:
    if status != ACID_OK:
        raise AcidError(status, load().acid_last_error().decode())
