"""ctypes mirror of include/dflow.h.  Loading fails loudly when the library is missing."""
from __future__ import annotations

import ctypes
import os

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libdflow.so")

DFLOW_F32, DFLOW_BF16 = 0, 1
MAX_FEAT = 8

STATUS = {0: "DFLOW_OK", 1: "DFLOW_ERR_INVALID_ARG", 2: "DFLOW_ERR_CUDA", 3: "DFLOW_ERR_CAPACITY",
          4: "DFLOW_ERR_DEVICE_TIMEOUT", 5: "DFLOW_ERR_UNSUPPORTED", 6: "DFLOW_ERR_BAD_STATE"}

c_i32p = ctypes.POINTER(ctypes.c_int32)


class Config(ctypes.Structure):
    _fields_ = [("dtype", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_layers", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("d_inter", ctypes.c_int32), ("vocab", ctypes.c_int32), ("draft_layers", ctypes.c_int32),
                ("n_feat", ctypes.c_int32), ("feat_layers", ctypes.c_int32 * MAX_FEAT),
                ("block", ctypes.c_int32), ("page_size", ctypes.c_int32), ("max_batch", ctypes.c_int32),
                ("max_ctx", ctypes.c_int32), ("num_pages", ctypes.c_int32), ("rope_theta", ctypes.c_float),
                ("rms_eps", ctypes.c_float), ("ln_eps", ctypes.c_float)]


class LayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("w_qkv", "w_o", "w_gate_up", "w_down", "attn_norm", "mlp_norm", "q_norm", "k_norm")]


class Weights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("lm_head", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("target", ctypes.POINTER(LayerWeights)), ("draft", ctypes.POINTER(LayerWeights)),
                ("draft_final_norm", ctypes.c_void_p), ("w_c", ctypes.c_void_p), ("c_norm", ctypes.c_void_p),
                ("e_mask", ctypes.c_void_p), ("relay_w1", ctypes.c_void_p), ("relay_w2", ctypes.c_void_p),
                ("ln_w", ctypes.c_void_p), ("ln_b", ctypes.c_void_p)]


class State(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("tokens", ctypes.c_void_p), ("seq_len", ctypes.c_void_p),
                ("page_table", ctypes.c_void_p), ("kv", ctypes.c_void_p), ("draft_kv", ctypes.c_void_p),
                ("carry", ctypes.c_void_p), ("n_carry", ctypes.c_void_p), ("boundary", ctypes.c_void_p),
                ("active", ctypes.c_void_p), ("status", ctypes.c_void_p)]


class KernelProfile(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_int64), ("total_ms", ctypes.c_double), ("alg_bytes", ctypes.c_double),
                ("alg_flops", ctypes.c_double)]


PROF_GEMM, PROF_ATTN, PROF_OTHER, PROF_N = 0, 1, 2, 3

# (name, argtypes) of every exported function of include/dflow.h
_P = ctypes.c_void_p
_SIGS = {
    "dflow_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "dflow_create": ([ctypes.POINTER(Config), ctypes.POINTER(Weights), ctypes.POINTER(_P)], ctypes.c_int),
    "dflow_workspace_size": ([_P, ctypes.POINTER(ctypes.c_size_t)], ctypes.c_int),
    "dflow_set_workspace": ([_P, _P, ctypes.c_size_t], ctypes.c_int),
    "dflow_destroy": ([_P], ctypes.c_int),
    "dflow_prefill": ([_P, ctypes.POINTER(State), _P, ctypes.c_int32, c_i32p, _P], ctypes.c_int),
    "dflow_draft_block": ([_P, ctypes.POINTER(State), _P, _P, _P], ctypes.c_int),
    "dflow_verify_block": ([_P, ctypes.POINTER(State), _P, _P, _P, _P, _P], ctypes.c_int),
    "dflow_accept_commit": ([_P, ctypes.POINTER(State), _P, _P, _P, _P, _P, _P], ctypes.c_int),
    "dflow_carry_hidden": ([_P, ctypes.POINTER(State), _P, _P, _P, _P], ctypes.c_int),
    "dflow_decode_step": ([_P, ctypes.POINTER(State), _P, ctypes.c_int32, _P], ctypes.c_int),
    "dflow_round": ([_P, ctypes.POINTER(State), _P, _P, _P, ctypes.c_int32, _P], ctypes.c_int),
    "dflow_round_sampled": ([_P, ctypes.POINTER(State), ctypes.c_uint64, ctypes.c_int32, _P, _P, ctypes.c_int32, _P,
                             _P, _P], ctypes.c_int),
    "dflow_read_status": ([_P, ctypes.POINTER(State), c_i32p, _P], ctypes.c_int),
    "dflow_profile_enable": ([_P, ctypes.c_int32], ctypes.c_int),
    "dflow_profile_read": ([_P, ctypes.POINTER(KernelProfile)], ctypes.c_int),
    "dflow_launch_count": ([_P, ctypes.POINTER(ctypes.c_uint64)], ctypes.c_int),
    "dflow_greedy_tokens_noalloc": ([_P, ctypes.c_int32, ctypes.c_int32, _P, ctypes.c_int32, _P, _P], ctypes.c_int),
    "dflow_debug_seq_schedule": ([ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, c_i32p, c_i32p],
                                 ctypes.c_int),
    "dflow_debug_wide_schedule": ([ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64,
                                   c_i32p, c_i32p, ctypes.c_int32], ctypes.c_int),
    "dflow_debug_gemm": ([_P, ctypes.c_int32, _P, ctypes.c_int32, ctypes.c_int32, _P, ctypes.c_int32, ctypes.c_int32,
                          ctypes.c_int32, _P, ctypes.c_int32, _P, _P], ctypes.c_int),
}
EXPORTS = tuple(_SIGS)

_lib = None


class DFlowError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} returned {STATUS.get(code, code)}")
        self.code = code


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2609_06498_gb300.build.build()")
        l = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGS.items():
            f = getattr(l, name)
            f.argtypes = args
            f.restype = res
        _lib = l
    return _lib


def call(name: str, *args) -> None:
    code = getattr(lib(), name)(*args)
    if code != 0:
        raise DFlowError(name, code)
