"""ctypes loader for the in-tree libeqb.so (C ABI declared in include/eqb.h).

There is no fallback: if the library is missing or fails to load, every call
raises.  Build it with ``python -m paper_2609_28053_gb300.build``.
"""
from __future__ import annotations

import ctypes
import os
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libeqb.so")

EXPORTS = (
    "eqb_status_string", "eqb_version", "eqb_target_rank", "eqb_route_topk",
    "eqb_margin_hist_pass1", "eqb_margin_hist_pass2", "eqb_select_quantile",
    "eqb_bias_update", "lei_inject_grad", "eqb_router_logits", "eqb_layer_workspace_bytes",
    "eqb_layer_step", "eqb_layer_step_noalloc", "eqb_router_route",
    "eqb_router_layer_step", "eqb_maxvio", "gshard_inject_grad",
    "eqb_rank_averaged_bias", "eqb_fixed_hist_bias", "eqb_rank_averaged_workspace_bytes",
    "eqb_selftest_stalled_wait", "lei_coefficients", "eqb_margin_hist_lei", "eqb_route_hist_fused",
)

STATUS = {0: "EQB_OK", 1: "EQB_ERR_INVALID_ARG", 2: "EQB_ERR_UNSUPPORTED", 3: "EQB_ERR_CUDA",
          4: "EQB_ERR_NONFINITE", 5: "EQB_ERR_RANK"}

_lock = threading.Lock()
_lib = None


class EqbError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {STATUS.get(status, status)}")


def load(path: str | None = None) -> ctypes.CDLL:
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(
                f"libeqb.so not found at {p}: build the CUDA extension first "
                "(python -m paper_2609_28053_gb300.build); there is no CPU fallback")
        lib = ctypes.CDLL(p)
        P, i64, i32, f32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float
        sigs = {
            "eqb_route_topk": [P, P, i64, i32, i32, P, i32, P, P, P, P, P, P],
            "eqb_margin_hist_pass1": [P, P, i64, i32, P, P, P],
            "eqb_margin_hist_pass2": [P, P, i64, i32, P, P, P],
            "eqb_select_quantile": [P, i32, i32, i64, P, P, P, P, P],
            "eqb_bias_update": [P, i32, P, P],
            "lei_inject_grad": [P, P, P, i32, i64, i32, i32, f32, f32, P],
            "lei_coefficients": [P, P, i32, i32, i32, f32, f32, P, P],
            "eqb_margin_hist_lei": [P, P, i64, i32, i32, P, P, P, P, P, P, i32, i64, i64, P],
            "eqb_route_hist_fused": [P, P, i64, i32, i32, P, i32, P, P, P, P, P, P],
            "eqb_router_logits": [P, P, i64, i32, i32, P, P, P],
            "eqb_maxvio": [P, P, i32, i32, i32, P, P, P],
            "eqb_selftest_stalled_wait": [P, i32, P],
            "gshard_inject_grad": [P, P, P, P, i32, i64, i32, i32, f32, P],
            "eqb_rank_averaged_bias": [P, P, i64, i32, i32, P, i32, P, P, P, ctypes.c_size_t, P, P],
            "eqb_fixed_hist_bias": [P, P, i64, i32, i32, f32, f32, P, P, P, ctypes.c_size_t, P, P],
            "eqb_router_route": [P, P, i64, i32, i32, i32, P, P, i32, P, P, P, P, P, P, P],
            "eqb_router_layer_step": [P, P, i64, i32, i32, i32, P, P, P, i32, i64, P, P, P, P, P, P,
                                      f32, f32, P, ctypes.c_size_t, P, P],
            "eqb_layer_step": [P, P, i64, i32, i32, P, P, i32, i64, P, P, P, P, P, f32, f32, P,
                               ctypes.c_size_t, P, P],
            "eqb_layer_step_noalloc": [P, P, i64, i32, i32, P, P, i32, i64, P, P, P, P, P, f32,
                                       f32, P, P],
        }
        for name, args in sigs.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        lib.eqb_status_string.argtypes = [ctypes.c_int]
        lib.eqb_status_string.restype = ctypes.c_char_p
        lib.eqb_version.argtypes = []
        lib.eqb_version.restype = ctypes.c_int
        lib.eqb_layer_workspace_bytes.argtypes = [i32]
        lib.eqb_layer_workspace_bytes.restype = ctypes.c_size_t
        lib.eqb_rank_averaged_workspace_bytes.argtypes = [i32, i32]
        lib.eqb_rank_averaged_workspace_bytes.restype = ctypes.c_size_t
        lib.eqb_target_rank.argtypes = [i64, i32, i32]
        lib.eqb_target_rank.restype = i64
        if path is None:
            _lib = lib
        return lib
