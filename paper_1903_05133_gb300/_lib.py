"""ctypes loader for libhier_avg.so (the C ABI declared in include/hier_avg.h).

There is no fallback: if the library is missing or fails to load, every call
raises.  Build it with ``paper_1903_05133_gb300._build.build()``.
"""
from __future__ import annotations

import ctypes
import os

from . import _build

c_int, c_int64, c_float, c_double = ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_double
c_void_p, c_char_p = ctypes.c_void_p, ctypes.c_char_p
P_int64, P_float, P_double = (ctypes.POINTER(c_int64), ctypes.POINTER(c_float),
                              ctypes.POINTER(c_double))

# name -> (restype, argtypes); every function of include/hier_avg.h
SIGNATURES = {
    "hier_avg_local_average_buffer": (c_int, [c_void_p, c_int64, c_int64, c_int64, c_int64, c_void_p]),
    "hier_avg_global_average_buffer": (c_int, [c_void_p, c_int64, c_int64, c_int64, c_void_p]),
    "hier_avg_local_global_average_buffer": (c_int, [c_void_p, c_int64, c_int64, c_int64, c_int64,
                                                     c_void_p]),
    "hier_avg_create": (c_int, [c_int, c_int, c_int, c_int, c_float, c_int,
                                ctypes.POINTER(c_int), c_int, c_int, ctypes.POINTER(c_void_p)]),
    "hier_avg_destroy": (None, [c_void_p]),
    "hier_avg_param_layout": (c_int, [c_void_p, P_int64, P_int64, P_int64]),
    "hier_avg_workspace_bytes": (c_int, [c_void_p, P_int64]),
    "hier_avg_bind": (c_int, [c_void_p, c_void_p, c_void_p, c_int64, c_void_p, c_void_p, c_int64,
                              c_void_p]),
    "hier_avg_step": (c_int, [c_void_p]),
    "hier_avg_local_average": (c_int, [c_void_p]),
    "hier_avg_global_average": (c_int, [c_void_p]),
    "hier_avg_round": (c_int, [c_void_p]),
    "hier_avg_round_host": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p]),
    "hier_avg_step_static": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p, c_int64, c_void_p]),
    "hier_avg_get_step": (c_int, [c_void_p, P_int64]),
    "hier_avg_set_step": (c_int, [c_void_p, c_int64]),
    "hier_avg_losses": (c_int, [c_void_p, c_void_p]),
    "hier_avg_check": (c_int, [c_void_p]),
    "hier_avg_wait_selftest": (c_int, [c_void_p, c_int64]),
    "hier_avg_profile": (c_int, [c_void_p, c_int]),
    "hier_avg_profile_kinds": (c_int, [c_void_p, ctypes.c_uint]),
    "hier_avg_launches": (c_int, [c_void_p, c_void_p]),
    "hier_avg_set_global_steps": (c_int, [c_void_p, c_int]),
    "hier_avg_set_lr": (c_int, [c_void_p, ctypes.c_float]),
    "hier_avg_set_batch": (c_int, [c_void_p, c_int]),
    "hier_avg_profile_every": (c_int, [c_void_p, c_int]),
    "hier_avg_profile_read": (c_int, [c_void_p, c_int, P_double, P_int64, P_double, P_double]),
    "hier_avg_strerror": (c_char_p, [c_int]),
    "hier_avg_last_error": (c_char_p, [c_void_p]),
}

_lib = None


def load() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        if not os.path.exists(_build.LIB_PATH):
            raise RuntimeError(
                f"{_build.LIB_PATH} is missing: the CUDA library must be built "
                "(paper_1903_05133_gb300._build.build(), needs nvcc); there is no fallback")
        lib = ctypes.CDLL(_build.LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


class HierAvgError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str = ""):
        name = load().hier_avg_strerror(status).decode()
        super().__init__(f"{where}: {name} ({status}){': ' + detail if detail else ''}")
        self.status = status


def check(status: int, where: str, handle=None) -> None:
    if status != 0:
        detail = load().hier_avg_last_error(handle).decode() if handle else ""
        raise HierAvgError(status, where, detail)
