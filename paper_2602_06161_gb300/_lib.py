"""ctypes loader for libcover.so (the C ABI in include/cover.h, include/cover_debug.h).

There is no CPU fallback: if the library cannot be built or loaded, every call
raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

_P = ctypes.c_void_p
_I = ctypes.c_int
_lock = threading.Lock()
_lib = None

# name -> (restype, argtypes)
_SIGNATURES = {
    "cover_attn_fwd": (_I, [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P]),
    "cover_attn_fwd_f32": (_I, [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P]),
    "cover_attn_fwd_prefix": (_I, [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _I, _P, _P, _P]),
    "cover_attn_fwd_prefix_f32": (_I, [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _I, _P, _P, _P]),
    "cover_seed_route": (_I, [_P, _I, _I, _I, _P, _P, _P, _P]),
    "cover_seed_route_debug": (_I, [_P, _I, _I, _I, _P, _P, _P, _P]),
    "cover_score_workspace_bytes": (ctypes.c_size_t, [_I]),
    "cover_score_fwd": (_I, [_P, _I, _I, _I, _P, _P, _P, _P, _I, _P, _P, _P, _P, _P, _P, _P, _P]),
    "cover_score_fwd_noalloc": (_I, [_P, _I, _I, _I, _P, _P, _P, _P, _I, _P, _P, _P, _P, _P, _P, _P]),
    "cover_seed_kv_gather": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P]),
    "cover_seed_kv_override": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P]),
    "cover_decide_workspace_bytes": (ctypes.c_size_t, [_I, _I]),
    "cover_score_decide_fwd": (_I, [_P, _I, _I, _I, _P, _P, _P, ctypes.c_float, _I, _I, _I, _I, _I, _I, _I,
                                    _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P]),
    "cover_seed_select_fwd": (_I, [_I, _I, _P, _P, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P]),
    "cover_attn_mass_workspace_bytes": (ctypes.c_size_t, [_I, _I, _I]),
    "cover_attn_mass_fwd": (_I, [_P, _P, _P, _P, _I, _P, _I, _I, _I, _I, _I, _P, _P, _I, _I, _I, _P, _P, _P, _P]),
    "cover_device_status": (_I, [_P]),
    "cover_status_str": (ctypes.c_char_p, [_I]),
    "cover_debug_umma_tile": (_I, [_P, _P, _P, _P, _P, _P, _P]),
    "cover_debug_wait_timeout": (_I, [_I, _P]),
    "cover_debug_attn_prefix_packed": (_I, [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _I, _P, _P, _I, _I,
                                            _P]),
    "cover_debug_attn_fault": (_I, [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _I, _P, _P, _I, _I, _I,
                                    _P]),
    "cover_debug_status_detail": (_I, [_P, _P]),
    "cover_debug_window_model": (_I, [_I, _I, _I, _I, _I, _I, _I, _P, _P, _P]),
}


class CoverError(RuntimeError):
    def __init__(self, fn: str, code: int):
        self.code = code
        super().__init__(f"{fn} failed: {status_str(code)} ({code})")


def lib_path() -> str:
    return _build.LIB


def load(build_if_needed: bool = True):
    """Load libcover.so (building it first when missing or stale)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if build_if_needed:
            _build.build()
        if not os.path.exists(_build.LIB):
            raise RuntimeError(f"libcover.so not found at {_build.LIB}; run paper_2602_06161_gb300.build.build()")
        lib = ctypes.CDLL(_build.LIB)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def exported_symbols():
    return list(_SIGNATURES)


def status_str(code: int) -> str:
    return load().cover_status_str(int(code)).decode()


def check(fn: str, code: int) -> None:
    if code != 0:
        raise CoverError(fn, code)
