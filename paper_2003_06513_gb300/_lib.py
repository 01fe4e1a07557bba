"""ctypes loader for libpatconv.so (the C ABI declared in include/patconv.h).

Argument marshalling only.  There is no fallback: if the library is missing or fails to load,
``load`` raises, and nothing in this package computes a convolution any other way.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

_c_int, _c_void_p, _c_size_t = ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t

# name -> (restype, argtypes); the exported symbols of include/patconv.h
SIGNATURES = {
    "pp_default_patterns": (_c_int, [ctypes.POINTER(ctypes.c_uint16), _c_int]),
    "pp_pack": (_c_int, [ctypes.POINTER(ctypes.c_float), _c_int, _c_int, _c_int, _c_int,
                         ctypes.POINTER(ctypes.c_uint16), _c_int, ctypes.c_double,
                         ctypes.POINTER(_c_void_p)]),
    "pp_query": (_c_int, [_c_void_p, _c_int, ctypes.POINTER(ctypes.c_int64)]),
    "pp_export": (_c_int, [_c_void_p, _c_int, _c_void_p, _c_size_t]),
    "pp_bind_device": (_c_int, [_c_void_p, _c_void_p, _c_size_t, _c_void_p]),
    "pp_conv": (_c_int, [_c_void_p, _c_void_p, _c_int, _c_int, _c_int, _c_int, _c_void_p, _c_int,
                         _c_void_p, _c_void_p]),
    "pp_conv_ws": (_c_int, [_c_void_p, _c_void_p, _c_int, _c_int, _c_int, _c_int, _c_void_p, _c_int,
                            _c_void_p, _c_void_p, _c_size_t, _c_void_p]),
    "pp_design_patterns": (_c_int, [ctypes.POINTER(ctypes.c_float), _c_size_t, _c_int,
                                    ctypes.POINTER(ctypes.c_uint16), ctypes.POINTER(_c_int)]),
    "pp_conv_pool_ws": (_c_int, [_c_void_p, _c_void_p, _c_int, _c_int, _c_int, _c_int, _c_void_p, _c_int,
                                 _c_void_p, _c_void_p, _c_size_t, _c_void_p]),
    "pp_conv_workspace_size": (_c_int, [_c_void_p, _c_int, _c_int, _c_int, ctypes.POINTER(_c_size_t)]),
    "pp_conv_plan": (_c_int, [_c_void_p, _c_int, _c_int, _c_int, _c_size_t, ctypes.POINTER(ctypes.c_int64),
                              _c_int]),
    "pp_conv_pool_plan": (_c_int, [_c_void_p, _c_int, _c_int, _c_int, _c_size_t,
                                   ctypes.POINTER(ctypes.c_int64), _c_int]),
    "pp_conv_plan_dt": (_c_int, [_c_void_p, _c_int, _c_int, _c_int, _c_int, _c_int, _c_size_t,
                                 ctypes.POINTER(ctypes.c_int64), _c_int]),
    "pp_conv_static_scratch": (_c_int, [_c_void_p, _c_void_p, _c_int, _c_int, _c_int, _c_int, _c_void_p,
                                        _c_int, _c_void_p, _c_void_p]),
    "pp_static_scratch_bytes": (_c_int, [ctypes.POINTER(_c_size_t)]),
    "pp_debug_inject_timeout": (_c_int, []),
    "pp_measure_fp32_peak": (_c_int, [_c_int, ctypes.POINTER(ctypes.c_double)]),
    "pp_maxpool2x2": (_c_int, [_c_void_p, _c_int, _c_int, _c_int, _c_int, _c_int, _c_void_p,
                               _c_void_p]),
    "pp_device_status": (_c_int, [_c_int, ctypes.POINTER(ctypes.c_uint)]),
    "pp_destroy": (_c_int, [_c_void_p]),
    "pp_status_string": (ctypes.c_char_p, [_c_int]),
}

_lock = threading.Lock()
_lib = None


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load (building first if needed) and return the library with typed signatures."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if build_if_missing:
            path = _build.build()
        if not os.path.exists(path):
            raise RuntimeError(f"libpatconv is not built ({path} missing); run "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        lib = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


class PatconvError(RuntimeError):
    def __init__(self, fn: str, status: int):
        msg = load().pp_status_string(status).decode()
        super().__init__(f"{fn} failed with status {status}: {msg}")
        self.status = status


def check(fn: str, status: int) -> None:
    if status != 0:
        raise PatconvError(fn, status)
