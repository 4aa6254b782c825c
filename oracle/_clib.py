"""Builds and loads the oracle's C part (``pvs_ref.c``) with gcc.

Test infrastructure only (see the package docstring).  The library is built
at -O0 with -frounding-math and -ffp-contract=off so that every operation
runs in the rounding mode that ``pvs_ref.c`` sets around it.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pvs_ref.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_OUT_DIR, "liborc.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``pvs_ref.c`` into ``oracle/_build/liborc.so``; return its path."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O0", "-std=c11", "-frounding-math", "-ffp-contract=off",
           "-fno-fast-math", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def lib() -> ctypes.CDLL:
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            L = ctypes.CDLL(path)
            P = ctypes.c_void_p
            i32, i64, f32 = ctypes.c_int32, ctypes.c_int64, ctypes.c_float
            L.orc_norm_bound.restype = f32
            L.orc_norm_bound.argtypes = [P, i32]
            L.orc_gamma.restype = f32
            L.orc_gamma.argtypes = [i32]
            L.orc_quantize.restype = i32
            L.orc_quantize.argtypes = [P, i64, i32, P, i32, P, P, P, P]
            L.orc_global_scale.restype = ctypes.c_float
            L.orc_global_scale.argtypes = [P, i64, i32]
            L.orc_quantize_fixed.restype = i32
            L.orc_quantize_fixed.argtypes = [P, i64, i32, P, i32, ctypes.c_float, P, P, P, P]
            L.orc_qhat_norm.restype = f32
            L.orc_qhat_norm.argtypes = [P, f32, i32, P]
            L.orc_interval_one.restype = None
            L.orc_interval_one.argtypes = [i64, f32, f32, f32, f32, f32, f32, f32, f32, P, P]
            L.orc_intervals.restype = None
            L.orc_intervals.argtypes = [P, f32, f32, f32, f32, f32, P, i64, i32, i32,
                                        P, P, P, P, P]
            _lib = L
    return _lib
