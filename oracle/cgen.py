"""ctypes access to the oracle's C regenerator (oracle/csrc/ogen.c).

Test infrastructure only. ``build()`` compiles the C file with gcc into
``oracle/_ogen.so``; ``available()`` says whether it is loadable. The pure
numpy path in ``oracle.weights`` is the fallback and the two are pinned to
each other bit-exactly in the tests.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "csrc", "ogen.c")
_SO = os.path.join(_HERE, "_ogen.so")
_lib = None


def build(force: bool = False) -> str:
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-pthread",
               _SRC, "-o", _SO, "-lm"]
        subprocess.run(cmd, check=True)
    return _SO


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(_SO):
            build()
        lib = ctypes.CDLL(_SO)
        lib.og_stream_key.restype = ctypes.c_uint64
        lib.og_stream_key.argtypes = [ctypes.c_uint64] * 4
        lib.og_normal.restype = None
        lib.og_normal.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64, ctypes.c_float,
                                  ctypes.c_void_p]
        lib.og_quant_row.restype = None
        lib.og_quant_row.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]
        lib.og_weight_int8.restype = ctypes.c_int
        lib.og_weight_int8.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                       ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int]
        lib.og_quant_row_grouped.restype = None
        lib.og_quant_row_grouped.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
                                             ctypes.c_void_p]
        lib.og_weight_int8_grouped.restype = ctypes.c_int
        lib.og_weight_int8_grouped.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                               ctypes.c_int64, ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p,
                                               ctypes.c_int]
        _lib = lib
    return _lib


def available() -> bool:
    try:
        _load()
        return True
    except Exception:
        return False


def n_threads() -> int:
    return max(1, min(64, os.cpu_count() or 1))


def stream_key(seed: int, tensor: int, layer: int, sub: int) -> int:
    return int(_load().og_stream_key(seed, tensor, layer, sub))


def normal(key: int, start: int, count: int, sigma: float) -> np.ndarray:
    out = np.empty(count, dtype=np.float32)
    _load().og_normal(key, start, count, sigma, out.ctypes.data)
    return out


def quant_row(w: np.ndarray):
    w = np.ascontiguousarray(w, dtype=np.float32)
    q = np.empty(w.shape[0], dtype=np.int8)
    s = np.empty(1, dtype=np.float32)
    _load().og_quant_row(w.ctypes.data, w.shape[0], q.ctypes.data, s.ctypes.data)
    return q, s[0]


def weight_int8(key: int, row0: int, nrows: int, cols: int, sigma: float):
    q = np.empty((nrows, cols), dtype=np.int8)
    s = np.empty(nrows, dtype=np.float32)
    rc = _load().og_weight_int8(key, row0, nrows, cols, sigma, q.ctypes.data, s.ctypes.data, n_threads())
    if rc != 0:
        raise RuntimeError(f"og_weight_int8 failed with {rc}")
    return q, s


def quant_row_grouped(w: np.ndarray, group: int):
    w = np.ascontiguousarray(w, dtype=np.float32)
    q = np.empty(w.shape[0], dtype=np.int8)
    s = np.empty(w.shape[0] // group, dtype=np.float32)
    _load().og_quant_row_grouped(w.ctypes.data, w.shape[0], group, q.ctypes.data, s.ctypes.data)
    return q, s


def weight_int8_grouped(key: int, row0: int, nrows: int, cols: int, group: int, sigma: float):
    q = np.empty((nrows, cols), dtype=np.int8)
    s = np.empty((nrows, cols // group), dtype=np.float32)
    rc = _load().og_weight_int8_grouped(key, row0, nrows, cols, group, sigma, q.ctypes.data, s.ctypes.data,
                                        n_threads())
    if rc != 0:
        raise RuntimeError(f"og_weight_int8_grouped failed with {rc}")
    return q, s
