"""ctypes front end of the counter-based generator in ``synth.c``."""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB = os.path.join(_HERE, "libdflare_synth.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``synth.c`` into ``libdflare_synth.so`` next to it (gcc, OpenMP)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB)
            u64, i64, dbl, vp = ctypes.c_uint64, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p
            L.synth_normal_f32.argtypes = [u64, u64, u64, i64, dbl, dbl, vp]
            L.synth_normal_bf16.argtypes = [u64, u64, u64, i64, dbl, dbl, vp]
            L.synth_uniform_f64.argtypes = [u64, u64, u64, i64, vp]
            L.synth_uniform_u32.argtypes = [u64, u64, u64, i64, vp]
            L.synth_randint_i32.argtypes = [u64, u64, u64, i64, i64, i64, vp]
            for f in (L.synth_normal_f32, L.synth_normal_bf16, L.synth_uniform_f64,
                      L.synth_uniform_u32, L.synth_randint_i32):
                f.restype = None
            _lib = L
    return _lib


def tensor_id(name: str) -> int:
    """64-bit FNV-1a hash of a tensor name: the generator's stream id for that tensor."""
    h = 0xCBF29CE484222325
    for b in name.encode():
        h = ((h ^ b) * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def normal(seed: int, name: str, shape, *, mean: float = 0.0, std: float = 1.0,
           dtype: str = "bf16", offset: int = 0, out: np.ndarray | None = None) -> np.ndarray:
    """Gaussian N(mean, std^2) samples of tensor `name`, elements [offset, offset + size)."""
    n = int(np.prod(shape))
    if dtype == "bf16":
        a = out if out is not None else np.empty(shape, np.uint16)
        lib().synth_normal_bf16(seed, tensor_id(name), offset, n, mean, std, a.ctypes.data)
    elif dtype == "f32":
        a = out if out is not None else np.empty(shape, np.float32)
        lib().synth_normal_f32(seed, tensor_id(name), offset, n, mean, std, a.ctypes.data)
    else:
        raise ValueError(f"dtype {dtype!r}")
    return a


def uniform(seed: int, name: str, shape, *, offset: int = 0) -> np.ndarray:
    """U(0,1) float64 samples."""
    a = np.empty(shape, np.float64)
    lib().synth_uniform_f64(seed, tensor_id(name), offset, int(np.prod(shape)), a.ctypes.data)
    return a


def uniform_u32(seed: int, name: str, shape, *, offset: int = 0) -> np.ndarray:
    """Uniform uint32 samples."""
    a = np.empty(shape, np.uint32)
    lib().synth_uniform_u32(seed, tensor_id(name), offset, int(np.prod(shape)), a.ctypes.data)
    return a


def randint(seed: int, name: str, shape, lo: int, hi: int, *, offset: int = 0) -> np.ndarray:
    """Uniform integers in [lo, hi) as int32."""
    a = np.empty(shape, np.int32)
    lib().synth_randint_i32(seed, tensor_id(name), offset, int(np.prod(shape)), lo, hi, a.ctypes.data)
    return a
