"""Seeded synthetic inputs shared by the oracle tests, the GPU tests and the bench.

This package holds no arithmetic of the draft model.  It turns
(seed, tensor tag, element index) into numbers through a counter-based
SplitMix64 stream (see ``gen.c``) and lays them out in the shapes the
draft round takes.  Both the CPU oracle and the CUDA path receive the very
same host arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gen.c")
_LIB = os.path.join(_HERE, "libsynth.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``libsynth.so`` with gcc (no FMA contraction, so every machine
    produces identical bits)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
             _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            u64, i64, dbl, vp = ctypes.c_uint64, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p
            lib.synth_splitmix64_next.argtypes = [ctypes.POINTER(u64)]
            lib.synth_splitmix64_next.restype = u64
            lib.synth_raw.argtypes = [u64, u64, u64]
            lib.synth_raw.restype = u64
            lib.synth_normal_f32.argtypes = [u64, u64, dbl, dbl, i64, vp]
            lib.synth_normal_bf16.argtypes = [u64, u64, dbl, dbl, i64, vp]
            lib.synth_uniform_i32.argtypes = [u64, u64, i64, i64, i64, vp]
            lib.synth_uniform_f64.argtypes = [u64, u64, i64, vp]
            for f in (lib.synth_normal_f32, lib.synth_normal_bf16,
                      lib.synth_uniform_i32, lib.synth_uniform_f64):
                f.restype = None
            _lib = lib
    return _lib


def tag(name: str) -> int:
    """64-bit FNV-1a hash of a tensor name: the stream tag of that tensor."""
    h = 0xcbf29ce484222325
    for b in name.encode():
        h ^= b
        h = (h * 0x100000001b3) & 0xFFFFFFFFFFFFFFFF
    return h


def splitmix64_sequence(state: int, n: int) -> list[int]:
    s = ctypes.c_uint64(state)
    lib = _load()
    return [int(lib.synth_splitmix64_next(ctypes.byref(s))) for _ in range(n)]


def raw(seed: int, name: str, i: int) -> int:
    return int(_load().synth_raw(seed, tag(name), i))


def normal(seed: int, name: str, shape, sigma: float, dtype: str, mean: float = 0.0) -> np.ndarray:
    """Normal-shaped draws (Irwin-Hall of eight 16-bit uniforms) of the given
    standard deviation.  ``dtype`` "bf16" returns the bf16 bit patterns as
    uint16 (round to nearest even); "f32" returns float32."""
    n = int(np.prod(shape, dtype=np.int64))
    if dtype == "bf16":
        out = np.empty(shape, dtype=np.uint16)
        _load().synth_normal_bf16(seed, tag(name), mean, sigma, n, out.ctypes.data)
    elif dtype == "f32":
        out = np.empty(shape, dtype=np.float32)
        _load().synth_normal_f32(seed, tag(name), mean, sigma, n, out.ctypes.data)
    else:
        raise ValueError(dtype)
    return out


def uniform_int(seed: int, name: str, shape, lo: int, hi: int) -> np.ndarray:
    """Uniform integers in [lo, hi] (inclusive), int32."""
    out = np.empty(shape, dtype=np.int32)
    n = int(np.prod(shape, dtype=np.int64))
    _load().synth_uniform_i32(seed, tag(name), lo, hi - lo + 1, n, out.ctypes.data)
    return out


def uniform01(seed: int, name: str, shape) -> np.ndarray:
    out = np.empty(shape, dtype=np.float64)
    n = int(np.prod(shape, dtype=np.int64))
    _load().synth_uniform_f64(seed, tag(name), n, out.ctypes.data)
    return out


def bf16_to_f32(a: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns (uint16) to float32 (exact)."""
    return (a.astype(np.uint32) << 16).view(np.float32)


from .workloads import (Shape, Workload, WORKLOADS, make_weights,  # noqa: E402
                        make_round_inputs, make_targets, make_tree_targets, max_ctx_of)

__all__ = ["build", "tag", "normal", "uniform_int", "uniform01", "raw",
           "splitmix64_sequence", "bf16_to_f32", "Shape", "Workload",
           "WORKLOADS", "make_weights", "make_round_inputs", "make_targets",
           "make_tree_targets", "max_ctx_of"]
