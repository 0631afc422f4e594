"""Seeded synthetic inputs shaped like the paper's square GEMM sweeps.

This package holds no arithmetic of the emulation method.  It wraps the
SplitMix64 counter generator in ``synth.c`` and the input recipes used by the
tests and by ``bench.py``.  The CPU oracle and the CUDA path are both fed the
very same host arrays produced here.

Input classes (Section 7.3 of the paper, "Input Matrices and Accuracy
Metrics"): uniform random entries in [-1, 1] (the class the paper reports),
and the "scaled" class ``(u - 0.5) * exp(phi * g)`` clamped into the BF16
exponent range.  Matrix A is drawn first (row-major), then B continues the
same stream.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import tempfile

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_SO = os.path.join(_HERE, "_synth.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile ``synth.c`` into ``_synth.so`` beside it (gcc, OpenMP)."""
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_HERE)
    os.close(fd)
    cmd = ["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-std=c11", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        i64, u64, vp, f64 = ctypes.c_int64, ctypes.c_uint64, ctypes.c_void_p, ctypes.c_double
        lib.synth_uniform_f64.argtypes = [u64, u64, vp, i64]
        lib.synth_uniform_f32.argtypes = [u64, u64, vp, i64]
        lib.synth_scaled_f64.argtypes = [u64, u64, f64, vp, i64]
        lib.synth_splitmix64.argtypes = [u64, u64]
        lib.synth_splitmix64.restype = u64
        _lib = lib
    return _lib


def splitmix64(seed: int, i: int) -> int:
    return int(_load().synth_splitmix64(seed, i))


def uniform_f64(seed: int, offset: int, shape) -> np.ndarray:
    out = np.empty(shape, dtype=np.float64)
    _load().synth_uniform_f64(seed, offset, out.ctypes.data, out.size)
    return out


def uniform_f32(seed: int, offset: int, shape) -> np.ndarray:
    out = np.empty(shape, dtype=np.float32)
    _load().synth_uniform_f32(seed, offset, out.ctypes.data, out.size)
    return out


def scaled_f64(seed: int, offset: int, phi: float, shape) -> np.ndarray:
    out = np.empty(shape, dtype=np.float64)
    _load().synth_scaled_f64(seed, offset, float(phi), out.ctypes.data, out.size)
    return out


def gemm_inputs(kind: str, M: int, N: int, K: int, seed: int, phi: float = 0.0):
    """A (M x K) and B (K x N), row-major, from one stream: A first, then B.

    kind: "f32" (uniform FP32), "f64" (uniform FP64), "f64_scaled" (scaled class).
    """
    if kind == "f32":
        return uniform_f32(seed, 0, (M, K)), uniform_f32(seed, M * K, (K, N))
    if kind == "f64":
        return uniform_f64(seed, 0, (M, K)), uniform_f64(seed, M * K, (K, N))
    if kind == "f64_scaled":
        return scaled_f64(seed, 0, phi, (M, K)), scaled_f64(seed, M * K, phi, (K, N))
    raise ValueError(kind)


# The workloads of the paper's evaluation, restated as synthetic recipes.
# Each entry: (name, kind, M, N, K, seed, phi, product counts).
WORKLOADS = {
    "fp32_n256": ("f32", 256, 256, 256, 0, 0.0, (6,)),
    **{f"fp32_n{n}": ("f32", n, n, n, n, 0.0, (6,)) for n in (1024, 2048, 4096, 8192, 16384)},
    "fp64_n4096": ("f64", 4096, 4096, 4096, 1, 0.0, (6, 10, 15, 21)),
    "fp64_scaled_phi0.5_n8192": ("f64_scaled", 8192, 8192, 8192, 3, 0.5, (21, 10)),
    "fp64_scaled_phi2_n8192": ("f64_scaled", 8192, 8192, 8192, 4, 2.0, (21, 10)),
    "fp64_scaled_phi4_n8192": ("f64_scaled", 8192, 8192, 8192, 5, 4.0, (21, 10)),
    "fp32_largek": ("f32", 2048, 2048, 65536, 2, 0.0, (6,)),
    "fp64_largek": ("f64", 2048, 2048, 65536, 2, 0.0, (6, 10, 15, 21)),
}
