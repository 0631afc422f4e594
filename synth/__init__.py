"""Seeded synthetic inputs shaped like the paper's square GEMM sweeps.

This package holds no arithmetic of the emulation method.  It wraps the
SplitMix64 counter generator in ``synth.c`` and the input recipes used by the
tests and by ``bench.py``.  The CPU oracle and the CUDA path are both fed the
very same host arrays produced here.

Input classes (Section 7.3 of the paper, "Input Matrices and Accuracy
Metrics"): uniform random entries in [-1, 1] (the class the paper reports),
the "scaled" class ``(u - 0.5) * exp(phi * g)`` clamped into the BF16
exponent range, and a cancellation-sensitive class (the paper names it but
does not define it; see ``cancel_inputs``).  Matrix A is drawn first
(row-major), then B continues the same stream.
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


CANCEL_EXP = -20


def cancel_inputs(dtype, M: int, N: int, K: int, seed: int):
    """A cancellation-sensitive pair: A = [P | P] and B = [Q ; -Q + 2^-20 R]
    (P, Q, R uniform in [-1, 1], K even; an odd K gets one extra uniform
    column of A and row of B).  The exact product P Q - P Q + 2^-20 P R is
    about 2^-20 of |A||B|, so every dot product cancels two large halves and
    truncation and summation-order effects show up in the result."""
    K2 = K // 2
    uni = uniform_f64 if dtype == np.float64 else uniform_f32
    P = uni(seed, 0, (M, K2))
    Q = uni(seed, M * K2, (K2, N))
    R = uni(seed, M * K2 + K2 * N, (K2, N))
    A = np.concatenate([P, P], axis=1)
    B = np.concatenate([Q, (-Q + dtype(2.0 ** CANCEL_EXP) * R).astype(dtype)], axis=0)
    if K % 2:
        off = M * K2 + 2 * K2 * N
        A = np.concatenate([A, uni(seed, off, (M, 1))], axis=1)
        B = np.concatenate([B, uni(seed, off + M, (1, N))], axis=0)
    return np.ascontiguousarray(A, dtype=dtype), np.ascontiguousarray(B, dtype=dtype)


def gemm_inputs(kind: str, M: int, N: int, K: int, seed: int, phi: float = 0.0):
    """A (M x K) and B (K x N), row-major, from one stream: A first, then B.

    kind: "f32" (uniform FP32), "f64" (uniform FP64), "f64_scaled" (scaled class),
    "f32_cancel" / "f64_cancel" (cancellation-sensitive class, cancel_inputs).
    """
    if kind == "f32":
        return uniform_f32(seed, 0, (M, K)), uniform_f32(seed, M * K, (K, N))
    if kind == "f64":
        return uniform_f64(seed, 0, (M, K)), uniform_f64(seed, M * K, (K, N))
    if kind == "f64_scaled":
        return scaled_f64(seed, 0, phi, (M, K)), scaled_f64(seed, M * K, phi, (K, N))
    if kind == "f32_cancel":
        return cancel_inputs(np.float32, M, N, K, seed)
    if kind == "f64_cancel":
        return cancel_inputs(np.float64, M, N, K, seed)
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
    "fp32_cancel_n4096": ("f32_cancel", 4096, 4096, 4096, 6, 0.0, (6,)),
    "fp64_cancel_n4096": ("f64_cancel", 4096, 4096, 4096, 7, 0.0, (21, 10)),
    "fp64_largek": ("f64", 2048, 2048, 65536, 2, 0.0, (6, 10, 15, 21)),
}
