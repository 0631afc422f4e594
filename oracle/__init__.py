"""ORACLE -- test infrastructure, not part of the product.

Python access to the plain-C CPU oracle in ``oracle.c`` (a slow, literal
restatement of the paper's split, product selection and product-sum, see that
file's header).  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s
CPU-baseline / reference leg may import this package; the CUDA library never
does, and shares no code with it.

Layout conventions (row-major, dense): A planes ``[s, M, K]``, B planes
``[s, K, N]`` (the mathematical orientation), BF16 stored as uint16 bit
patterns.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import tempfile

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_SO = os.path.join(_HERE, "_oracle.so")
_lib = None

FLAG_NONFINITE = 0x1
FLAG_RANGE = 0x2
FLAG_SLICE = 0x4
ZERO_LEVEL = -(2 ** 31)
KCHUNK = 256
NPROD_TO_D = {6: 3, 10: 4, 15: 5, 21: 6}
# FP64 summation orders of the exact chunk partials (see oracle.c)
ORDER_CHUNK_OUTER = 0
ORDER_PRODUCT_OUTER = 1
ORDERS = {"chunk": ORDER_CHUNK_OUTER, "product": ORDER_PRODUCT_OUTER}


def build(force: bool = False) -> str:
    """Compile ``oracle.c`` (gcc -O2 -ffp-contract=off -fopenmp, no fast-math)."""
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_HERE)
    os.close(fd)
    cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           "-fopenmp", "-std=c11", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        i64, vp, i32, u16, f64 = ctypes.c_int64, ctypes.c_void_p, ctypes.c_int, ctypes.c_uint16, ctypes.c_double
        lib.oracle_fl_bf16.argtypes = [f64]
        lib.oracle_fl_bf16.restype = u16
        lib.oracle_bf16_value.argtypes = [u16]
        lib.oracle_bf16_value.restype = f64
        lib.oracle_ceil_log2.argtypes = [f64]
        lib.oracle_ceil_log2.restype = i32
        lib.oracle_split_f32.argtypes = [vp, i64, i64, i64, vp]
        lib.oracle_split_f32.restype = ctypes.c_uint32
        lib.oracle_split_f64.argtypes = [vp, i64, i64, i64, vp, vp]
        lib.oracle_split_f64.restype = ctypes.c_uint32
        lib.oracle_products.argtypes = [i32, i32, vp]
        lib.oracle_products.restype = i32
        lib.oracle_prodsum_f32.argtypes = [i64, i64, i64, vp, vp, i64, i64, vp]
        lib.oracle_prodsum_f64.argtypes = [i64, i64, i64, vp, vp, i32, i32, i64, i64, vp, vp]
        lib.oracle_ref_dd.argtypes = [i64, i64, i64, vp, i64, vp, i64, i64, i64, vp, vp]
        _lib = lib
    return _lib


def fl_bf16(x: float) -> int:
    """fl_BF16 of one value (Section 4.2), as a BF16 bit pattern."""
    return int(_load().oracle_fl_bf16(float(x)))


def bf16_value(bits: int) -> float:
    return float(_load().oracle_bf16_value(int(bits) & 0xFFFF))


def ceil_log2(m: float) -> int:
    return int(_load().oracle_ceil_log2(float(m)))


def bf16_to_f32(planes: np.ndarray) -> np.ndarray:
    """Exact value of BF16 bit patterns as float32 (a BF16 is the upper half of an FP32)."""
    return (planes.astype(np.uint32) << 16).view(np.float32)


def split_f32(X: np.ndarray):
    """Eq. (fp32split): returns (planes uint16 [3, rows, cols], flags)."""
    X = np.ascontiguousarray(X, dtype=np.float32)
    rows, cols = X.shape
    planes = np.empty((3, rows, cols), dtype=np.uint16)
    flags = _load().oracle_split_f32(X.ctypes.data, rows, cols, cols, planes.ctypes.data)
    return planes, int(flags)


def split_f64(X: np.ndarray):
    """Eq. (fp64split): returns (planes uint16 [6, rows, cols], v int32 [6], flags)."""
    X = np.ascontiguousarray(X, dtype=np.float64)
    rows, cols = X.shape
    planes = np.empty((6, rows, cols), dtype=np.uint16)
    v = np.empty(6, dtype=np.int32)
    flags = _load().oracle_split_f64(X.ctypes.data, rows, cols, cols, planes.ctypes.data, v.ctypes.data)
    return planes, v, int(flags)


def split_f64_rows(X: np.ndarray):
    """Eq. (fp64split) with one set of levels per row: the standard Ozaki
    scaling of Eq. (ozakiscaled) on row vectors (Section 4.3).  Each row is
    split exactly as the whole-matrix split splits a one-row matrix.  Returns
    (planes uint16 [6, rows, cols], v int32 [rows, 6], flags)."""
    X = np.ascontiguousarray(X, dtype=np.float64)
    rows, cols = X.shape
    planes = np.zeros((6, rows, cols), dtype=np.uint16)
    v = np.empty((rows, 6), dtype=np.int32)
    flags = 0
    for i in range(rows):
        p, vi, f = split_f64(X[i:i + 1])
        planes[:, i:i + 1, :] = p
        v[i] = vi
        flags |= f
    return planes, v, flags


def gemm_f64_rowcol(A: np.ndarray, B: np.ndarray, nprod: int, rows=None):
    """Algorithm 2 with per-row levels for A and per-column levels for B: the
    slices of A are split row by row, those of B column by column (rows of
    B^T), and the product-sum is Algorithm 2's product-outer sum.  Returns
    (C, flags)."""
    Ap, _, fa = split_f64_rows(A)
    Bt, _, fb = split_f64_rows(np.ascontiguousarray(B.T))
    Bp = np.ascontiguousarray(Bt.transpose(0, 2, 1))
    if rows is not None:
        Ap = Ap[:, rows[0]:rows[1]]
    return prodsum_f64(Ap, Bp, nprod), fa | fb


def products(mode: int, nprod: int):
    """Executed (i, j) order: FP32 reuse chain, or FP64 diagonal order."""
    buf = np.zeros(2 * 21, dtype=np.int32)
    n = _load().oracle_products(mode, nprod, buf.ctypes.data)
    if n < 0:
        raise ValueError(f"no product set for mode={mode} nprod={nprod}")
    return [(int(buf[2 * q]), int(buf[2 * q + 1])) for q in range(n)]


def prodsum_f32(Ap: np.ndarray, Bp: np.ndarray, rows=None) -> np.ndarray:
    """FP32-mode product-sum of A planes [3,M,K] and B planes [3,K,N], rows [r0, r1)."""
    Ap = np.ascontiguousarray(Ap, dtype=np.uint16)
    Bp = np.ascontiguousarray(Bp, dtype=np.uint16)
    _, M, K = Ap.shape
    N = Bp.shape[2]
    r0, r1 = (0, M) if rows is None else rows
    C = np.empty((r1 - r0, N), dtype=np.float32)
    _load().oracle_prodsum_f32(M, N, K, Ap.ctypes.data, Bp.ctypes.data, r0, r1 - r0, C.ctypes.data)
    return C


def prodsum_f64(Ap: np.ndarray, Bp: np.ndarray, nprod: int, rows=None, check_exact: bool = False,
                order: str = "product"):
    """FP64-mode product-sum (Eq. (fp64reconstruction)); order "product"
    (Algorithm 2 as written, chunk partials summed exactly per product) or
    "chunk" (chunk outer, every partial added in FP64).  Optionally counts
    inexact FP32 partials."""
    Ap = np.ascontiguousarray(Ap, dtype=np.uint16)
    Bp = np.ascontiguousarray(Bp, dtype=np.uint16)
    _, M, K = Ap.shape
    N = Bp.shape[2]
    r0, r1 = (0, M) if rows is None else rows
    C = np.empty((r1 - r0, N), dtype=np.float64)
    bad = ctypes.c_int64(-1)
    _load().oracle_prodsum_f64(M, N, K, Ap.ctypes.data, Bp.ctypes.data, int(nprod), ORDERS[order], r0, r1 - r0,
                               C.ctypes.data, ctypes.byref(bad) if check_exact else None)
    return (C, int(bad.value)) if check_exact else C


def gemm_f32(A: np.ndarray, B: np.ndarray, rows=None):
    """Algorithm 1 end to end: split A (rows needed) and B, then the product-sum."""
    r0, r1 = (0, A.shape[0]) if rows is None else rows
    Ap, fa = split_f32(A[r0:r1])
    Bp, fb = split_f32(B)
    return prodsum_f32(Ap, Bp), fa | fb


def gemm_f64(A: np.ndarray, B: np.ndarray, nprod: int, rows=None, order: str = "product"):
    """Algorithm 2 end to end (the split of A is global, so A is split whole)."""
    Ap, _, fa = split_f64(A)
    Bp, _, fb = split_f64(B)
    return prodsum_f64(Ap, Bp, nprod, rows=rows, order=order), fa | fb


def tail_products(nprod: int, merge_from: int):
    """Products (i, j) with merge_from <= i + j < d, in Algorithm 2's diagonal
    order (the tail that the merged variant accumulates in one FP32 sum)."""
    d = NPROD_TO_D[nprod]
    return [(i, l - i) for l in range(merge_from, d) for i in range(l + 1)]


def _slice_ints(planes: np.ndarray, v: np.ndarray, r: int):
    """Slice r as exact integers n with value n * 2^(v[r] - 8) (Eq. (fp64split):
    every slice entry is a multiple of 2^(v - 8) of magnitude <= 2^v), and that
    exponent; (None, None) for an all-zero level."""
    if int(v[r]) == ZERO_LEVEL:
        return None, None
    e = int(v[r]) - 8
    vals = np.ldexp(bf16_to_f32(planes[r]).astype(np.float64), -e)
    n = vals.astype(np.int64)
    assert np.array_equal(n.astype(np.float64), vals), "slice entry not a multiple of 2^(v-8)"
    return n, e


def gemm_f64_merged(A: np.ndarray, B: np.ndarray, nprod: int, merge_from: int, rows=None):
    """FP64 mode with merged tail diagonals (an extension, not in the paper).

    The products with i + j < merge_from are summed as in Algorithm 2 (product
    outer, diagonal order, one FP64 addition each); the remaining products of
    S_d (merge_from <= i + j < d) form one tail T = sum of A_i B_j that is added
    once, last: C = fl64(C_head + T).  The GPU accumulates T in FP32 on the
    tensor cores (order unspecified); here T is the EXACT sum, computed in
    integers (slice entries are integer multiples of 2^(v - 8)), and rounded
    once to FP64 only if it needs more than 53 bits.  Returns (C, T, S, flags)
    with S = sum over the tail of |A_i| |B_j| (the scale of the FP32
    accumulation error bound)."""
    d = NPROD_TO_D[nprod]
    if not 1 <= merge_from <= d:
        raise ValueError("merge_from must lie in 1 .. d")
    Ap, va, fa = split_f64(A)
    Bp, vb, fb = split_f64(B)
    r0, r1 = (0, A.shape[0]) if rows is None else rows
    n_head = merge_from * (merge_from + 1) // 2
    C = prodsum_f64(Ap, Bp, n_head, rows=(r0, r1))
    N = B.shape[1]
    terms = []
    for i, j in tail_products(nprod, merge_from):
        na, ea = _slice_ints(Ap[:, r0:r1], va, i)
        nb, eb = _slice_ints(Bp, vb, j)
        if na is None or nb is None:
            continue
        terms.append((na @ nb, ea + eb))          # exact: |entries| <= K * 2^16
    T = np.zeros((r1 - r0, N), dtype=np.float64)
    S = np.zeros((r1 - r0, N), dtype=np.float64)
    if terms:
        e_min = min(e for _, e in terms)
        tot = np.zeros((r1 - r0, N), dtype=object)
        for prod, e in terms:
            tot = tot + prod.astype(object) * (1 << (e - e_min))
        T = np.array([[float(x) for x in row] for row in tot], dtype=np.float64).reshape(r1 - r0, N)
        T = np.ldexp(T, e_min)
        for i, j in tail_products(nprod, merge_from):
            S += np.abs(bf16_to_f32(Ap[i, r0:r1]).astype(np.float64)) @ np.abs(bf16_to_f32(Bp[j]).astype(np.float64))
    return C + T, T, S, fa | fb


def gemm_ex(opA: int, opB: int, alpha, A: np.ndarray, B: np.ndarray, beta, C: np.ndarray | None = None,
            nprod: int | None = None):
    """General GEMM C <- alpha op(A) op(B) + beta C (the BLAS semantics that
    Section 9 leaves as future work), row-major, op = 1 transposes the stored
    matrix.  P = op(A) op(B) is Algorithm 1 (FP32 inputs) or Algorithm 2 with
    nprod products (FP64 inputs); the epilogue rounds each operation once in
    the input format: alpha = 1, beta = 0 gives P; beta = 0 gives alpha * P
    (C not read); otherwise (alpha * P) + (beta * C).  Returns (C, flags)."""
    f64 = A.dtype == np.float64
    dt = np.float64 if f64 else np.float32
    Ae = np.ascontiguousarray(A.T if opA else A)
    Be = np.ascontiguousarray(B.T if opB else B)
    M, K = Ae.shape
    N = Be.shape[1]
    if K == 0:
        P, flags = np.zeros((M, N), dtype=dt), 0
    elif f64:
        P, flags = gemm_f64(Ae, Be, nprod)
    else:
        P, flags = gemm_f32(Ae, Be)
    a, b = dt(alpha), dt(beta)
    if a == 1 and b == 0:
        return P, flags
    aP = a * P                                   # one rounding in the input format
    if b == 0:
        return aP, flags
    return aP + b * np.asarray(C, dtype=dt), flags


def ref_dd(A: np.ndarray, B: np.ndarray, rows=None):
    """Double-double reference A.B (rows [r0, r1)): returns (hi, lo)."""
    A = np.ascontiguousarray(A, dtype=np.float64)
    B = np.ascontiguousarray(B, dtype=np.float64)
    M, K = A.shape
    N = B.shape[1]
    r0, r1 = (0, M) if rows is None else rows
    hi = np.empty((r1 - r0, N), dtype=np.float64)
    lo = np.empty((r1 - r0, N), dtype=np.float64)
    _load().oracle_ref_dd(M, N, K, A.ctypes.data, K, B.ctypes.data, N, r0, r1 - r0,
                          hi.ctypes.data, lo.ctypes.data)
    return hi, lo


def errors(C_hat: np.ndarray, hi: np.ndarray, lo: np.ndarray, absAB: np.ndarray | None = None):
    """Accuracy metrics of Section 7.3 against a double-double reference.

    e_F (Eq. (froerror)), e_max = max |C_hat - C_ref|, and, when |A||B| is
    given, e_scaled (Eq. (scalederror)) over entries with a nonzero
    denominator (entries with a zero denominator are reported as absolute
    error in ``e_abs_zero_den``).
    """
    d = (C_hat.astype(np.float64) - hi) - lo
    out = {
        "e_F": float(np.sqrt(np.sum(d * d)) / max(np.sqrt(np.sum(hi * hi)), np.finfo(float).tiny)),
        "e_max": float(np.max(np.abs(d))) if d.size else 0.0,
    }
    if absAB is not None:
        nz = absAB != 0
        out["e_scaled"] = float(np.max(np.abs(d[nz]) / absAB[nz])) if np.any(nz) else 0.0
        out["e_abs_zero_den"] = float(np.max(np.abs(d[~nz]))) if np.any(~nz) else 0.0
    return out
