"""GB300-native BF16 component-product GEMM emulation (arXiv 2609.04663).

Thin ctypes binding over the C-ABI of ``include/emu.h`` (library
``_emu.so`` built in-tree by ``_build.py``).  The functions named ``emu_*``
take plain integers (device pointers, sizes, the raw CUDA stream handle) and
return the ``emu_status`` code, exactly as the C entry points do.  The
tensor-level helpers below them only allocate device memory with PyTorch and
marshal pointers: every step of the method runs in the CUDA kernels.

There is no CPU fallback: importing this package without the compiled
library raises.
"""
from __future__ import annotations

import ctypes
import os

from . import _build

_lib = None

EMU_OK = 0
STATUS = {0: "ok", 1: "invalid argument", 2: "misaligned", 3: "workspace too small", 4: "CUDA error",
          5: "unsupported size"}
FLAG_NONFINITE, FLAG_RANGE, FLAG_SLICE, FLAG_TIMEOUT = 0x1, 0x2, 0x4, 0x8
OP_N, OP_T = 0, 1
ZERO_LEVEL = -(2 ** 31)

_SIGS = {
    # name: (restype, argtypes)
    "emu_split_workspace_bytes": ("size", ["i"]),
    "emu_split_f32": ("i", ["p", "l", "l", "l", "i", "p", "l", "p", "size", "p"]),
    "emu_split_f64": ("i", ["p", "l", "l", "l", "i", "p", "l", "p", "p", "size", "p"]),
    "emu_split_f64_slices": ("i", ["p", "l", "l", "l", "i", "p", "l", "i", "p", "p", "size", "p"]),
    "emu_gemm_workspace_bytes": ("size", ["i", "l", "l", "l"]),
    "emu_split_f32_pair": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "p", "l", "p", "size", "p"]),
    "emu_split_f64_pair": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "p", "l", "i", "p", "p", "p", "size", "p"]),
    "emu_gemm_f32": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "l", "p", "size", "p"]),
    "emu_gemm_f64": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "l", "i", "p", "size", "p"]),
    "emu_gemm_f32_fused": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "l", "p", "size", "p"]),
    "emu_gemm_f64_merged_workspace_bytes": ("size", ["l", "l", "l"]),
    "emu_gemm_f64_merged": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "l", "i", "i", "p", "size", "p"]),
    "emu_prodsum_f32": ("i", ["l", "l", "l", "p", "p", "l", "p", "l", "p", "size", "p"]),
    "emu_prodsum_f64": ("i", ["l", "l", "l", "p", "p", "l", "p", "p", "i", "p", "l", "p", "size", "p"]),
    "emu_gemm_f64_noalloc": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "l", "i", "p", "p"]),
    "emu_gemm_host_workspace_bytes": ("size", ["i", "l", "l", "l"]),
    "emu_gemm_ex_workspace_bytes": ("size", ["i", "l", "l", "l"]),
    "emu_prodsum_workspace_bytes": ("size", ["i", "l", "l"]),
    "emu_prodsum_f64_tile_columns": ("i", ["l", "l"]),
    "emu_prodsum_f64_tile_rows": ("i", ["l", "l"]),
    "emu_prodsum_f64_launches": ("i", ["l", "l"]),
    "emu_prodsum_f32_launches": ("i", ["l", "l"]),
    "emu_prodsum_f32_tile_columns": ("i", ["l", "l"]),
    "emu_prodsum_f32_tile_rows": ("i", ["l", "l"]),
    "emu_split_f64_rowcol_workspace_bytes": ("size", ["l"]),
    "emu_split_f64_rowcol": ("i", ["p", "l", "l", "l", "i", "p", "l", "p", "p", "size", "p"]),
    "emu_gemm_f64_rowcol_workspace_bytes": ("size", ["l", "l", "l"]),
    "emu_gemm_f64_rowcol": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "l", "i", "p", "size", "p"]),
    "emu_gemm_ex_f32": ("i", ["i", "i", "l", "l", "l", "f", "p", "l", "p", "l", "f", "p", "l", "p", "size", "p"]),
    "emu_gemm_ex_f64": ("i", ["i", "i", "l", "l", "l", "d", "p", "l", "p", "l", "d", "p", "l", "i", "p", "size", "p"]),
    "emu_gemm_f32_host": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "l", "p", "size", "p"]),
    "emu_gemm_f64_host": ("i", ["l", "l", "l", "p", "l", "p", "l", "p", "l", "i", "p", "size", "p"]),
    "emu_read_flags": ("i", ["p", "p", "p"]),
    "emu_selftest_timeout": ("i", ["p", "size", "u32", "p"]),
    "emu_status_string": ("str", ["i"]),
}
_CT = {"i": ctypes.c_int, "l": ctypes.c_int64, "p": ctypes.c_void_p, "size": ctypes.c_size_t,
       "u32": ctypes.c_uint32, "str": ctypes.c_char_p, "f": ctypes.c_float, "d": ctypes.c_double}


class EmuError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {STATUS.get(status, status)} (status {status})")
        self.status = status


def library_path() -> str:
    return _build.SO


def load():
    """Load ``_emu.so`` (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_build.SO):
            raise ImportError(f"CUDA emulation library not built: {_build.SO} is missing "
                              "(run paper_2609_04663_gb300._build.build())")
        lib = ctypes.CDLL(_build.SO)
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype = _CT[res]
            fn.argtypes = [_CT[a] for a in args]
        _lib = lib
    return _lib


def _mk(name):
    def f(*args):
        return getattr(load(), name)(*args)
    f.__name__ = name
    f.__doc__ = f"C-ABI ``{name}`` (include/emu.h); returns its result unchanged."
    return f


emu_split_workspace_bytes = _mk("emu_split_workspace_bytes")
emu_split_f32 = _mk("emu_split_f32")
emu_split_f64 = _mk("emu_split_f64")
emu_split_f64_slices = _mk("emu_split_f64_slices")
emu_gemm_workspace_bytes = _mk("emu_gemm_workspace_bytes")
emu_split_f32_pair = _mk("emu_split_f32_pair")
emu_split_f64_pair = _mk("emu_split_f64_pair")
emu_gemm_f32 = _mk("emu_gemm_f32")
emu_gemm_f64 = _mk("emu_gemm_f64")
emu_gemm_f32_fused = _mk("emu_gemm_f32_fused")
emu_gemm_f64_merged_workspace_bytes = _mk("emu_gemm_f64_merged_workspace_bytes")
emu_gemm_f64_merged = _mk("emu_gemm_f64_merged")
emu_prodsum_f32 = _mk("emu_prodsum_f32")
emu_prodsum_f64 = _mk("emu_prodsum_f64")
emu_gemm_f64_noalloc = _mk("emu_gemm_f64_noalloc")
emu_gemm_host_workspace_bytes = _mk("emu_gemm_host_workspace_bytes")
emu_gemm_ex_workspace_bytes = _mk("emu_gemm_ex_workspace_bytes")
emu_prodsum_workspace_bytes = _mk("emu_prodsum_workspace_bytes")
emu_prodsum_f64_tile_columns = _mk("emu_prodsum_f64_tile_columns")
emu_prodsum_f64_tile_rows = _mk("emu_prodsum_f64_tile_rows")
emu_prodsum_f64_launches = _mk("emu_prodsum_f64_launches")
emu_prodsum_f32_launches = _mk("emu_prodsum_f32_launches")
emu_prodsum_f32_tile_columns = _mk("emu_prodsum_f32_tile_columns")
emu_prodsum_f32_tile_rows = _mk("emu_prodsum_f32_tile_rows")
emu_split_f64_rowcol_workspace_bytes = _mk("emu_split_f64_rowcol_workspace_bytes")
emu_split_f64_rowcol = _mk("emu_split_f64_rowcol")
emu_gemm_f64_rowcol_workspace_bytes = _mk("emu_gemm_f64_rowcol_workspace_bytes")
emu_gemm_f64_rowcol = _mk("emu_gemm_f64_rowcol")
emu_gemm_ex_f32 = _mk("emu_gemm_ex_f32")
emu_gemm_ex_f64 = _mk("emu_gemm_ex_f64")
emu_gemm_f32_host = _mk("emu_gemm_f32_host")
emu_gemm_f64_host = _mk("emu_gemm_f64_host")
emu_read_flags = _mk("emu_read_flags")
emu_selftest_timeout = _mk("emu_selftest_timeout")
emu_status_string = _mk("emu_status_string")


# ------------------------------------------------------------ tensor helpers
def _torch():
    import torch
    return torch


def _stream(stream):
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream if hasattr(s, "cuda_stream") else int(s)


def _check(status, where):
    if status != EMU_OK:
        raise EmuError(status, where)


def workspace(nbytes: int, device="cuda"):
    """A device workspace (uint8 tensor) of at least nbytes, 256-byte aligned by the allocator."""
    torch = _torch()
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device)


def read_flags(ws, stream=None) -> int:
    out = ctypes.c_uint32(0)
    _check(emu_read_flags(ws.data_ptr(), ctypes.addressof(out), _stream(stream)), "emu_read_flags")
    return int(out.value)


def gemm_ldk(K: int) -> int:
    """Leading dimension of the K-major planes inside a GEMM workspace."""
    return (max(K, 1) + 7) // 8 * 8


def split_f32(X, transpose: bool = False, ldcomp: int | None = None, ws=None, stream=None):
    """Eq. (fp32split) on the GPU: returns (planes int16 [3, rows_out, ldcomp], ws)."""
    torch = _torch()
    rows, cols = X.shape
    rows_out, cols_out = (cols, rows) if transpose else (rows, cols)
    ldcomp = ldcomp or cols_out
    planes = torch.zeros((3, rows_out, ldcomp), dtype=torch.int16, device=X.device)
    ws = ws if ws is not None else workspace(emu_split_workspace_bytes(32), X.device)
    _check(emu_split_f32(X.data_ptr(), rows, cols, X.stride(0), int(transpose), planes.data_ptr(), ldcomp,
                         ws.data_ptr(), ws.numel(), _stream(stream)), "emu_split_f32")
    return planes, ws


def split_f64(X, transpose: bool = False, ldcomp: int | None = None, ws=None, stream=None, nslices: int = 6):
    """Eq. (fp64split) on the GPU: returns (planes int16 [6, rows_out, ldcomp], v int32[6] (device), ws).
    nslices < 6 calls emu_split_f64_slices (planes and levels from nslices on unspecified)."""
    torch = _torch()
    rows, cols = X.shape
    rows_out, cols_out = (cols, rows) if transpose else (rows, cols)
    ldcomp = ldcomp or cols_out
    planes = torch.zeros((6, rows_out, ldcomp), dtype=torch.int16, device=X.device)
    v = torch.empty(6, dtype=torch.int32, device=X.device)
    ws = ws if ws is not None else workspace(emu_split_workspace_bytes(64), X.device)
    if nslices == 6:
        _check(emu_split_f64(X.data_ptr(), rows, cols, X.stride(0), int(transpose), planes.data_ptr(), ldcomp,
                             v.data_ptr(), ws.data_ptr(), ws.numel(), _stream(stream)), "emu_split_f64")
    else:
        _check(emu_split_f64_slices(X.data_ptr(), rows, cols, X.stride(0), int(transpose), planes.data_ptr(), ldcomp,
                                    int(nslices), v.data_ptr(), ws.data_ptr(), ws.numel(), _stream(stream)),
               "emu_split_f64_slices")
    return planes, v, ws


def split_f64_rowcol(X, transpose: bool = False, ldcomp: int | None = None, ws=None, stream=None):
    """emu_split_f64_rowcol: levels per row of X (per column when transposed).
    Returns (planes int16 [6, plane_rows, ldcomp], v int32 [6, plane_rows] (device), ws)."""
    torch = _torch()
    rows, cols = X.shape
    prow, pcols = (cols, rows) if transpose else (rows, cols)
    ldcomp = ldcomp or pcols
    planes = torch.zeros((6, prow, ldcomp), dtype=torch.int16, device=X.device)
    v = torch.empty((6, prow), dtype=torch.int32, device=X.device)
    ws = ws if ws is not None else workspace(emu_split_f64_rowcol_workspace_bytes(prow), X.device)
    _check(emu_split_f64_rowcol(X.data_ptr(), rows, cols, X.stride(0), int(transpose), planes.data_ptr(), ldcomp,
                                v.data_ptr(), ws.data_ptr(), ws.numel(), _stream(stream)), "emu_split_f64_rowcol")
    return planes, v, ws


def gemm_f64_rowcol(A, B, nprod: int, C=None, ws=None, stream=None):
    """emu_gemm_f64_rowcol: Algorithm 2 with levels per row of A and per column of B."""
    torch = _torch()
    M, K = A.shape
    N = B.shape[1]
    C = C if C is not None else torch.empty((M, N), dtype=torch.float64, device=A.device)
    ws = ws if ws is not None else workspace(emu_gemm_f64_rowcol_workspace_bytes(M, N, K), A.device)
    _check(emu_gemm_f64_rowcol(M, N, K, A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0), C.data_ptr(),
                               C.stride(0), int(nprod), ws.data_ptr(), ws.numel(), _stream(stream)),
           "emu_gemm_f64_rowcol")
    return C, ws


def gemm_f32(A, B, C=None, ws=None, stream=None):
    """Algorithm 1 on the GPU: C = A.B for FP32 row-major A (M x K), B (K x N)."""
    torch = _torch()
    M, K = A.shape
    N = B.shape[1]
    C = C if C is not None else torch.empty((M, N), dtype=torch.float32, device=A.device)
    ws = ws if ws is not None else workspace(emu_gemm_workspace_bytes(32, M, N, K), A.device)
    _check(emu_gemm_f32(M, N, K, A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0), C.data_ptr(), C.stride(0),
                        ws.data_ptr(), ws.numel(), _stream(stream)), "emu_gemm_f32")
    return C, ws


def gemm_f32_fused(A, B, C=None, ws=None, stream=None):
    """emu_gemm_f32_fused: Algorithm 1 with the split inside the product-sum
    (no planes in memory); C bit-identical to gemm_f32."""
    torch = _torch()
    M, K = A.shape
    N = B.shape[1]
    C = C if C is not None else torch.empty((M, N), dtype=torch.float32, device=A.device)
    ws = ws if ws is not None else workspace(emu_split_workspace_bytes(32), A.device)
    _check(emu_gemm_f32_fused(M, N, K, A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0), C.data_ptr(),
                              C.stride(0), ws.data_ptr(), ws.numel(), _stream(stream)), "emu_gemm_f32_fused")
    return C, ws


def gemm_f64(A, B, nprod: int, C=None, ws=None, stream=None):
    """Algorithm 2 on the GPU: C = A.B for FP64 A, B with nprod in {6, 10, 15, 21}."""
    torch = _torch()
    M, K = A.shape
    N = B.shape[1]
    C = C if C is not None else torch.empty((M, N), dtype=torch.float64, device=A.device)
    ws = ws if ws is not None else workspace(emu_gemm_workspace_bytes(64, M, N, K), A.device)
    _check(emu_gemm_f64(M, N, K, A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0), C.data_ptr(), C.stride(0),
                        int(nprod), ws.data_ptr(), ws.numel(), _stream(stream)), "emu_gemm_f64")
    return C, ws


def gemm_f64_merged(A, B, nprod: int, merge_from: int, C=None, ws=None, stream=None):
    """emu_gemm_f64_merged: Algorithm 2's head (i + j < merge_from) plus the
    remaining products of S_d accumulated in one FP32 tail, added last."""
    torch = _torch()
    M, K = A.shape
    N = B.shape[1]
    C = C if C is not None else torch.empty((M, N), dtype=torch.float64, device=A.device)
    ws = ws if ws is not None else workspace(emu_gemm_f64_merged_workspace_bytes(M, N, K), A.device)
    _check(emu_gemm_f64_merged(M, N, K, A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0), C.data_ptr(),
                               C.stride(0), int(nprod), int(merge_from), ws.data_ptr(), ws.numel(), _stream(stream)),
           "emu_gemm_f64_merged")
    return C, ws


def gemm_ex(A, B, opA: int = OP_N, opB: int = OP_N, alpha: float = 1.0, beta: float = 0.0, C=None,
            nprod: int | None = None, ws=None, stream=None):
    """emu_gemm_ex_*: C <- alpha op(A) op(B) + beta C for device tensors A, B
    as stored (op = OP_T reads the stored matrix transposed).  FP32 tensors
    run Algorithm 1, FP64 tensors Algorithm 2 with nprod products."""
    torch = _torch()
    M, K = (A.shape[1], A.shape[0]) if opA == OP_T else (A.shape[0], A.shape[1])
    N = B.shape[0] if opB == OP_T else B.shape[1]
    f64 = A.dtype == torch.float64
    C = C if C is not None else torch.zeros((M, N), dtype=A.dtype, device=A.device)
    ws = ws if ws is not None else workspace(emu_gemm_ex_workspace_bytes(64 if f64 else 32, M, N, K), A.device)
    if f64:
        r = emu_gemm_ex_f64(opA, opB, M, N, K, float(alpha), A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0),
                            float(beta), C.data_ptr(), C.stride(0), int(nprod), ws.data_ptr(), ws.numel(),
                            _stream(stream))
    else:
        r = emu_gemm_ex_f32(opA, opB, M, N, K, float(alpha), A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0),
                            float(beta), C.data_ptr(), C.stride(0), ws.data_ptr(), ws.numel(), _stream(stream))
    _check(r, "emu_gemm_ex_f64" if f64 else "emu_gemm_ex_f32")
    return C, ws


def gemm_host(A, B, nprod: int | None = None, C=None, ws=None, stream=None, device="cuda"):
    """emu_gemm_f32_host / emu_gemm_f64_host: C = A.B with A, B, C in host
    memory (CPU tensors; pinned ones give asynchronous full-speed copies).
    FP32 inputs run Algorithm 1, FP64 inputs Algorithm 2 with nprod products.
    Returns (C, ws) after enqueueing; synchronise the stream before reading C."""
    torch = _torch()
    M, K = A.shape
    N = B.shape[1]
    f64 = A.dtype == torch.float64
    C = C if C is not None else torch.empty((M, N), dtype=A.dtype, pin_memory=True)
    mode = 64 if f64 else 32
    ws = ws if ws is not None else workspace(emu_gemm_host_workspace_bytes(mode, M, N, K), device)
    if f64:
        r = emu_gemm_f64_host(M, N, K, A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0), C.data_ptr(),
                              C.stride(0), int(nprod), ws.data_ptr(), ws.numel(), _stream(stream))
    else:
        r = emu_gemm_f32_host(M, N, K, A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0), C.data_ptr(),
                              C.stride(0), ws.data_ptr(), ws.numel(), _stream(stream))
    _check(r, "emu_gemm_f64_host" if f64 else "emu_gemm_f32_host")
    return C, ws


def prodsum_f32(Ap, Bp, M: int, N: int, K: int, C=None, ws=None, stream=None):
    """Product-sum alone from planes Ap [3, M, ldcomp], Bp [3, N, ldcomp] (K-major)."""
    torch = _torch()
    C = C if C is not None else torch.empty((M, N), dtype=torch.float32, device=Ap.device)
    ws = ws if ws is not None else workspace(emu_split_workspace_bytes(32), Ap.device)
    _check(emu_prodsum_f32(M, N, K, Ap.data_ptr(), Bp.data_ptr(), Ap.shape[2], C.data_ptr(), C.stride(0),
                           ws.data_ptr(), ws.numel(), _stream(stream)), "emu_prodsum_f32")
    return C, ws


def prodsum_f64(Ap, Bp, M: int, N: int, K: int, nprod: int, vA=None, vB=None, C=None, ws=None, stream=None):
    """FP64-mode product-sum alone from planes Ap [6, M, ldcomp], Bp [6, N, ldcomp];
    vA, vB: the level exponents emu_split_f64 returned for A and B (or None)."""
    torch = _torch()
    C = C if C is not None else torch.empty((M, N), dtype=torch.float64, device=Ap.device)
    ws = ws if ws is not None else workspace(emu_prodsum_workspace_bytes(64, M, N), Ap.device)
    _check(emu_prodsum_f64(M, N, K, Ap.data_ptr(), Bp.data_ptr(), Ap.shape[2],
                           vA.data_ptr() if vA is not None else None, vB.data_ptr() if vB is not None else None,
                           int(nprod), C.data_ptr(), C.stride(0), ws.data_ptr(), ws.numel(), _stream(stream)),
           "emu_prodsum_f64")
    return C, ws
