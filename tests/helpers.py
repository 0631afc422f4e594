"""Shared helpers of the GPU parity tests (inputs, device transfer, bounds)."""
import numpy as np
import pytest

import paper_2609_04663_gb300 as emu


def device():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU tests need a CUDA device; the library has no CPU path")
    emu._build.build()
    emu.load()
    return torch.device("cuda:0")


def to_dev(a, dev, ld_pad: int = 0):
    """Copy a 2-D host array to the device; ld_pad > 0 gives it a wider row pitch."""
    import torch
    a = np.ascontiguousarray(a)
    if ld_pad:
        big = np.zeros((a.shape[0], a.shape[1] + ld_pad), dtype=a.dtype)
        big[:, : a.shape[1]] = a
        return torch.from_numpy(big).to(dev)[:, : a.shape[1]]
    return torch.from_numpy(a).to(dev)


def planes_np(t):
    return t.cpu().numpy().view(np.uint16)


def abs_ab(A, B):
    """(|A||B|) in FP64, the GEMM-scaled denominator of Eq. (scalederror)."""
    return np.abs(A.astype(np.float64)) @ np.abs(B.astype(np.float64))


def fp32_within_tolerance(C_gpu, C_or, A, B):
    """The FP32-mode bar: |C - C_oracle| <= 1e-5 (|A||B|) elementwise."""
    bound = 1e-5 * abs_ab(A, B)
    err = np.abs(C_gpu.astype(np.float64) - C_or.astype(np.float64))
    return bool(np.all(err <= bound)), float(np.max(err / np.maximum(bound, 1e-300)))


def random_finite_f32(shape, seed, emax_field=253):
    """Random FP32 bit patterns: zeros, subnormals and normals up to 2^(emax_field-126)."""
    rng = np.random.default_rng(seed)
    n = int(np.prod(shape))
    mant = rng.integers(0, 2**23, size=n, dtype=np.uint32)
    exp = rng.integers(0, emax_field + 1, size=n).astype(np.uint32)
    sign = rng.integers(0, 2, size=n).astype(np.uint32)
    x = ((sign << 31) | (exp << 23) | mant).view(np.float32)
    x[rng.random(n) < 0.02] = 0.0
    return x.reshape(shape)


def sample_rows(M, count, seed):
    rng = np.random.default_rng(seed)
    rows = sorted(set(int(r) for r in rng.integers(0, M, size=count)) | {0, M - 1})
    return rows


def gemm_f32_one_accumulator(A_d, B_d):
    """FP32 mode as split + product-sum through the separate C-ABI calls: all
    of K in one FP32 accumulator per tile.  emu_gemm_f32 itself may split K
    in two for small results, which changes FP32 rounding; the kernels that
    must match the one-accumulator sum bit for bit are compared with this.
    Returns (C, the splits' flag words or-ed)."""
    M, K = A_d.shape
    N = B_d.shape[1]
    Ap, wa = emu.split_f32(A_d, ldcomp=emu.gemm_ldk(K))
    Bp, wb = emu.split_f32(B_d, transpose=True, ldcomp=emu.gemm_ldk(K))
    C, _ = emu.prodsum_f32(Ap, Bp, M, N, K)
    return C, emu.read_flags(wa) | emu.read_flags(wb)
