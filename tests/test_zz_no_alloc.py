"""emu_gemm_f64_noalloc: the FP64-mode GEMM for callers that cannot allocate
device memory (it keeps its scratch in a static device array instead of a
caller-provided workspace).  It must give what emu_gemm_f64 gives -- FP64
mode is bit-exact, so the bar here is equality, both with that entry point
and with the oracle -- on consecutive calls that reuse the shared array,
report the same flags, and refuse problems too large for the array.

This file is collected last on purpose: it also runs after every other test
in the same process, and on its own in a fresh one."""
import ctypes

import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import device, to_dev

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 40 << 20


def _noalloc(A, B, nprod, flags):
    torch = emu._torch()
    M, K = A.shape
    N = B.shape[1]
    C = torch.full((M, N), np.nan, dtype=torch.float64, device=A.device)
    st = emu.emu_gemm_f64_noalloc(M, N, K, A.data_ptr(), A.stride(0), B.data_ptr(), B.stride(0), C.data_ptr(),
                                  C.stride(0), nprod, flags.data_ptr(), emu._stream(None))
    return st, C


def test_noalloc_matches_workspace_entry_point_twice():
    dev = device()
    torch = emu._torch()
    flags = torch.full((1,), 0xFFFF, dtype=torch.int32, device=dev)
    # two calls in a row with different shapes and data reuse the shared scratch
    for (M, N, K, seed, nprod) in [(200, 136, 300, 1, 21), (129, 257, 520, 2, 10)]:
        A, B = synth.gemm_inputs("f64", M, N, K, seed)
        Ad, Bd = to_dev(A, dev), to_dev(B, dev)
        st, C = _noalloc(Ad, Bd, nprod, flags)
        assert st == 0
        Cref, ws = emu.gemm_f64(Ad, Bd, nprod)
        assert emu.read_flags(ws) == 0
        assert int(flags.item()) == 0
        Cn = C.cpu().numpy()
        assert np.array_equal(Cn, Cref.cpu().numpy())
        C_or, f_or = oracle.gemm_f64(A, B, nprod)
        assert f_or == 0
        assert np.array_equal(Cn, C_or)


def test_noalloc_flags_equal_workspace_entry_point_on_small_slices():
    """A scaled by 2^-80: its slices 0-2 are normal BF16 values, but slices 4
    and 5 hold values below 2^-126.  With 6 products only slices 0-2 are
    formed and read, so neither entry point may flag anything, and C equals
    the oracle's bit for bit (every product unit stays a normal FP32 number)."""
    dev = device()
    torch = emu._torch()
    flags = torch.full((1,), 0xFFFF, dtype=torch.int32, device=dev)
    A, B = synth.gemm_inputs("f64", 160, 144, 520, 4)
    A = A * 2.0**-80
    assert np.all(np.abs(A[A != 0]) >= 2.0**-126)
    Ad, Bd = to_dev(A, dev), to_dev(B, dev)
    for _ in range(2):
        st, C = _noalloc(Ad, Bd, 6, flags)
        assert st == 0
        Cref, ws = emu.gemm_f64(Ad, Bd, 6)
        assert int(flags.item()) == emu.read_flags(ws) == 0
        Cn = C.cpu().numpy()
        assert np.array_equal(Cn, Cref.cpu().numpy())
        assert np.array_equal(Cn, oracle.gemm_f64(A, B, 6)[0])


def test_noalloc_limit_and_flags():
    dev = device()
    torch = emu._torch()
    flags = torch.zeros((1,), dtype=torch.int32, device=dev)
    # planes 512 + 2 * 12 * n * n plus the FP64 accumulator 8 * roundup(n, 128) * roundup(n, 256)
    # must fit 40 MiB: n = 1024 fits, 1184 does not
    def need(n):
        return 512 + 2 * 6 * n * n * 2 + 8 * ((n + 127) // 128 * 128) * ((n + 255) // 256 * 256)
    n = 1024
    assert need(n) <= SCRATCH_BYTES < need(1184)
    A, B = synth.gemm_inputs("f64", n, n, n, 3)
    Ad, Bd = to_dev(A, dev), to_dev(B, dev)
    st, C = _noalloc(Ad, Bd, 6, flags)
    assert st == 0
    Cref, _ = emu.gemm_f64(Ad, Bd, 6)
    assert np.array_equal(C.cpu().numpy(), Cref.cpu().numpy())
    Cn = C.cpu().numpy()
    for r in (0, 511, n - 1):                              # sampled rows against the oracle
        assert np.array_equal(Cn[r], oracle.gemm_f64(A, B, 6, rows=(r, r + 1))[0][0])
    big = torch.zeros((1184, 1184), dtype=torch.float64, device=dev)
    st, _ = _noalloc(big, big, 6, flags)
    assert st == 5                                       # EMU_ERR_UNSUPPORTED: beyond the static scratch
    # a domain violation is reported through flags_out
    A[5, 5] = 2.0**-130
    st, _ = _noalloc(to_dev(A[:64, :64], dev), to_dev(B[:64, :64], dev), 6, flags)
    assert st == 0 and int(flags.item()) & emu.FLAG_RANGE
