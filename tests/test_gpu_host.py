"""GEMM from host buffers (emu_gemm_f32_host / emu_gemm_f64_host) through the
C-ABI.  The host entry points pipeline copies, splits and product-sums over
panels; they run the same kernels in the same per-tile order as the
device-buffer GEMMs, so their results must be bit-identical to those (which
the other GPU tests hold to the oracle) and, in FP64 mode, to the oracle
itself.  Sizes are chosen so that row panels, K-panels and both ring slots
are reused and the last panel of each kind is ragged."""
import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import device, fp32_within_tolerance, gemm_f32_one_accumulator, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def host(a, pinned=True, ld_pad=0):
    """A host tensor holding a, optionally with a wider row pitch."""
    torch = emu._torch()
    a = np.ascontiguousarray(a)
    big = torch.zeros((a.shape[0], a.shape[1] + ld_pad), dtype=torch.from_numpy(a).dtype, pin_memory=pinned)
    big[:, : a.shape[1]] = torch.from_numpy(a)
    return big[:, : a.shape[1]]


def run_host(A, B, nprod=None, pinned=True, pads=(0, 0, 0)):
    torch = emu._torch()
    M, K = A.shape
    N = B.shape[1]
    Ah, Bh = host(A, pinned, pads[0]), host(B, pinned, pads[1])
    Ch = host(np.full((M, N), np.nan, dtype=A.dtype), pinned, pads[2])
    C, ws = emu.gemm_host(Ah, Bh, nprod=nprod, C=Ch)
    torch.cuda.synchronize()
    return C.numpy().copy(), emu.read_flags(ws)


@pytest.mark.parametrize("M,N,K,seed", [
    (300, 200, 700, 21),     # 3 row panels, 1 column panel, ragged
    (2048, 384, 2048, 22),   # 8 row panels, 2 column panels: both rings reused
    (1100, 2300, 520, 25),   # 5 row panels, 5 column panels, ragged edges
    (1, 1, 1, 23),
    (129, 257, 33, 24),
])
def test_gemm_f32_host_equals_device_path(dev, M, N, K, seed):
    A, B = synth.gemm_inputs("f32", M, N, K, seed)
    Ch, flags = run_host(A, B, pads=(3, 5, 7))
    assert flags == 0
    Cd, _ = gemm_f32_one_accumulator(to_dev(A, dev), to_dev(B, dev))
    np.testing.assert_array_equal(Ch.view(np.uint32), Cd.cpu().numpy().view(np.uint32))
    if M * N * K <= 300 * 200 * 700:
        Co, _ = oracle.gemm_f32(A, B)
        ok, worst = fp32_within_tolerance(Ch, Co, A, B)
        assert ok, worst


@pytest.mark.parametrize("M,N,K,nprod,seed", [
    (300, 200, 700, 21, 31),
    (1100, 260, 520, 10, 32),   # 8 row panels of 256 (last one 76 rows)
    (5, 3, 1, 6, 33),
])
def test_gemm_f64_host_equals_oracle(dev, M, N, K, nprod, seed):
    A, B = synth.gemm_inputs("f64", M, N, K, seed)
    Ch, flags = run_host(A, B, nprod=nprod, pads=(1, 2, 3))
    assert flags == 0
    Cd, _ = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
    np.testing.assert_array_equal(Ch.view(np.uint64), Cd.cpu().numpy().view(np.uint64))
    if M <= 300:
        Co, _ = oracle.gemm_f64(A, B, nprod)
        np.testing.assert_array_equal(Ch.view(np.uint64), Co.view(np.uint64))


def test_host_pageable_buffers(dev):
    A, B = synth.gemm_inputs("f32", 200, 100, 300, 41)
    Ch, flags = run_host(A, B, pinned=False)
    Cd, _ = gemm_f32_one_accumulator(to_dev(A, dev), to_dev(B, dev))
    np.testing.assert_array_equal(Ch.view(np.uint32), Cd.cpu().numpy().view(np.uint32))


@pytest.mark.parametrize("kind", ["f32", "f64"])
def test_host_k_zero_writes_zeros_and_empty_is_noop(dev, kind):
    dt = np.float32 if kind == "f32" else np.float64
    nprod = None if kind == "f32" else 6
    Ch, flags = run_host(np.zeros((300, 0), dt), np.zeros((0, 70), dt), nprod=nprod)
    assert flags == 0 and np.all(Ch == 0)
    Ch, flags = run_host(np.zeros((0, 5), dt), np.zeros((5, 7), dt), nprod=nprod)
    assert Ch.shape == (0, 7)


def test_host_flags_report_nonfinite_input(dev):
    A, B = synth.gemm_inputs("f32", 64, 64, 64, 42)
    A[3, 5] = np.inf
    _, flags = run_host(A, B)
    assert flags & emu.FLAG_NONFINITE


def test_host_repeated_calls_and_interleaving(dev):
    """Back-to-back calls reuse the library's streams and events; every call
    must still see its own inputs."""
    torch = emu._torch()
    outs = []
    for seed in (51, 52, 53):
        A, B = synth.gemm_inputs("f32", 700, 300, 600, seed)
        Ah, Bh = host(A), host(B)
        C, ws = emu.gemm_host(Ah, Bh)
        outs.append((A, B, Ah, Bh, C, ws))
    torch.cuda.synchronize()
    for A, B, _, _, C, _ in outs:
        Cd, _ = gemm_f32_one_accumulator(to_dev(A, dev), to_dev(B, dev))
        np.testing.assert_array_equal(C.numpy().view(np.uint32), Cd.cpu().numpy().view(np.uint32))
