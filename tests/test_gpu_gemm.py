"""Emulated GEMM on the GPU against the oracle, through the C-ABI.

FP32 mode: |C - C_oracle| <= 1e-5 (|A||B|) per element (the tensor cores
accumulate the six products in a different FP32 order than the oracle).
FP64 mode: every FP32 chunk partial is exact and the drain adds them in the
oracle's order, so C must equal the oracle bit for bit; the accuracy bar
against a double-double reference (no more than 2x the oracle's own e_F and
e_max) then holds with equality.
"""
import ctypes

import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import abs_ab, device, fp32_within_tolerance, sample_rows, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


# ----------------------------------------------------------------- FP32 mode
@pytest.mark.parametrize("M,N,K,seed", [
    (256, 256, 256, 0),      # the paper's smallest square case
    (300, 333, 700, 1),      # ragged in every dimension, three K-chunks
    (37, 200, 513, 2),       # fewer rows than one tile, chunk tail of 1
    (129, 257, 33, 3),       # one element past a tile edge, K below one K-block
    (1, 1, 1, 4),
    (128, 512, 64, 5),
])
def test_gemm_f32_parity(dev, M, N, K, seed):
    A, B = synth.gemm_inputs("f32", M, N, K, seed)
    C, ws = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    assert emu.read_flags(ws) == 0
    Co, _ = oracle.gemm_f32(A, B)
    ok, worst = fp32_within_tolerance(C.cpu().numpy(), Co, A, B)
    assert ok, worst


def test_gemm_f32_strided_operands(dev):
    M, N, K = 190, 140, 300
    A, B = synth.gemm_inputs("f32", M, N, K, 11)
    Cbig = emu._torch().zeros((M, N + 12), dtype=emu._torch().float32, device=dev)
    C = Cbig[:, :N]
    emu.gemm_f32(to_dev(A, dev, ld_pad=4), to_dev(B, dev, ld_pad=9), C=C)
    Co, _ = oracle.gemm_f32(A, B)
    ok, worst = fp32_within_tolerance(C.cpu().numpy(), Co, A, B)
    assert ok, worst
    assert not Cbig[:, N:].any()


def test_gemm_f32_chunk_edge_case(dev):
    """The chunk-length pin's input: the product is exactly representable."""
    A = np.zeros((2, 512), dtype=np.float32)
    A[0, :256] = 1.0
    A[0, 256:] = 2.0**-22
    A[1, :128] = 1.0
    A[1, 128:256] = 2.0**-22
    B = np.ones((512, 1), dtype=np.float32)
    C, _ = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    Co, _ = oracle.gemm_f32(A, B)
    ok, worst = fp32_within_tolerance(C.cpu().numpy(), Co, A, B)
    assert ok, worst


def test_gemm_f32_exact_integers(dev):
    rng = np.random.default_rng(4)
    A = rng.integers(-12, 13, size=(160, 700)).astype(np.float32)
    B = rng.integers(-12, 13, size=(700, 300)).astype(np.float32)
    C, _ = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    assert np.array_equal(C.cpu().numpy().astype(np.int64), A.astype(np.int64) @ B.astype(np.int64))


def test_prodsum_f32_from_gpu_planes(dev):
    M, N, K = 260, 300, 520
    A, B = synth.gemm_inputs("f32", M, N, K, 21)
    ldk = emu.gemm_ldk(K)
    Ap, ws = emu.split_f32(to_dev(A, dev), ldcomp=ldk)
    Bp, _ = emu.split_f32(to_dev(B, dev), transpose=True, ldcomp=ldk, ws=ws)
    C, _ = emu.prodsum_f32(Ap, Bp, M, N, K)
    Co = oracle.prodsum_f32(oracle.split_f32(A)[0], oracle.split_f32(B)[0])
    ok, worst = fp32_within_tolerance(C.cpu().numpy(), Co, A, B)
    assert ok, worst


# ----------------------------------------------------------------- FP64 mode
@pytest.mark.parametrize("nprod", [6, 10, 15, 21])
@pytest.mark.parametrize("M,N,K,seed", [(200, 136, 300, 1), (130, 257, 520, 2), (1, 1, 1, 3)])
def test_gemm_f64_bitexact(dev, nprod, M, N, K, seed):
    A, B = synth.gemm_inputs("f64", M, N, K, seed)
    C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
    assert emu.read_flags(ws) == 0
    Co, _ = oracle.gemm_f64(A, B, nprod)
    assert np.array_equal(C.cpu().numpy(), Co)


@pytest.mark.parametrize("phi", [0.5, 4.0])
@pytest.mark.parametrize("nprod", [10, 21])
def test_gemm_f64_scaled_bitexact(dev, phi, nprod):
    A, B = synth.gemm_inputs("f64_scaled", 96, 140, 600, 5, phi=phi)
    C, ws = emu.gemm_f64(to_dev(A, dev, ld_pad=3), to_dev(B, dev), nprod)
    assert emu.read_flags(ws) == 0
    Co, _ = oracle.gemm_f64(A, B, nprod)
    assert np.array_equal(C.cpu().numpy(), Co)


@pytest.mark.parametrize("M,N,K,seed", [(150, 260, 513, 8), (64, 130, 2048, 9)])
def test_cancel_class_parity(dev, M, N, K, seed):
    """Cancellation-sensitive inputs (A = [P | P], B = [Q ; -Q + 2^-20 R]):
    FP32 within the scaled bar, FP64 bit for bit, at a ragged odd K."""
    A, B = synth.gemm_inputs("f32_cancel", M, N, K, seed)
    C, ws = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    assert emu.read_flags(ws) == 0
    Co, _ = oracle.gemm_f32(A, B)
    ok, worst = fp32_within_tolerance(C.cpu().numpy(), Co, A, B)
    assert ok, worst
    A, B = synth.gemm_inputs("f64_cancel", M, N, K, seed)
    for nprod in (6, 21):
        C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
        assert emu.read_flags(ws) == 0
        assert np.array_equal(C.cpu().numpy(), oracle.gemm_f64(A, B, nprod)[0]), nprod


def test_gemm_f64_partials_at_the_2pow24_edge(dev):
    """Chunk partials needing all 24 FP32 bits must come out of the tensor
    cores exact (the oracle pin's input, widened to a full tile)."""
    K = 512
    A = np.full((130, K), -255 / 256)
    B = np.full((K, 140), -255 / 256)
    B[0, :] = -254 / 256
    C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), 6)
    assert emu.read_flags(ws) == 0
    assert np.all(C.cpu().numpy() == (65025 * 511 + 255 * 254) * 2.0**-16)


def test_gemm_f64_exact_integers(dev):
    rng = np.random.default_rng(5)
    A = rng.integers(-2**15, 2**15 + 1, size=(140, 520)).astype(np.float64)
    B = rng.integers(-2**15, 2**15 + 1, size=(520, 150)).astype(np.float64)
    C, _ = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), 6)
    assert np.array_equal(C.cpu().numpy(), (A.astype(np.int64) @ B.astype(np.int64)).astype(np.float64))


def test_prodsum_f64_from_gpu_planes(dev):
    M, N, K = 150, 170, 400
    A, B = synth.gemm_inputs("f64", M, N, K, 8)
    ldk = emu.gemm_ldk(K)
    Ap, vA, ws = emu.split_f64(to_dev(A, dev), ldcomp=ldk)
    Bp, vB, _ = emu.split_f64(to_dev(B, dev), transpose=True, ldcomp=ldk, ws=ws)
    for nprod in (6, 21):
        Co = oracle.prodsum_f64(oracle.split_f64(A)[0], oracle.split_f64(B)[0], nprod)
        C, _ = emu.prodsum_f64(Ap, Bp, M, N, K, nprod, vA=vA, vB=vB)       # bounded plain adds
        assert np.array_equal(C.cpu().numpy(), Co)
        C, _ = emu.prodsum_f64(Ap, Bp, M, N, K, nprod)                     # every add error-free
        assert np.array_equal(C.cpu().numpy(), Co)


def test_prodsum_f64_error_free_path_at_the_2pow24_edge(dev):
    """Without level exponents every partial goes through TwoSum; with them the
    running sums pass 2^24 units after two chunks and take the same path."""
    K = 768
    A = np.full((130, K), -255 / 256)
    B = np.full((K, 140), -255 / 256)
    B[0, :] = -254 / 256
    ldk = emu.gemm_ldk(K)
    Ap, vA, ws = emu.split_f64(to_dev(A, dev), ldcomp=ldk)
    Bp, vB, _ = emu.split_f64(to_dev(B, dev), transpose=True, ldcomp=ldk, ws=ws)
    want = (65025 * 767 + 255 * 254) * 2.0**-16
    for va, vb in ((vA, vB), (None, None)):
        C, _ = emu.prodsum_f64(Ap, Bp, 130, 140, K, 6, vA=va, vB=vb)
        assert np.all(C.cpu().numpy() == want)


@pytest.mark.parametrize("nprod", [6, 21])
def test_gemm_f64_long_k_positive_sums(dev, nprod):
    """Positive inputs: every product's running sum grows linearly, passes
    2^24 units within a few chunks and keeps moving its coarse part into the
    low word (40 chunks of K, ragged tiles); still bit for bit."""
    M, N, K = 130, 200, 256 * 40 + 17
    rng = np.random.default_rng(31)
    A = rng.uniform(0.5, 1.0, size=(M, K))
    B = rng.uniform(0.5, 1.0, size=(K, N))
    C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
    assert emu.read_flags(ws) == 0
    assert np.array_equal(C.cpu().numpy(), oracle.gemm_f64(A, B, nprod)[0])


def _level_gap_inputs(shape, seed, gap_level):
    """Entries whose residual after level gap_level - 1 is far below the
    speculative 2^-8 step, so the speculative levels hold below gap_level and
    fail at it."""
    rng = np.random.default_rng(seed)
    X = rng.integers(-127, 128, size=shape) * 2.0**10
    for r in range(1, gap_level):
        X = X + rng.integers(-127, 128, size=shape) * 2.0**(10 - 8 * r)
    X = X + rng.integers(-127, 128, size=shape) * 2.0**(10 - 8 * gap_level - 30)
    X.flat[0] = 127 * 2.0**10
    return X


@pytest.mark.parametrize("gap_level", [1, 4])
@pytest.mark.parametrize("nprod", [6, 10, 15, 21])
def test_gemm_f64_speculation_fails(dev, nprod, gap_level):
    """The GEMM's split forms only the d slices its product-sum uses; when the
    speculative levels fail below d the literal passes redo them, when they
    fail only from d on they are never needed.  Either way C is the oracle's."""
    A = _level_gap_inputs((300, 400), 40 + gap_level, gap_level)
    B = _level_gap_inputs((400, 260), 50 + gap_level, gap_level)
    _, vA, _ = oracle.split_f64(A)
    assert vA[gap_level] != vA[0] - 8 * gap_level
    C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
    assert emu.read_flags(ws) == 0
    assert np.array_equal(C.cpu().numpy(), oracle.gemm_f64(A, B, nprod)[0])


# ------------------------------------------------------------ edges, errors
def test_zero_sizes_and_empty_k(dev):
    torch = emu._torch()
    A = torch.ones((5, 0), dtype=torch.float32, device=dev)
    B = torch.ones((0, 7), dtype=torch.float32, device=dev)
    C = torch.full((5, 7), 3.0, dtype=torch.float32, device=dev)
    emu.gemm_f32(A, B, C=C)
    assert not C.any()                                  # K = 0 writes zeros
    C64 = torch.full((5, 7), 3.0, dtype=torch.float64, device=dev)
    emu.gemm_f64(A.double(), B.double(), 21, C=C64)
    assert not C64.any()
    Cm = torch.full((0, 7), 3.0, dtype=torch.float32, device=dev)
    emu.gemm_f32(torch.ones((0, 4), device=dev), torch.ones((4, 7), device=dev), C=Cm)   # no-op


def test_error_codes(dev):
    torch = emu._torch()
    A = torch.ones((64, 64), dtype=torch.float64, device=dev)
    ws = emu.workspace(emu.emu_gemm_workspace_bytes(64, 64, 64, 64), dev)
    C = torch.empty((64, 64), dtype=torch.float64, device=dev)
    s = emu._stream(None)
    assert emu.emu_gemm_f64(64, 64, 64, A.data_ptr(), 64, A.data_ptr(), 64, C.data_ptr(), 64, 9,
                            ws.data_ptr(), ws.numel(), s) == 1
    assert emu.emu_gemm_f64(64, 64, 64, A.data_ptr(), 64, A.data_ptr(), 64, C.data_ptr(), 64, 6,
                            ws.data_ptr(), ws.numel() - 1, s) == 3
    planes = torch.zeros((6, 64, 72), dtype=torch.int16, device=dev)
    # plane rows not a multiple of 16 bytes -> MISALIGNED; base off by 2 bytes -> MISALIGNED
    assert emu.emu_prodsum_f64(64, 64, 64, planes.data_ptr(), planes.data_ptr(), 66, None, None, 6, C.data_ptr(),
                               64, ws.data_ptr(), ws.numel(), s) == 2
    assert emu.emu_prodsum_f64(64, 64, 64, planes.data_ptr() + 2, planes.data_ptr(), 72, None, None, 6,
                               C.data_ptr(), 64, ws.data_ptr(), ws.numel(), s) == 2
    v = torch.zeros(6, dtype=torch.int32, device=dev)
    assert emu.emu_prodsum_f64(64, 64, 64, planes.data_ptr(), planes.data_ptr(), 72, v.data_ptr(), None, 6,
                               C.data_ptr(), 64, ws.data_ptr(), ws.numel(), s) == 1    # vA without vB


def test_watchdog_timeout_reports_and_context_survives(dev):
    """A bounded wait on a barrier nobody completes gives up, flags
    EMU_FLAG_TIMEOUT, and the context keeps working afterwards."""
    ws = emu.workspace(emu.emu_split_workspace_bytes(32), dev)
    assert emu.emu_selftest_timeout(ws.data_ptr(), ws.numel(), 2000, emu._stream(None)) == 0
    assert emu.read_flags(ws) == emu.FLAG_TIMEOUT
    A, B = synth.gemm_inputs("f64", 64, 64, 64, 1)
    C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), 6)
    assert emu.read_flags(ws) == 0
    assert np.array_equal(C.cpu().numpy(), oracle.gemm_f64(A, B, 6)[0])


def test_read_flags_reports_domain_violation(dev):
    A, B = synth.gemm_inputs("f64", 64, 64, 64, 1)
    A[3, 3] = 2.0**-130
    _, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), 6)
    assert emu.read_flags(ws) & emu.FLAG_RANGE


# -------------------------------------------- full sizes, sampled output rows
# Rows of C are independent once the (global) split is done, so the oracle
# computes only sampled rows: the A planes of those rows against all of B.
def _dd_rows(A, B, rows):
    return oracle.ref_dd(np.ascontiguousarray(A[rows]), B)


def test_fullsize_fp32_n16384_sampled(dev):
    n = 16384
    A, B = synth.gemm_inputs("f32", n, n, n, n)
    C, ws = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    assert emu.read_flags(ws) == 0
    rows = sample_rows(n, 3, 1)
    Cg = C.cpu().numpy()[rows]
    del C, ws
    Co = oracle.prodsum_f32(oracle.split_f32(A[rows])[0], oracle.split_f32(B)[0])
    ok, worst = fp32_within_tolerance(Cg, Co, A[rows], B)
    assert ok, worst


@pytest.mark.parametrize("nprod", [6, 10, 15, 21])
def test_fullsize_fp64_n4096_sampled(dev, nprod):
    n = 4096
    A, B = synth.gemm_inputs("f64", n, n, n, 1)
    C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
    assert emu.read_flags(ws) == 0
    rows = sample_rows(n, 3, nprod)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    Cg = C.cpu().numpy()[rows]
    Co = oracle.prodsum_f64(Ap[:, rows], Bp, nprod)
    assert np.array_equal(Cg, Co)
    hi, lo = _dd_rows(A, B, rows)
    eg, eo = oracle.errors(Cg, hi, lo), oracle.errors(Co, hi, lo)
    assert eg["e_F"] <= 2 * eo["e_F"] and eg["e_max"] <= 2 * eo["e_max"]


@pytest.mark.parametrize("phi,seed", [(0.5, 3), (2.0, 4), (4.0, 5)])
def test_fullsize_fp64_scaled_n8192_sampled(dev, phi, seed):
    n = 8192
    A, B = synth.gemm_inputs("f64_scaled", n, n, n, seed, phi=phi)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    rows = sample_rows(n, 2, seed)
    for nprod in (21, 10):
        C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
        assert emu.read_flags(ws) == 0
        Cg = C.cpu().numpy()[rows]
        Co = oracle.prodsum_f64(Ap[:, rows], Bp, nprod)
        assert np.array_equal(Cg, Co)
        del C, ws


def test_fullsize_cancel_n4096_sampled(dev):
    n = 4096
    A, B = synth.gemm_inputs("f32_cancel", n, n, n, 6)
    C, ws = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    assert emu.read_flags(ws) == 0
    rows = sample_rows(n, 2, 6)
    Cg = C.cpu().numpy()[rows]
    del C, ws
    Co = oracle.prodsum_f32(oracle.split_f32(A[rows])[0], oracle.split_f32(B)[0])
    ok, worst = fp32_within_tolerance(Cg, Co, A[rows], B)
    assert ok, worst
    A, B = synth.gemm_inputs("f64_cancel", n, n, n, 7)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    for nprod in (21, 10):
        C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
        assert emu.read_flags(ws) == 0
        Cg = C.cpu().numpy()[rows]
        assert np.array_equal(Cg, oracle.prodsum_f64(Ap[:, rows], Bp, nprod)), nprod
        del C, ws


def test_fullsize_large_k_sampled(dev):
    M = N = 2048
    K = 65536
    A, B = synth.gemm_inputs("f32", M, N, K, 2)
    C, ws = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    assert emu.read_flags(ws) == 0
    rows = sample_rows(M, 1, 2)
    Cg = C.cpu().numpy()[rows]
    del C, ws
    Co = oracle.prodsum_f32(oracle.split_f32(A[rows])[0], oracle.split_f32(B)[0])
    ok, worst = fp32_within_tolerance(Cg, Co, A[rows], B)
    assert ok, worst
    A, B = synth.gemm_inputs("f64", M, N, K, 2)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    for nprod in (6, 10, 15, 21):
        C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
        assert emu.read_flags(ws) == 0
        Cg = C.cpu().numpy()[rows]
        Co = oracle.prodsum_f64(Ap[:, rows], Bp, nprod)
        assert np.array_equal(Cg, Co), nprod
        del C, ws


@pytest.mark.parametrize("M,N,K,seed", [(1024, 1024, 1024, 41), (300, 333, 700, 42), (256, 1000, 4096, 43),
                                        (129, 64, 256, 44)])
def test_gemm_f32_k_split_small_results(M, N, K, seed):
    """Small results: emu_gemm_f32 splits K in two and adds the halves into C
    in L2.  Within the FP32-mode bar of the oracle, and the same bits on a
    second run (two addends: the order of arrival does not matter)."""
    dev = device()
    A, B = synth.gemm_inputs("f32", M, N, K, seed)
    Ad, Bd = to_dev(A, dev), to_dev(B, dev)
    C1, ws = emu.gemm_f32(Ad, Bd)
    assert emu.read_flags(ws) == 0
    C2, _ = emu.gemm_f32(Ad, Bd)
    C1n = C1.cpu().numpy()
    assert np.array_equal(C1n.view(np.uint32), C2.cpu().numpy().view(np.uint32))
    rows = sample_rows(M, 6, seed) if M * N * K > 400 * 400 * 1000 else list(range(M))
    Co = oracle.prodsum_f32(oracle.split_f32(A[rows])[0], oracle.split_f32(B)[0])
    ok, worst = fp32_within_tolerance(C1n[rows], Co, A[rows], B)
    assert ok, worst
