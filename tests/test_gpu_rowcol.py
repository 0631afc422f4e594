"""FP64 split and GEMM with levels per row of A and per column of B (the
vector scaling of the standard Ozaki scheme, Eq. (ozakiscaled)) on the GPU
against the oracle's split_f64_rows / gemm_f64_rowcol.  The split is
integer work and FP64 mode keeps every chunk partial exact, so planes,
levels, flags and C must all match bit for bit."""
import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import device, planes_np, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def _check_split(X, dev, transpose, pad=0, ld_pad=0):
    prow, pcols = (X.shape[1], X.shape[0]) if transpose else X.shape
    planes, v, ws = emu.split_f64_rowcol(to_dev(X, dev, ld_pad), transpose=transpose, ldcomp=pcols + pad)
    flags = emu.read_flags(ws)
    want, wv, wflags = oracle.split_f64_rows(np.ascontiguousarray(X.T) if transpose else X)
    assert flags == wflags
    assert np.array_equal(v.cpu().numpy(), wv.T)
    if wflags == 0:
        assert np.array_equal(planes_np(planes)[:, :prow, :pcols], want)
    return wv


def _row_scaled(seed, shape, lo=-60, hi=60):
    U = synth.uniform_f64(seed, 0, shape)
    e = np.random.default_rng(seed).integers(lo, hi + 1, size=shape[0])
    return U * np.ldexp(1.0, e)[:, None]


@pytest.mark.parametrize("shape", [(1, 1), (12, 17), (64, 64), (300, 700), (257, 513)])
@pytest.mark.parametrize("transpose", [False, True])
def test_split_rowcol_uniform_bitexact(dev, shape, transpose):
    _check_split(synth.uniform_f64(41, 0, shape), dev, transpose)


@pytest.mark.parametrize("transpose", [False, True])
def test_split_rowcol_scaled_vectors_bitexact(dev, transpose):
    X = _row_scaled(42, (190, 333))
    _check_split(X.T.copy() if transpose else X, dev, transpose, pad=5, ld_pad=3)
    _check_split(synth.scaled_f64(43, 0, 4.0, (150, 90)), dev, transpose)


@pytest.mark.parametrize("transpose", [False, True])
def test_split_rowcol_early_stop_zero_and_tiny_vectors(dev, transpose):
    rng = np.random.default_rng(44)
    X = synth.uniform_f64(44, 0, (70, 50))
    X[3] = rng.integers(-100, 101, size=50)          # integers: one slice, then zero levels
    X[5] = 0.0                                       # a zero vector
    X[7] *= 2.0 ** -100                              # tiny: low slices leave the BF16 range (flagged)
    X[9] = 2.0 ** -60 * rng.integers(-127, 128, size=50) + 2.0 ** -90
    X = np.ascontiguousarray(X.T) if transpose else X
    _check_split(X, dev, transpose)


def test_split_rowcol_flags(dev):
    X = synth.uniform_f64(45, 0, (33, 47))
    for val in (np.nan, np.inf, 2.0 ** -127, 2.0 ** 129):
        Y = X.copy()
        Y[4, 5] = val
        _, _, ws = emu.split_f64_rowcol(to_dev(Y, dev))
        assert emu.read_flags(ws) == oracle.split_f64_rows(Y)[2] != 0, val


@pytest.mark.parametrize("M,N,K,nprod", [(150, 130, 300, 21), (300, 200, 700, 10), (129, 257, 520, 6), (5, 3, 1, 15)])
def test_gemm_rowcol_bitexact(dev, M, N, K, nprod):
    U, V = synth.gemm_inputs("f64", M, N, K, 46)
    rng = np.random.default_rng(46)
    A = U * np.ldexp(1.0, rng.integers(-15, 41, size=M))[:, None]      # every product unit stays normal FP32
    B = V * np.ldexp(1.0, rng.integers(-15, 41, size=N))[None, :]
    C, ws = emu.gemm_f64_rowcol(to_dev(A, dev, ld_pad=1), to_dev(B, dev, ld_pad=2), nprod)
    assert emu.read_flags(ws) == 0
    want, flags = oracle.gemm_f64_rowcol(A, B, nprod)
    assert flags == 0
    np.testing.assert_array_equal(C.cpu().numpy().view(np.uint64), want.view(np.uint64))


@pytest.mark.parametrize("nprod", [6, 21])
def test_gemm_rowcol_long_k_positive_sums(dev, nprod):
    """Positive entries over 40 K-chunks with row and column scalings of up
    to 2^6 either way: the running sums pass 2^24 units of the smallest unit
    of a thread's columns within a few chunks, and each element then carries
    at its own unit (or redoes its additions as TwoSums); bit for bit."""
    M, N, K = 130, 200, 256 * 40 + 17
    rng = np.random.default_rng(48)
    U = rng.uniform(0.5, 1.0, size=(M, K))
    V = rng.uniform(0.5, 1.0, size=(K, N))
    A = U * np.ldexp(1.0, rng.integers(-6, 7, size=M))[:, None]
    B = V * np.ldexp(1.0, rng.integers(-6, 7, size=N))[None, :]
    C, ws = emu.gemm_f64_rowcol(to_dev(A, dev), to_dev(B, dev), nprod)
    assert emu.read_flags(ws) == 0
    want, flags = oracle.gemm_f64_rowcol(A, B, nprod)
    assert flags == 0
    np.testing.assert_array_equal(C.cpu().numpy().view(np.uint64), want.view(np.uint64))


def test_gemm_rowcol_commutes_with_scaling_on_gpu(dev):
    """D_A U times V D_B equals D_A (U V) D_B exactly on the GPU path too.
    Scalings stay where every product's unit 2^(vA_5 + vB_5 - 16), about
    2^(ea + eb - 96) here, is a normal FP32 number (ea + eb >= -30): below
    that the tensor cores' FP32 partials underflow, outside the method's
    domain."""
    M, N, K = 256, 384, 1024
    U, V = synth.gemm_inputs("f64", M, N, K, 47)
    rng = np.random.default_rng(47)
    ea, eb = rng.integers(-15, 41, size=M), rng.integers(-15, 41, size=N)
    A, B = U * np.ldexp(1.0, ea)[:, None], V * np.ldexp(1.0, eb)[None, :]
    C1, _ = emu.gemm_f64_rowcol(to_dev(A, dev), to_dev(B, dev), 21)
    C0, _ = emu.gemm_f64_rowcol(to_dev(U, dev), to_dev(V, dev), 21)
    scale = np.ldexp(1.0, ea)[:, None] * np.ldexp(1.0, eb)[None, :]
    np.testing.assert_array_equal(C1.cpu().numpy(), C0.cpu().numpy() * scale)
    # whole-matrix levels are not scale-invariant on such inputs
    Cg, _ = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), 21)
    assert not np.array_equal(Cg.cpu().numpy(), C0.cpu().numpy() * scale)


@pytest.mark.parametrize("transpose", [False, True])
def test_split_rowcol_some_vectors_fail_speculation(dev, transpose):
    """Rows whose residual shrinks by far more than 2^-8 per level (integers at
    three widely separated scales) fail the speculative levels and are redone
    by the literal passes alone; uniform rows keep their speculative levels."""
    rng = np.random.default_rng(48)
    X = synth.uniform_f64(48, 0, (96, 130))
    for i in (3, 17, 40, 95):
        X[i] = (rng.integers(-127, 128, size=130) * 2.0 ** 10 + rng.integers(-127, 128, size=130) * 2.0 ** -20
                + rng.integers(-127, 128, size=130) * 2.0 ** -50)
        X[i, 0] = 127 * 2.0 ** 10
    X = np.ascontiguousarray(X.T) if transpose else X
    wv = _check_split(X, dev, transpose)
    assert wv[3, 1] != wv[3, 0] - 8 and wv[4, 1] == wv[4, 0] - 8


@pytest.mark.parametrize("transpose", [False, True])
def test_split_rowcol_fix_path_large(dev, transpose):
    """Failed vectors spread over a matrix that spans every block of the
    launch: the literal passes run across the whole grid with barriers."""
    rng = np.random.default_rng(49)
    X = synth.uniform_f64(49, 0, (1500, 1100))
    bad = rng.choice(1500, size=60, replace=False)
    for i in bad:
        X[i] = (rng.integers(-127, 128, size=1100) * 2.0 ** 10 + rng.integers(-127, 128, size=1100) * 2.0 ** -20
                + rng.integers(-127, 128, size=1100) * 2.0 ** -50)
        X[i, 0] = 127 * 2.0 ** 10
    X = np.ascontiguousarray(X.T) if transpose else X
    wv = _check_split(X, dev, transpose)
    good = next(i for i in range(1500) if i not in set(bad))
    assert wv[bad[0], 1] != wv[bad[0], 0] - 8 and wv[good, 1] == wv[good, 0] - 8
