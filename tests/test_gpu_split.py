"""GPU split kernels against the oracle: bit-exact planes, levels and flags.

Eq. (fp32split) and Eq. (fp64split) are integer-valued decisions on FP32/FP64
arithmetic, so the bar is bit equality.  B operands are split transposed
(K-major planes); they are compared with the oracle's planes transposed.
"""
import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import device, planes_np, random_finite_f32, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def _check_f32(X, dev, transpose, pad, ld_pad=0):
    rows, cols = X.shape
    rows_out, cols_out = (cols, rows) if transpose else (rows, cols)
    ldcomp = cols_out + pad
    planes, ws = emu.split_f32(to_dev(X, dev, ld_pad), transpose=transpose, ldcomp=ldcomp)
    flags = emu.read_flags(ws)
    want, wflags = oracle.split_f32(X)
    if transpose:
        want = want.transpose(0, 2, 1)
    got = planes_np(planes)
    assert flags == wflags
    assert np.array_equal(got[:, :rows_out, :cols_out], want)
    assert not got[:, :, cols_out:].any()          # padding untouched (zero-initialised)


@pytest.mark.parametrize("shape", [(1, 1), (37, 129), (64, 64), (65, 3), (300, 700), (129, 1000)])
@pytest.mark.parametrize("transpose", [False, True])
def test_split_f32_uniform_bitexact(dev, shape, transpose):
    X = synth.uniform_f32(7, 0, shape)
    _check_f32(X, dev, transpose, pad=0)


@pytest.mark.parametrize("transpose", [False, True])
@pytest.mark.parametrize("pad,ld_pad", [(0, 0), (3, 5), (8, 4)])
def test_split_f32_bit_patterns(dev, transpose, pad, ld_pad):
    """Zeros, subnormals, ties and large magnitudes; odd leading dimensions."""
    X = random_finite_f32((131, 203), 3)
    _check_f32(X, dev, transpose, pad, ld_pad)


def test_split_f32_flags(dev):
    X = synth.uniform_f32(1, 0, (40, 50))
    X[5, 7] = np.nan
    planes, ws = emu.split_f32(to_dev(X, dev))
    assert emu.read_flags(ws) & emu.FLAG_NONFINITE
    X = synth.uniform_f32(1, 0, (40, 50))
    X[0, 0] = np.float32(3.4e38)                   # the first slice rounds past the largest BF16
    planes, ws = emu.split_f32(to_dev(X, dev))
    assert emu.read_flags(ws) == oracle.split_f32(X)[1] == emu.FLAG_SLICE


def _check_f64(X, dev, transpose, pad=0, ld_pad=0):
    rows, cols = X.shape
    rows_out, cols_out = (cols, rows) if transpose else (rows, cols)
    planes, v, ws = emu.split_f64(to_dev(X, dev, ld_pad), transpose=transpose, ldcomp=cols_out + pad)
    flags = emu.read_flags(ws)
    want, wv, wflags = oracle.split_f64(X)
    if transpose:
        want = want.transpose(0, 2, 1)
    assert flags == wflags
    assert np.array_equal(v.cpu().numpy(), wv)
    if wflags == 0:
        assert np.array_equal(planes_np(planes)[:, :rows_out, :cols_out], want)
    return wv


@pytest.mark.parametrize("shape", [(1, 1), (12, 17), (64, 64), (300, 700), (257, 513)])
@pytest.mark.parametrize("transpose", [False, True])
def test_split_f64_uniform_bitexact(dev, shape, transpose):
    wv = _check_f64(synth.uniform_f64(1, 0, shape), dev, transpose)
    if shape[0] * shape[1] >= 4096:
        assert list(np.diff(wv)) == [-8] * 5           # the speculative levels held


@pytest.mark.parametrize("phi", [0.5, 2.0, 4.0])
@pytest.mark.parametrize("transpose", [False, True])
def test_split_f64_scaled_class_bitexact(dev, phi, transpose):
    _check_f64(synth.scaled_f64(5, 0, phi, (190, 333)), dev, transpose, pad=5, ld_pad=3)


@pytest.mark.parametrize("transpose", [False, True])
def test_split_f64_fix_path_levels(dev, transpose):
    """Inputs whose residual shrinks by far more than 2^-8 per level: the
    speculative levels fail and the gated literal passes take over."""
    rng = np.random.default_rng(9)
    a = rng.integers(-127, 128, size=(150, 90)).astype(np.float64)
    b = rng.integers(-127, 128, size=(150, 90)).astype(np.float64)
    c = rng.integers(-127, 128, size=(150, 90)).astype(np.float64)
    X = a * 2.0**10 + b * 2.0**-20 + c * 2.0**-50
    X[0, 0] = 127 * 2.0**10
    wv = _check_f64(X, dev, transpose)
    assert wv[1] != wv[0] - 8                           # the fix path really ran
    # integers: one slice, then zero levels (verifier stops at the zero residual)
    Y = rng.integers(-100, 101, size=(70, 33)).astype(np.float64)
    Y[3, 3] = 100.0
    wv = _check_f64(Y, dev, transpose)
    assert wv[1] == oracle.ZERO_LEVEL
    _check_f64(np.zeros((20, 30)), dev, transpose)


@pytest.mark.parametrize("transpose", [False, True])
def test_split_f64_fix_path_large(dev, transpose):
    """The fix path on a matrix that spans every block of its launch: the
    literal passes run across the whole grid with barriers between them."""
    rng = np.random.default_rng(10)
    shape = (1500, 1300)
    X = (rng.integers(-127, 128, size=shape) * 2.0**10 + rng.integers(-127, 128, size=shape) * 2.0**-20
         + rng.integers(-127, 128, size=shape) * 2.0**-50)
    X[0, 0] = 127 * 2.0**10
    wv = _check_f64(X, dev, transpose)
    assert wv[1] != wv[0] - 8


@pytest.mark.parametrize("gap_level", [1, 2, 3, 4, 5])
@pytest.mark.parametrize("scale", [30, 3])
def test_split_f64_level_gap(dev, gap_level, scale):
    """The speculative levels hold below gap_level and fail at it, the residual
    there 2^-scale below the speculative step: far below (scale 30, under the
    fused pass's fixed-point unit, where only a sticky bit is left of it) or
    just below (scale 3).  Planes and levels as the oracle's, both layouts."""
    rng = np.random.default_rng(60 + gap_level)
    shape = (300, 270)
    X = rng.integers(-127, 128, size=shape) * 2.0**10
    for r in range(1, gap_level):
        X = X + rng.integers(-127, 128, size=shape) * 2.0**(10 - 8 * r)
    X = X + rng.integers(-127, 128, size=shape) * 2.0**(10 - 8 * gap_level - scale)
    X[0, 0] = 127 * 2.0**10
    for transpose in (False, True):
        wv = _check_f64(X, dev, transpose)
        assert wv[gap_level] != wv[0] - 8 * gap_level


@pytest.mark.parametrize("nslices", [3, 4, 5, 6])
@pytest.mark.parametrize("gap_level", [0, 2, 4])
def test_split_f64_slices(dev, nslices, gap_level):
    """emu_split_f64_slices: planes and levels below nslices as the oracle's,
    with the speculative levels holding (gap_level 0) or failing below or
    above nslices."""
    rng = np.random.default_rng(80 + gap_level)
    shape = (260, 190)
    if gap_level == 0:
        X = synth.uniform_f64(7, 0, shape)
    else:
        X = rng.integers(-127, 128, size=shape) * 2.0**10
        for r in range(1, gap_level):
            X = X + rng.integers(-127, 128, size=shape) * 2.0**(10 - 8 * r)
        X = X + rng.integers(-127, 128, size=shape) * 2.0**(10 - 8 * gap_level - 30)
        X[0, 0] = 127 * 2.0**10
    want, wv, wflags = oracle.split_f64(X)
    assert wflags == 0
    for transpose in (False, True):
        planes, v, ws = emu.split_f64(to_dev(X, dev), transpose=transpose, nslices=nslices)
        assert emu.read_flags(ws) == 0
        got = planes_np(planes)
        ref = want.transpose(0, 2, 1) if transpose else want
        assert np.array_equal(v.cpu().numpy()[:nslices], wv[:nslices])
        assert np.array_equal(got[:nslices], ref[:nslices])


def test_split_f64_flags(dev):
    X = synth.uniform_f64(3, 0, (33, 47))
    for val in (np.nan, np.inf, 2.0**-127, 2.0**129):
        Y = X.copy()
        Y[4, 5] = val
        planes, v, ws = emu.split_f64(to_dev(Y, dev))
        assert emu.read_flags(ws) == oracle.split_f64(Y)[2] != 0, val
    Y = np.full((4, 4), 2.0**-120)
    Y[0, 0] = 2.0**-120 + 2.0**-140                    # a nonzero slice below 2^-126
    _check_f64(Y, dev, False)
    assert oracle.split_f64(Y)[2] == emu.FLAG_SLICE


def test_split_fullsize_fp32_a_plane_bitexact(dev):
    """Full size (M = K = 16384, FP32 sweep top): every plane bit-exact."""
    n = 16384
    A = synth.uniform_f32(n, 0, (n, n))
    planes, ws = emu.split_f32(to_dev(A, dev))
    assert emu.read_flags(ws) == 0
    want, _ = oracle.split_f32(A)
    assert np.array_equal(planes_np(planes), want)


def test_split_fullsize_fp64_scaled_b_transposed_bitexact(dev):
    """Full size (8192 x 8192, scaled class phi = 4), B orientation."""
    n = 8192
    B = synth.scaled_f64(5, n * n, 4.0, (n, n))
    planes, v, ws = emu.split_f64(to_dev(B, dev), transpose=True)
    assert emu.read_flags(ws) == 0
    want, wv, _ = oracle.split_f64(B)
    assert np.array_equal(v.cpu().numpy(), wv)
    assert np.array_equal(planes_np(planes), want.transpose(0, 2, 1))


@pytest.mark.parametrize("scale_exp", [-70, -77, -78, -79, -100, 100, 126])
@pytest.mark.parametrize("transpose", [False, True])
def test_split_f64_scales_bitexact(dev, scale_exp, transpose):
    """Uniform data scaled by 2^e: the split takes its 32-bit fast form for
    v0 >= -78 and its checked general form below (where low slices leave the
    BF16 normal range and are flagged); both must match the oracle."""
    X = synth.uniform_f64(7, 0, (130, 75)) * 2.0**scale_exp
    _check_f64(X, dev, transpose, pad=3)


@pytest.mark.parametrize("shape", [(0, 5), (7, 0), (0, 0)])
@pytest.mark.parametrize("transpose", [False, True])
def test_split_f64_empty_operands(dev, shape, transpose):
    """An empty operand has no nonzero entry: all six levels are zero and no
    flag is raised, through the whole-matrix and the per-vector splits."""
    torch = emu._torch()
    X = torch.zeros(shape, dtype=torch.float64, device=dev)
    planes, v, ws = emu.split_f64(X, transpose=transpose, ldcomp=8)
    assert emu.read_flags(ws) == 0
    assert v.cpu().tolist() == [oracle.ZERO_LEVEL] * 6
    if (shape[1] if transpose else shape[0]) > 0:
        planes, v, ws = emu.split_f64_rowcol(X, transpose=transpose, ldcomp=8)
        assert emu.read_flags(ws) == 0
        assert (v.cpu().numpy() == oracle.ZERO_LEVEL).all()


def _gap_matrix(rng, shape, gap_level, scale=3):
    """Integers times descending powers of two, so that the speculative levels
    hold below gap_level and fail at it (gap_level 0: they all hold)."""
    X = rng.integers(-127, 128, size=shape) * 2.0**10
    for r in range(1, gap_level or 6):
        X = X + rng.integers(-127, 128, size=shape) * 2.0**(10 - 8 * r)
    if gap_level:
        X = X + rng.integers(-127, 128, size=shape) * 2.0**(10 - 8 * gap_level - scale)
    X[0, 0] = 127 * 2.0**10
    return X


@pytest.mark.parametrize("M,N,K", [(300, 333, 700), (129, 257, 33), (1000, 64, 520), (1, 1, 1)])
def test_pair_splits_equal_single_operand_splits(dev, M, N, K):
    """emu_split_f32_pair / emu_split_f64_pair (the split step the GEMMs run,
    both operands sharing launches): planes and levels identical to the
    single-operand splits; FP64 with the speculative levels holding, and
    failing at a level of A only or of B only."""
    torch = emu._torch()
    ldk = emu.gemm_ldk(K)
    A, B = synth.gemm_inputs("f32", M, N, K, 71)
    Ad, Bd = to_dev(A, dev), to_dev(B, dev)
    Ap = torch.zeros((3, M, ldk), dtype=torch.int16, device=dev)
    Bp = torch.zeros((3, N, ldk), dtype=torch.int16, device=dev)
    ws = emu.workspace(emu.emu_split_workspace_bytes(32), dev)
    assert emu.emu_split_f32_pair(M, N, K, Ad.data_ptr(), K, Bd.data_ptr(), N, Ap.data_ptr(), Bp.data_ptr(), ldk,
                                  ws.data_ptr(), ws.numel(), emu._stream(None)) == 0
    assert emu.read_flags(ws) == 0
    Ar, _ = emu.split_f32(Ad, ldcomp=ldk)
    Br, _ = emu.split_f32(Bd, transpose=True, ldcomp=ldk)
    assert torch.equal(Ap[:, :, :K], Ar[:, :, :K]) and torch.equal(Bp[:, :, :K], Br[:, :, :K])
    rng = np.random.default_rng(72)
    for nslices in (3, 6):
        for ga, gb in ((0, 0), (2, 0), (0, 4)):
            A64 = _gap_matrix(rng, (M, K), ga)
            B64 = _gap_matrix(rng, (K, N), gb)
            Ad, Bd = to_dev(A64, dev), to_dev(B64, dev)
            Ap = torch.zeros((6, M, ldk), dtype=torch.int16, device=dev)
            Bp = torch.zeros((6, N, ldk), dtype=torch.int16, device=dev)
            vA = torch.empty(6, dtype=torch.int32, device=dev)
            vB = torch.empty(6, dtype=torch.int32, device=dev)
            ws = emu.workspace(emu.emu_split_workspace_bytes(64), dev)
            assert emu.emu_split_f64_pair(M, N, K, Ad.data_ptr(), K, Bd.data_ptr(), N, Ap.data_ptr(), Bp.data_ptr(),
                                          ldk, nslices, vA.data_ptr(), vB.data_ptr(), ws.data_ptr(), ws.numel(),
                                          emu._stream(None)) == 0
            Ar, vAr, wa = emu.split_f64(Ad, ldcomp=ldk, nslices=nslices)
            Br, vBr, wb = emu.split_f64(Bd, transpose=True, ldcomp=ldk, nslices=nslices)
            assert emu.read_flags(ws) == emu.read_flags(wa) | emu.read_flags(wb)
            n = nslices
            assert torch.equal(Ap[:n, :, :K], Ar[:n, :, :K]), (nslices, ga, gb)
            assert torch.equal(Bp[:n, :, :K], Br[:n, :, :K]), (nslices, ga, gb)
            assert torch.equal(vA[:n], vAr[:n]) and torch.equal(vB[:n], vBr[:n]), (nslices, ga, gb)
