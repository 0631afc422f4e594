"""General GEMM (emu_gemm_ex_f32 / emu_gemm_ex_f64) on the GPU against the
oracle: C <- alpha op(A) op(B) + beta C for every placement of the operands.
FP32 mode: the product differs from the oracle's within the FP32 bar
(1e-5 |A||B|), scaled by |alpha|, plus the epilogue's own roundings.  FP64
mode: the product is bit-exact and the epilogue performs the same IEEE
operations, so C must equal the oracle bit for bit."""
import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import abs_ab, device, gemm_f32_one_accumulator, to_dev

pytestmark = pytest.mark.gpu

COMBOS = [(0, 0), (0, 1), (1, 0), (1, 1)]
SCALARS = [(1.0, 0.0), (2.5, 0.0), (-0.75, 1.5)]


@pytest.fixture(scope="module")
def dev():
    return device()


def _stored(A_eff, op):
    return np.ascontiguousarray(A_eff.T) if op else A_eff


@pytest.mark.parametrize("opA,opB", COMBOS)
@pytest.mark.parametrize("alpha,beta", SCALARS)
def test_gemm_ex_f32_parity(dev, opA, opB, alpha, beta):
    M, N, K = 150, 130, 300
    A_eff, B_eff = synth.gemm_inputs("f32", M, N, K, 61)
    C0 = synth.uniform_f32(62, 0, (M, N))
    A, B = _stored(A_eff, opA), _stored(B_eff, opB)
    Cd = to_dev(C0, dev, ld_pad=5)
    C, ws = emu.gemm_ex(to_dev(A, dev, ld_pad=3), to_dev(B, dev, ld_pad=7), opA, opB, alpha, beta, C=Cd)
    assert emu.read_flags(ws) == 0
    got = C.cpu().numpy()
    want, flags = oracle.gemm_ex(opA, opB, alpha, A, B, beta, C0)
    assert flags == 0
    P_or, _ = oracle.gemm_f32(A_eff, B_eff)
    bound = (abs(alpha) * 1e-5 * abs_ab(A_eff, B_eff)
             + 2.0**-21 * (np.abs(alpha * P_or.astype(np.float64)) + abs(beta) * np.abs(C0.astype(np.float64))))
    assert np.all(np.abs(got.astype(np.float64) - want.astype(np.float64)) <= bound)
    if (alpha, beta) == (1.0, 0.0) and (opA, opB) == (0, 0):
        Cg, _ = gemm_f32_one_accumulator(to_dev(A_eff, dev), to_dev(B_eff, dev))
        np.testing.assert_array_equal(got.view(np.uint32), Cg.cpu().numpy().view(np.uint32))


@pytest.mark.parametrize("opA,opB", COMBOS)
@pytest.mark.parametrize("alpha,beta", SCALARS + [(-2.0, 0.5)])
def test_gemm_ex_f64_bitexact(dev, opA, opB, alpha, beta):
    M, N, K = 140, 90, 520
    A_eff, B_eff = synth.gemm_inputs("f64", M, N, K, 63)
    C0 = synth.uniform_f64(64, 0, (M, N))
    A, B = _stored(A_eff, opA), _stored(B_eff, opB)
    C, ws = emu.gemm_ex(to_dev(A, dev, ld_pad=1), to_dev(B, dev, ld_pad=2), opA, opB, alpha, beta,
                        C=to_dev(C0, dev, ld_pad=3), nprod=15)
    assert emu.read_flags(ws) == 0
    want, _ = oracle.gemm_ex(opA, opB, alpha, A, B, beta, C0, nprod=15)
    np.testing.assert_array_equal(C.cpu().numpy().view(np.uint64), want.view(np.uint64))


@pytest.mark.parametrize("kind", ["f32", "f64"])
def test_gemm_ex_beta_zero_ignores_nan_c_and_k_zero(dev, kind):
    torch = emu._torch()
    dt = np.float32 if kind == "f32" else np.float64
    nprod = None if kind == "f32" else 6
    A, B = synth.gemm_inputs(kind, 33, 21, 70, 65)
    Cn = to_dev(np.full((33, 21), np.nan, dtype=dt), dev)
    C, _ = emu.gemm_ex(to_dev(A, dev), to_dev(B, dev), 0, 0, 1.5, 0.0, C=Cn, nprod=nprod)
    want, _ = oracle.gemm_ex(0, 0, 1.5, A, B, 0.0, None, nprod=nprod)
    got = C.cpu().numpy()
    assert not np.any(np.isnan(got))
    if kind == "f64":
        np.testing.assert_array_equal(got.view(np.uint64), want.view(np.uint64))
    # K = 0: the product is zero, so C <- beta C
    C0 = synth.uniform_f64(66, 0, (33, 21)).astype(dt)
    Cz, _ = emu.gemm_ex(torch.zeros((33, 0), dtype=Cn.dtype, device=dev),
                        torch.zeros((0, 21), dtype=Cn.dtype, device=dev), 0, 0, 2.0, -0.5,
                        C=to_dev(C0, dev), nprod=nprod)
    np.testing.assert_array_equal(Cz.cpu().numpy(), (dt(2.0) * np.zeros_like(C0)) + dt(-0.5) * C0)
