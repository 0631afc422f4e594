"""The cancellation-sensitive input class (Section 7.3 names it; synth
defines it as A = [P | P], B = [Q ; -Q + 2^-20 R]): its structure, and the
oracle's emulated products on it against a double-double reference.  Every
dot product cancels two halves about 2^20 times larger than the result, so
the errors are measured against |A||B| (Eq. (scalederror))."""
import numpy as np

import oracle
import synth


def test_cancel_structure():
    A, B = synth.gemm_inputs("f64_cancel", 6, 5, 40, 3)
    assert np.array_equal(A[:, :20], A[:, 20:])
    R = (B[20:] + B[:20]) * 2.0 ** 20
    assert np.all(np.abs(R) <= 1.0 + 1e-9) and np.any(R != 0)
    A3, B3 = synth.gemm_inputs("f32_cancel", 4, 3, 41, 3)                      # odd K: one extra pair
    assert A3.shape == (4, 41) and B3.shape == (41, 3) and A3.dtype == np.float32


def test_cancel_class_errors_stay_at_the_scaled_bar():
    M, N, K = 20, 16, 512
    for kind, bound in (("f32_cancel", 1e-5), ("f64_cancel", None)):
        A, B = synth.gemm_inputs(kind, M, N, K, 9)
        A64, B64 = A.astype(np.float64), B.astype(np.float64)
        hi, lo = oracle.ref_dd(A64, B64)
        absab = np.abs(A64) @ np.abs(B64)
        # the result is tiny against |A||B|: the class really cancels
        assert np.max(np.abs(hi) / absab) < 2.0 ** -17
        if kind == "f32_cancel":
            C, _ = oracle.gemm_f32(A, B)
            assert oracle.errors(C, hi, lo, absab)["e_scaled"] < bound
        else:
            e = [oracle.errors(oracle.gemm_f64(A, B, n)[0], hi, lo, absab)["e_scaled"] for n in (6, 10, 21)]
            assert e[0] > e[1] > e[2] and e[2] < 1e-14, e
