"""Oracle pins of the merged-tail FP64 variant (an extension: the products
with merge_from <= i + j < d summed into one tail T, added once after the
Algorithm 2 head).  CPU only.

The oracle's T is the exact tail sum.  Pinned against exact rational
arithmetic on small cases, and against Algorithm 2 itself where the two must
coincide."""
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth


def _frac_slices(planes, r):
    return [[Fraction(float(x)) for x in row] for row in oracle.bf16_to_f32(planes[r]).astype(np.float64)]


def _exact_sum(Ap, Bp, prods, m, n):
    """Exact rational sum over the products (i, j) of sum_k A_i[m, k] B_j[k, n]."""
    K = Ap.shape[2]
    a = {i: oracle.bf16_to_f32(Ap[i, m]).astype(np.float64) for i, _ in prods}
    b = {j: oracle.bf16_to_f32(Bp[j, :, n]).astype(np.float64) for _, j in prods}
    return sum(Fraction(float(a[i][k])) * Fraction(float(b[j][k])) for i, j in prods for k in range(K))


def test_tail_product_sets():
    """The tail is S_d minus the Algorithm 2 head, in diagonal order:
    d(d+1)/2 - L(L+1)/2 products."""
    for nprod, d in oracle.NPROD_TO_D.items():
        full = oracle.products(64, nprod)
        for L in range(1, d + 1):
            tail = oracle.tail_products(nprod, L)
            assert len(tail) == d * (d + 1) // 2 - L * (L + 1) // 2
            assert tail == full[L * (L + 1) // 2:]
            assert all(L <= i + j < d for i, j in tail)
    assert oracle.tail_products(21, 4) == [(0, 4), (1, 3), (2, 2), (3, 1), (4, 0),
                                           (0, 5), (1, 4), (2, 3), (3, 2), (4, 1), (5, 0)]


@pytest.mark.parametrize("nprod", [6, 10, 15, 21])
def test_no_tail_is_algorithm_2(nprod):
    A, B = synth.gemm_inputs("f64", 40, 30, 300, 5)
    d = oracle.NPROD_TO_D[nprod]
    C, T, S, _ = oracle.gemm_f64_merged(A, B, nprod, d)
    assert not T.any() and not S.any()
    assert np.array_equal(C, oracle.gemm_f64(A, B, nprod)[0])


@pytest.mark.parametrize("nprod,L", [(21, 4), (21, 5), (15, 4), (21, 3)])
def test_tail_is_the_exact_rational_sum(nprod, L):
    """T against exact rationals over two K-chunks; and head + tail products
    together are S_d exactly (no product dropped or counted twice)."""
    M, N, K = 3, 4, 300
    A, B = synth.gemm_inputs("f64", M, N, K, 9)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    C, T, S, _ = oracle.gemm_f64_merged(A, B, nprod, L)
    tail = oracle.tail_products(nprod, L)
    head = oracle.products(64, nprod)[: L * (L + 1) // 2]
    full = oracle.products(64, nprod)
    for m in range(M):
        for n in range(N):
            t = _exact_sum(Ap, Bp, tail, m, n)
            assert Fraction(float(T[m, n])) == t            # needs < 53 bits here, so exact
            assert _exact_sum(Ap, Bp, head, m, n) + t == _exact_sum(Ap, Bp, full, m, n)
            s = sum(abs(Fraction(float(x))) * abs(Fraction(float(y)))
                    for i, j in tail
                    for x, y in zip(oracle.bf16_to_f32(Ap[i, m]).astype(np.float64),
                                    oracle.bf16_to_f32(Bp[j, :, n]).astype(np.float64)))
            assert abs(Fraction(float(S[m, n])) - s) <= s * Fraction(1, 2**40)


def test_head_plus_exact_tail_rounds_once():
    """C = fl64(C_head + T): the head is Algorithm 2 over the first
    L(L+1)/2 products, and T enters with a single rounding."""
    A, B = synth.gemm_inputs("f64", 20, 24, 700, 12)
    C, T, _, _ = oracle.gemm_f64_merged(A, B, 21, 4)
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    head = oracle.prodsum_f64(Ap, Bp, 10)
    assert np.array_equal(C, head + T)
    # and it differs from Algorithm 2's eleven separate additions by rounding only
    C21 = oracle.gemm_f64(A, B, 21)[0]
    assert np.all(np.abs(C - C21) <= 16 * np.spacing(np.abs(C21)))


def test_merged_accuracy_matches_algorithm_2():
    """With the tail exact, the merged result is as accurate as Algorithm 2
    against the double-double reference (uniform [-1, 1], N = 128)."""
    n = 128
    A, B = synth.gemm_inputs("f64", n, n, n, 1)
    hi, lo = oracle.ref_dd(A, B)
    e_alg2 = oracle.errors(oracle.gemm_f64(A, B, 21)[0], hi, lo)["e_F"]
    e_merged = oracle.errors(oracle.gemm_f64_merged(A, B, 21, 4)[0], hi, lo)["e_F"]
    assert 0.5 * e_alg2 <= e_merged <= 1.5 * e_alg2
