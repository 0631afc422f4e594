"""FP32-mode GEMM with the split inside the product-sum (emu_gemm_f32_fused)
on the GPU, through the C-ABI.

It forms the same slices (Eq. (fp32split)) and issues the same MMAs in the
same order into the same accumulator as the split + product-sum pair, so C
must equal split + product-sum bit for bit (all of K in one accumulator;
emu_gemm_f32 may split K for small results), and the oracle within the FP32-mode bar
|C - C_oracle| <= 1e-5 (|A||B|).  Its loads take several paths (16-byte
vectors, scalars for ragged or unaligned rows, zeros past the edges), so the
cases cover each of them.
"""
import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import device, fp32_within_tolerance, gemm_f32_one_accumulator, random_finite_f32, sample_rows, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def _both(A_d, B_d):
    C2, f2 = gemm_f32_one_accumulator(A_d, B_d)
    C1, ws1 = emu.gemm_f32_fused(A_d, B_d)
    return C1, emu.read_flags(ws1), C2, f2


@pytest.mark.parametrize("M,N,K,seed", [
    (256, 256, 256, 0),
    (300, 333, 700, 1),      # ragged in every dimension
    (37, 200, 513, 2),       # one partial row tile, K tail of 1 element
    (129, 257, 33, 3),       # one past a tile edge in M and N, K just past one K-block
    (1, 1, 1, 4),
    (128, 512, 64, 5),
    (200, 700, 30, 6),       # K below one K-block, K % 4 != 0
    (513, 1000, 1027, 7),    # several tiles, K % 4 == 3
])
def test_fused_parity_and_bit_identity(dev, M, N, K, seed):
    A, B = synth.gemm_inputs("f32", M, N, K, seed)
    C1, f1, C2, f2 = _both(to_dev(A, dev), to_dev(B, dev))
    assert f1 == 0 and f2 == 0
    C1 = C1.cpu().numpy()
    assert np.array_equal(C1.view(np.uint32), C2.cpu().numpy().view(np.uint32))
    Co, _ = oracle.gemm_f32(A, B)
    ok, worst = fp32_within_tolerance(C1, Co, A, B)
    assert ok, worst


@pytest.mark.parametrize("pad_a,pad_b,offset_a", [(4, 9, 0), (1, 3, 0), (0, 0, 1), (3, 1, 1)])
def test_fused_strided_and_unaligned(dev, pad_a, pad_b, offset_a):
    """Odd leading dimensions and an A that starts 4 bytes past a 16-byte
    boundary take the scalar loads; C is written through a strided view."""
    torch = emu._torch()
    M, N, K = 190, 300, 301
    A, B = synth.gemm_inputs("f32", M, N, K, 11)
    Ad = to_dev(A if not offset_a else np.hstack([np.zeros((M, 1), np.float32), A]), dev, ld_pad=pad_a)
    if offset_a:
        Ad = Ad[:, 1:]
    Bd = to_dev(B, dev, ld_pad=pad_b)
    Cbig = torch.zeros((M, N + 5), dtype=torch.float32, device=dev)
    C = Cbig[:, :N]
    _, ws = emu.gemm_f32_fused(Ad, Bd, C=C)
    assert emu.read_flags(ws) == 0
    C2, _ = gemm_f32_one_accumulator(to_dev(A, dev), to_dev(B, dev))
    assert np.array_equal(C.cpu().numpy().view(np.uint32), C2.cpu().numpy().view(np.uint32))
    assert not Cbig[:, N:].any()


def test_fused_wide_exponent_range(dev):
    """Zeros, subnormals and normals over 2^-126 .. 2^34: every slice path of
    Eq. (fp32split), against the split kernels' slices, bit for bit."""
    A = random_finite_f32((160, 300), 21, emax_field=160)
    B = random_finite_f32((300, 270), 22, emax_field=160)
    C1, f1, C2, f2 = _both(to_dev(A, dev), to_dev(B, dev))
    assert f1 == f2 == 0
    assert np.array_equal(C1.cpu().numpy().view(np.uint32), C2.cpu().numpy().view(np.uint32))


def test_fused_exact_integers(dev):
    rng = np.random.default_rng(4)
    A = rng.integers(-12, 13, size=(160, 700)).astype(np.float32)
    B = rng.integers(-12, 13, size=(700, 300)).astype(np.float32)
    C, _ = emu.gemm_f32_fused(to_dev(A, dev), to_dev(B, dev))
    assert np.array_equal(C.cpu().numpy().astype(np.int64), A.astype(np.int64) @ B.astype(np.int64))


def test_fused_domain_flags(dev):
    """Non-finite inputs and a slice that overflows BF16 raise the same flags
    as the split kernels, wherever the element sits (A or B, edge tiles)."""
    M, N, K = 130, 260, 70
    for where, val, flag in [("A", np.inf, emu.FLAG_NONFINITE), ("B", np.nan, emu.FLAG_NONFINITE),
                             ("B", np.float32(3.4e38), emu.FLAG_SLICE)]:
        A, B = synth.gemm_inputs("f32", M, N, K, 3)
        if where == "A":
            A[M - 1, K - 1] = val
        else:
            B[K - 1, N - 1] = val
        _, f1, _, f2 = _both(to_dev(A, dev), to_dev(B, dev))
        assert f1 == f2 and f1 & flag, (where, f1, f2)


def test_fused_zero_sizes_and_empty_k(dev):
    torch = emu._torch()
    C = torch.full((5, 7), 3.0, dtype=torch.float32, device=dev)
    emu.gemm_f32_fused(torch.ones((5, 0), device=dev), torch.ones((0, 7), device=dev), C=C)
    assert not C.any()
    Cm = torch.full((0, 7), 3.0, dtype=torch.float32, device=dev)
    emu.gemm_f32_fused(torch.ones((0, 4), device=dev), torch.ones((4, 7), device=dev), C=Cm)


def test_fused_fullsize_fp32_n16384_sampled(dev):
    """At the full FP32 sweep size: sampled rows against the oracle, and the
    whole C against the split + product-sum pair."""
    n = 16384
    A, B = synth.gemm_inputs("f32", n, n, n, n)
    Ad, Bd = to_dev(A, dev), to_dev(B, dev)
    C1, ws = emu.gemm_f32_fused(Ad, Bd)
    assert emu.read_flags(ws) == 0
    C2, _ = gemm_f32_one_accumulator(Ad, Bd)
    assert bool((C1.view(emu._torch().int32) == C2.view(emu._torch().int32)).all())
    del C2
    rows = sample_rows(n, 3, 1)
    Cg = C1.cpu().numpy()[rows]
    Co = oracle.prodsum_f32(oracle.split_f32(A[rows])[0], oracle.split_f32(B)[0])
    ok, worst = fp32_within_tolerance(Cg, Co, A[rows], B)
    assert ok, worst
