"""FP64 mode with merged tail diagonals (emu_gemm_f64_merged) on the GPU,
through the C-ABI, against the oracle (oracle.gemm_f64_merged).

The head (products with i + j < L) is Algorithm 2 and must equal the
oracle's head bit for bit; the tail T is an FP32 tensor-core sum, read back
from the workspace.  So: (1) C == fl64(head_oracle + T_gpu) exactly, and
(2) |T_gpu - T_exact| <= steps * 2^-22 * S, where steps = (tail products) x
ceil(K / 16) is the number of accumulating MMA steps, each rounding to FP32
(at most 2^-23 relative, twice for the products' internal sum and the
accumulator), and S = sum over the tail of |A_i||B_j|.
"""
import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import device, sample_rows, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    return device()


def _tail_of(ws, M, N, K):
    off = emu.emu_gemm_workspace_bytes(64, M, N, K)
    return ws[off:off + 4 * M * N].view(emu._torch().float32).reshape(M, N).cpu().numpy()


def _check(A, B, C, ws, nprod, L, rows=None):
    M, K = A.shape
    N = B.shape[1]
    r0, r1 = (0, M) if rows is None else rows
    d = oracle.NPROD_TO_D[nprod]
    Ap, _, _ = oracle.split_f64(A)
    Bp, _, _ = oracle.split_f64(B)
    head = oracle.prodsum_f64(Ap, Bp, L * (L + 1) // 2, rows=(r0, r1))
    Cg = C[r0:r1]
    if L == d:
        assert np.array_equal(Cg, head)
        return
    Tg = _tail_of(ws, M, N, K)[r0:r1].astype(np.float64)
    assert np.array_equal(Cg, head + Tg)                     # head bit-exact, T added once
    _, T, S, _ = oracle.gemm_f64_merged(A, B, nprod, L, rows=(r0, r1))
    steps = len(oracle.tail_products(nprod, L)) * -(-K // 16)
    err = np.abs(Tg - T)
    bound = steps * 2.0**-22 * S
    assert np.all(err <= bound), float(np.max(err / np.maximum(bound, 1e-300)))


@pytest.mark.parametrize("nprod,L", [(21, 4), (21, 5), (15, 4), (21, 3), (10, 3), (15, 3)])
@pytest.mark.parametrize("M,N,K,seed", [
    (256, 256, 256, 1),
    (300, 333, 700, 2),      # ragged in every dimension
    (129, 257, 33, 3),       # one past a tile edge, K just past one K-block
    (1, 1, 1, 4),
])
def test_merged_parity(dev, nprod, L, M, N, K, seed):
    A, B = synth.gemm_inputs("f64", M, N, K, seed)
    C, ws = emu.gemm_f64_merged(to_dev(A, dev), to_dev(B, dev), nprod, L)
    assert emu.read_flags(ws) == 0
    _check(A, B, C.cpu().numpy(), ws, nprod, L)


@pytest.mark.parametrize("nprod", [6, 10, 15, 21])
def test_merged_without_tail_is_emu_gemm_f64(dev, nprod):
    A, B = synth.gemm_inputs("f64", 200, 300, 600, 7)
    d = oracle.NPROD_TO_D[nprod]
    Ad, Bd = to_dev(A, dev), to_dev(B, dev)
    C1, _ = emu.gemm_f64_merged(Ad, Bd, nprod, d)
    C2, _ = emu.gemm_f64(Ad, Bd, nprod)
    assert np.array_equal(C1.cpu().numpy(), C2.cpu().numpy())


@pytest.mark.parametrize("phi,seed", [(2.0, 4), (4.0, 5)])
def test_merged_scaled_class(dev, phi, seed):
    """The scaled input class: wide exponent ranges inside each operand."""
    A, B = synth.gemm_inputs("f64", 192, 160, 520, seed, phi=phi)
    C, ws = emu.gemm_f64_merged(to_dev(A, dev), to_dev(B, dev), 21, 4)
    assert emu.read_flags(ws) == 0
    _check(A, B, C.cpu().numpy(), ws, 21, 4)


def test_merged_argument_errors(dev):
    torch = emu._torch()
    A = torch.ones((8, 8), dtype=torch.float64, device=dev)
    ws = emu.workspace(emu.emu_gemm_f64_merged_workspace_bytes(8, 8, 8), dev)
    s = emu._stream(None)
    for nprod, L in [(21, 2), (21, 7), (10, 5), (7, 3)]:
        assert emu.emu_gemm_f64_merged(8, 8, 8, A.data_ptr(), 8, A.data_ptr(), 8, A.data_ptr(), 8, nprod, L,
                                       ws.data_ptr(), ws.numel(), s) == 1
    assert emu.emu_gemm_f64_merged(8, 8, 8, A.data_ptr(), 8, A.data_ptr(), 8, A.data_ptr(), 8, 21, 4,
                                   ws.data_ptr(), ws.numel() - 1, s) == 3


def test_merged_fullsize_n4096_sampled(dev):
    """4096^3, 21 products, tail from diagonal 4: sampled rows against the
    oracle; against the double-double reference its error lies between
    Algorithm 2's with 21 products (at most 4x it: the FP32 sum of the tail
    over K = 4096 about doubles e_F) and far below Algorithm 2's with 15."""
    n = 4096
    A, B = synth.gemm_inputs("f64", n, n, n, 1)
    Ad, Bd = to_dev(A, dev), to_dev(B, dev)
    C, ws = emu.gemm_f64_merged(Ad, Bd, 21, 4)
    assert emu.read_flags(ws) == 0
    C21, _ = emu.gemm_f64(Ad, Bd, 21)
    C15, _ = emu.gemm_f64(Ad, Bd, 15)
    rows = sample_rows(n, 2, 3)
    Cn, C21n, C15n = C.cpu().numpy(), C21.cpu().numpy(), C15.cpu().numpy()
    for r in rows:
        _check(A, B, Cn, ws, 21, 4, rows=(r, r + 1))
    hi, lo = oracle.ref_dd(np.ascontiguousarray(A[rows]), B)
    e_m = oracle.errors(Cn[rows], hi, lo)["e_F"]
    e_21 = oracle.errors(C21n[rows], hi, lo)["e_F"]
    e_15 = oracle.errors(C15n[rows], hi, lo)["e_F"]
    assert e_m <= 4 * e_21 and e_m <= 0.05 * e_15, (e_m, e_21, e_15)
