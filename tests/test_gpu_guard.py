"""Guard bands: the library writes only what it owns.

There is no sanitizer on this pool, so every buffer the C-ABI calls touch is
surrounded by canaries -- padding columns and rows past the end of C, the
padding of the component planes (ldcomp > cols) and a band after the last
plane, and a band after the workspace -- and the canaries must be intact
after the call.  Inputs (with their own padding) must come back unchanged.
The results inside the bands are checked against the oracle as well, so a
kernel that wrote its output one row or column off would fail twice."""
import numpy as np
import pytest

import oracle
import synth
import paper_2609_04663_gb300 as emu
from helpers import device, fp32_within_tolerance, sample_rows

pytestmark = pytest.mark.gpu

CANARY32 = 0x7FA5A5A5                 # a NaN bit pattern
CANARY64 = 0x7FF5A5A5A5A5A5A5
CANARY16 = 0x5A5A
CANARY8 = 0xA5
BAND = 4096


def _torch():
    import torch
    return torch


def _padded(host, dev, pad_cols, pad_rows, canary):
    """Device copy of a 2-D host array inside a larger canary-filled buffer:
    returns (view of the live part, the whole buffer)."""
    torch = _torch()
    rows, cols = host.shape
    itype = torch.int32 if host.dtype == np.float32 else torch.int64
    ftype = torch.float32 if host.dtype == np.float32 else torch.float64
    big = torch.full((rows + pad_rows, cols + pad_cols), canary, dtype=itype, device=dev)
    bigf = big.view(ftype)
    bigf[:rows, :cols] = torch.from_numpy(np.ascontiguousarray(host)).to(dev)
    return bigf[:rows, :cols], big


def _outside_intact(big, rows, cols, canary):
    b = big.cpu().numpy()
    mask = np.ones(b.shape, dtype=bool)
    mask[:rows, :cols] = False
    return bool(np.all(b[mask] == np.array(canary, dtype=b.dtype)))


def _ws(nbytes, dev):
    torch = _torch()
    buf = torch.full((nbytes + BAND,), CANARY8, dtype=torch.uint8, device=dev)
    return buf


def _band_intact(buf, nbytes):
    return bool(np.all(buf[nbytes:].cpu().numpy() == CANARY8))


@pytest.mark.parametrize("M,N,K,cpad", [(300, 333, 700, 7), (129, 257, 33, 7), (300, 336, 700, 8), (1000, 1024, 512, 4),
                                        (4000, 1000, 64, 4)])
def test_gemm_f32_guard_bands(M, N, K, cpad):
    """cpad: padding columns of C.  From the third shape on N and the row
    pitch of C are multiples of 4, so the product-sum writes C by bulk tensor
    copies: the few-tile results split K and add their K-parts into C by
    bulk tensor reductions; the last one (4000 rows: the second CTA of the
    last pair holds 32 of them) runs 256 x 256 tiles on CTA pairs."""
    dev = device()
    torch = _torch()
    A, B = synth.gemm_inputs("f32", M, N, K, 21)
    Ad, Abig = _padded(A, dev, 5, 2, CANARY32)
    Bd, Bbig = _padded(B, dev, 3, 1, CANARY32)
    Abefore, Bbefore = Abig.clone(), Bbig.clone()
    Cbig = torch.full((M + 3, N + cpad), CANARY32, dtype=torch.int32, device=dev)
    C = Cbig.view(torch.float32)
    need = emu.emu_gemm_workspace_bytes(32, M, N, K)
    ws = _ws(need, dev)
    st = emu.emu_gemm_f32(M, N, K, Ad.data_ptr(), Ad.stride(0), Bd.data_ptr(), Bd.stride(0), C.data_ptr(),
                          C.stride(0), ws.data_ptr(), need, emu._stream(None))
    assert st == 0
    torch.cuda.synchronize()
    assert emu.read_flags(ws) == 0
    assert _outside_intact(Cbig, M, N, CANARY32)
    assert _band_intact(ws, need)
    assert torch.equal(Abig, Abefore) and torch.equal(Bbig, Bbefore)
    ok, worst = fp32_within_tolerance(C[:M, :N].cpu().numpy(), oracle.gemm_f32(A, B)[0], A, B)
    assert ok, worst


@pytest.mark.parametrize("M,N,K,nprod,cpad", [(300, 333, 700, 21, 7), (129, 257, 520, 6, 7), (3000, 3000, 300, 21, 7),
                                               (3000, 3000, 300, 6, 8)])
def test_gemm_f64_guard_bands(M, N, K, nprod, cpad):
    """cpad: padding columns of C.  In the last shape N and the row pitch of C
    are even, so the product-sum on 256-column tiles writes C by bulk tensor
    stores."""
    dev = device()
    torch = _torch()
    A, B = synth.gemm_inputs("f64", M, N, K, 22)
    Ad, Abig = _padded(A, dev, 5, 2, CANARY64)
    Bd, Bbig = _padded(B, dev, 3, 1, CANARY64)
    Abefore, Bbefore = Abig.clone(), Bbig.clone()
    Cbig = torch.full((M + 3, N + cpad), CANARY64, dtype=torch.int64, device=dev)
    C = Cbig.view(torch.float64)
    need = emu.emu_gemm_workspace_bytes(64, M, N, K)
    ws = _ws(need, dev)
    st = emu.emu_gemm_f64(M, N, K, Ad.data_ptr(), Ad.stride(0), Bd.data_ptr(), Bd.stride(0), C.data_ptr(),
                          C.stride(0), nprod, ws.data_ptr(), need, emu._stream(None))
    assert st == 0
    torch.cuda.synchronize()
    assert emu.read_flags(ws) == 0
    assert _outside_intact(Cbig, M, N, CANARY64)
    assert _band_intact(ws, need)
    assert torch.equal(Abig, Abefore) and torch.equal(Bbig, Bbefore)
    Cn = C[:M, :N].cpu().numpy()
    if M * N * K * nprod <= 4e9:
        assert np.array_equal(Cn, oracle.gemm_f64(A, B, nprod)[0])
    else:
        # 256 x 256 tiles on CTA pairs at a ragged size: sampled rows against the oracle
        assert emu.emu_prodsum_f64_tile_columns(M, N) == 256 and emu.emu_prodsum_f64_tile_rows(M, N) == 256
        for r in sample_rows(M, 4, 5):
            assert np.array_equal(Cn[r], oracle.gemm_f64(A, B, nprod, rows=(r, r + 1))[0][0]), r


@pytest.mark.parametrize("mode,transpose", [(32, 0), (32, 1), (64, 0), (64, 1)])
def test_split_plane_padding_and_band(mode, transpose):
    dev = device()
    torch = _torch()
    rows, cols = 131, 77
    rng = np.random.default_rng(24)
    X = (rng.random((rows, cols)) * 2 - 1).astype(np.float32 if mode == 32 else np.float64)
    Xd, _ = _padded(X, dev, 3, 0, CANARY32 if mode == 32 else CANARY64)
    s = 3 if mode == 32 else 6
    rows_out, cols_out = (cols, rows) if transpose else (rows, cols)
    ldcomp = (cols_out + 7) // 8 * 8 + 24
    plane = rows_out * ldcomp
    planes = torch.full((s * plane + BAND // 2,), CANARY16, dtype=torch.int16, device=dev)
    need = emu.emu_split_workspace_bytes(mode)
    ws = _ws(need, dev)
    if mode == 32:
        st = emu.emu_split_f32(Xd.data_ptr(), rows, cols, Xd.stride(0), transpose, planes.data_ptr(), ldcomp,
                               ws.data_ptr(), need, emu._stream(None))
    else:
        v = torch.empty(6, dtype=torch.int32, device=dev)
        st = emu.emu_split_f64(Xd.data_ptr(), rows, cols, Xd.stride(0), transpose, planes.data_ptr(), ldcomp,
                               v.data_ptr(), ws.data_ptr(), need, emu._stream(None))
    assert st == 0
    torch.cuda.synchronize()
    assert emu.read_flags(ws) == 0
    p = planes.cpu().numpy().view(np.uint16)
    assert np.all(p[s * plane:] == CANARY16)                            # band after the last plane
    body = p[: s * plane].reshape(s, rows_out, ldcomp)
    assert np.all(body[:, :, cols_out:] == CANARY16)                    # padding columns of every plane
    assert _band_intact(ws, need)
    ref = oracle.split_f32(X if not transpose else np.ascontiguousarray(X.T))[0] if mode == 32 else \
        oracle.split_f64(X if not transpose else np.ascontiguousarray(X.T))[0]
    assert np.array_equal(body[:, :, :cols_out], ref.view(np.uint16))


def test_prodsum_guard_bands():
    dev = device()
    torch = _torch()
    M, N, K = 200, 300, 520
    for mode in (32, 64):
        A, B = synth.gemm_inputs("f32" if mode == 32 else "f64", M, N, K, 25)
        Ad, Bd = torch.from_numpy(A).to(dev), torch.from_numpy(B).to(dev)
        if mode == 32:
            Ap, _ = emu.split_f32(Ad)
            Bp, _ = emu.split_f32(Bd, transpose=True, ldcomp=Ap.shape[2])
        else:
            Ap, vA, _ = emu.split_f64(Ad)
            Bp, vB, _ = emu.split_f64(Bd, transpose=True, ldcomp=Ap.shape[2])
        canary = CANARY32 if mode == 32 else CANARY64
        Cbig = torch.full((M + 2, N + 5), canary, dtype=torch.int32 if mode == 32 else torch.int64, device=dev)
        C = Cbig.view(torch.float32 if mode == 32 else torch.float64)
        need = emu.emu_prodsum_workspace_bytes(mode, M, N)
        ws = _ws(need, dev)
        if mode == 32:
            st = emu.emu_prodsum_f32(M, N, K, Ap.data_ptr(), Bp.data_ptr(), Ap.shape[2], C.data_ptr(), C.stride(0),
                                     ws.data_ptr(), need, emu._stream(None))
        else:
            st = emu.emu_prodsum_f64(M, N, K, Ap.data_ptr(), Bp.data_ptr(), Ap.shape[2], vA.data_ptr(),
                                     vB.data_ptr(), 21, C.data_ptr(), C.stride(0), ws.data_ptr(), need,
                                     emu._stream(None))
        assert st == 0
        torch.cuda.synchronize()
        assert emu.read_flags(ws) == 0
        assert _outside_intact(Cbig, M, N, canary), mode
        assert _band_intact(ws, need), mode
        if mode == 64:
            assert np.array_equal(C[:M, :N].cpu().numpy(), oracle.gemm_f64(A, B, 21)[0])


def test_noalloc_and_host_gemm_guard_bands():
    dev = device()
    torch = _torch()
    M, N, K = 150, 270, 400
    A, B = synth.gemm_inputs("f64", M, N, K, 26)
    Ad, Abig = _padded(A, dev, 4, 0, CANARY64)
    Bd, Bbig = _padded(B, dev, 2, 0, CANARY64)
    Cbig = torch.full((M + 2, N + 6), CANARY64, dtype=torch.int64, device=dev)
    C = Cbig.view(torch.float64)
    flags = torch.zeros(1, dtype=torch.int32, device=dev)
    st = emu.emu_gemm_f64_noalloc(M, N, K, Ad.data_ptr(), Ad.stride(0), Bd.data_ptr(), Bd.stride(0), C.data_ptr(),
                                  C.stride(0), 10, flags.data_ptr(), emu._stream(None))
    assert st == 0
    torch.cuda.synchronize()
    assert int(flags.item()) == 0
    assert _outside_intact(Cbig, M, N, CANARY64)
    C_or = oracle.gemm_f64(A, B, 10)[0]
    assert np.array_equal(C[:M, :N].cpu().numpy(), C_or)
    # host buffers: pinned C with padding columns and rows
    Ah = torch.from_numpy(A).pin_memory()
    Bh = torch.from_numpy(B).pin_memory()
    Chbig = torch.full((M + 2, N + 6), CANARY64, dtype=torch.int64).pin_memory()
    Ch = Chbig.view(torch.float64)
    need = emu.emu_gemm_host_workspace_bytes(64, M, N, K)
    ws = _ws(need, dev)
    st = emu.emu_gemm_f64_host(M, N, K, Ah.data_ptr(), K, Bh.data_ptr(), N, Ch.data_ptr(), Ch.stride(0), 10,
                               ws.data_ptr(), need, emu._stream(None))
    assert st == 0
    torch.cuda.synchronize()
    assert _outside_intact(Chbig, M, N, CANARY64)
    assert _band_intact(ws, need)
    assert np.array_equal(Ch[:M, :N].numpy(), C_or)
