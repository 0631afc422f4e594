"""The C-ABI library loads without a GPU, exports every entry point that
include/emu.h declares, and rejects bad arguments on the host before any
CUDA call."""
import ctypes
import os
import re

import pytest

import paper_2609_04663_gb300 as emu
from paper_2609_04663_gb300 import _build

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "emu.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(emu_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return emu.load()


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("emu_split_f32", "emu_split_f64", "emu_gemm_f32", "emu_gemm_f64",
                     "emu_prodsum_f32", "emu_prodsum_f64", "emu_read_flags"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert name in emu._SIGS, f"binding lacks {name}"


def test_library_is_built_for_sm103a_only():
    assert "arch=compute_103a,code=sm_103a" in " ".join(_build.ARCH)


def test_status_strings_and_sizes(lib):
    assert emu.emu_status_string(0) == b"ok"
    assert emu.emu_status_string(3) == b"workspace too small"
    assert emu.emu_split_workspace_bytes(64) >= 256
    M, N, K = 300, 200, 700
    ldk = emu.gemm_ldk(K)
    assert ldk == 704
    need = emu.emu_gemm_workspace_bytes(64, M, N, K)
    assert need >= 6 * (M + N) * ldk * 2
    assert emu.emu_gemm_workspace_bytes(32, M, N, K) < need


def test_host_argument_checks_need_no_gpu(lib):
    # every call below fails validation before touching CUDA
    P = 16  # a dummy, 16-byte aligned, never dereferenced
    assert emu.emu_gemm_f32(-1, 4, 4, P, 4, P, 4, P, 4, P, 1 << 20, None) == 1
    assert emu.emu_gemm_f32(4, 4, 4, P, 3, P, 4, P, 4, P, 1 << 20, None) == 1       # lda < K
    assert emu.emu_gemm_f64(4, 4, 4, P, 4, P, 4, P, 4, 7, P, 1 << 20, None) == 1    # nprod
    assert emu.emu_gemm_f64(4, 4, 4, P, 4, P, 4, P, 4, 6, P, 16, None) == 3         # workspace
    assert emu.emu_gemm_f32(1 << 31, 4, 4, P, 4, P, 4, P, 4, P, 1 << 62, None) == 5  # size limit
    assert emu.emu_split_f64(P, 4, 4, 2, 0, P, 4, P, P, 4096, None) == 1              # ldx < cols
    assert emu.emu_selftest_timeout(P, 4096, 0, None) == 1
    assert emu.emu_split_f64_slices(P, 4, 4, 4, 0, P, 4, 2, P, P, 4096, None) == 1      # nslices < 3
    assert emu.emu_split_f64_slices(P, 4, 4, 4, 0, P, 4, 7, P, P, 4096, None) == 1      # nslices > 6
    assert emu.emu_split_f64_slices(P, 4, 4, 4, 0, P, 4, 4, P, P, 16, None) == 3        # workspace
    # merged FP64 tail: merge_from range and workspace size are checked on the host
    assert emu.emu_gemm_f64_merged(4, 4, 4, P, 4, P, 4, P, 4, 21, 2, P, 1 << 30, None) == 1
    assert emu.emu_gemm_f64_merged(4, 4, 4, P, 4, P, 4, P, 4, 10, 5, P, 1 << 30, None) == 1
    assert emu.emu_gemm_f64_merged(4, 4, 4, P, 4, P, 4, P, 4, 21, 4, P, 16, None) == 3
    assert emu.emu_gemm_f64_merged_workspace_bytes(300, 200, 700) == \
        emu.emu_gemm_workspace_bytes(64, 300, 200, 700) + 300 * 200 * 4 + 128
    # the fused FP32 GEMM needs only the flag word
    assert emu.emu_gemm_f32_fused(4, 4, 4, P, 3, P, 4, P, 4, P, 512, None) == 1       # lda < K
    assert emu.emu_gemm_f32_fused(4, 4, 4, P, 4, P, 4, P, 4, P, 511, None) == 3       # workspace
    assert emu.emu_gemm_f32_fused(4, 4, 4, P, 4, P, 4, P, 4, P + 8, 512, None) == 2   # ws alignment
    assert emu.emu_gemm_f32_fused(4, 4, 4, 0, 4, P, 4, P, 4, P, 512, None) == 1       # null A
    # host-buffer GEMMs: validation precedes every CUDA call
    W = 256  # 256-byte aligned dummy workspace address
    assert emu.emu_gemm_f32_host(4, 4, 4, P, 3, P, 4, P, 4, W, 1 << 40, None) == 1      # lda < K
    assert emu.emu_gemm_f64_host(4, 4, 4, P, 4, P, 4, P, 4, 5, W, 1 << 40, None) == 1   # nprod
    assert emu.emu_gemm_f32_host(4, 4, 4, P, 4, P, 4, P, 4, P, 1 << 40, None) == 2      # ws not 256-aligned
    assert emu.emu_gemm_f32_host(4, 4, 4, P, 4, P, 4, P, 4, W, 64, None) == 3           # workspace
    assert emu.emu_gemm_f64_host(4, 4, 4, 0, 4, P, 4, P, 4, 6, W, 1 << 40, None) == 1   # null A


def test_host_workspace_sizes(lib):
    M, N, K = 300, 200, 700
    for mode in (32, 64):
        need = emu.emu_gemm_host_workspace_bytes(mode, M, N, K)
        assert need > emu.emu_gemm_workspace_bytes(mode, M, N, K)
    assert emu.emu_gemm_host_workspace_bytes(16, M, N, K) == 0
    assert emu.emu_gemm_host_workspace_bytes(32, -1, N, K) == 0
    # FP64 stages both operands whole: at least 8 (MK + KN) bytes beyond the planes
    assert emu.emu_gemm_host_workspace_bytes(64, M, N, K) >= emu.emu_gemm_workspace_bytes(64, M, N, K) + 8 * (M * K + K * N)


def test_gemm_ex_argument_checks_need_no_gpu(lib):
    P = 16
    big = 1 << 40
    assert emu.emu_gemm_ex_f32(2, 0, 4, 4, 4, 1.0, P, 4, P, 4, 0.0, P, 4, P, big, None) == 1   # op
    assert emu.emu_gemm_ex_f32(1, 0, 4, 4, 8, 1.0, P, 3, P, 4, 0.0, P, 4, P, big, None) == 1   # op(A) = T: lda >= M
    assert emu.emu_gemm_ex_f32(0, 1, 4, 5, 8, 1.0, P, 8, P, 7, 0.0, P, 5, P, big, None) == 1   # op(B) = T: ldb >= K
    assert emu.emu_gemm_ex_f64(0, 0, 4, 4, 4, 1.0, P, 4, P, 4, 0.0, P, 4, 7, P, big, None) == 1  # nprod
    assert emu.emu_gemm_ex_f64(0, 0, 4, 4, 4, 1.0, P, 4, P, 4, 0.0, P, 4, 6, P, 64, None) == 3   # workspace
    assert emu.emu_gemm_ex_workspace_bytes(32, 10, 20, 30) == (
        emu.emu_gemm_workspace_bytes(32, 10, 20, 30) + (10 * 20 * 4 + 255) // 256 * 256)
    assert emu.emu_gemm_ex_workspace_bytes(48, 10, 20, 30) == 0



def test_prodsum_workspace_sizes_and_check(lib):
    assert emu.emu_prodsum_workspace_bytes(32, 300, 200) == emu.emu_split_workspace_bytes(32)
    # FP64: the header plus one 128 x 128 FP64 accumulator tile per CTA tile
    assert emu.emu_prodsum_workspace_bytes(64, 300, 200) == emu.emu_split_workspace_bytes(64) + 3 * 2 * 128 * 128 * 8
    assert emu.emu_prodsum_workspace_bytes(64, -1, 2) == 0
    P = 16
    small = emu.emu_split_workspace_bytes(64)
    assert emu.emu_prodsum_f64(300, 200, 64, P, P, 64, P, P, 6, P, 200, P, small, None) == 3


def test_rowcol_argument_checks_need_no_gpu(lib):
    P = 16
    # header plus 28 bytes per plane row (literal maxima, speculative maxima, fix marks), 256-byte rounded
    assert emu.emu_split_f64_rowcol_workspace_bytes(100) == emu.emu_split_workspace_bytes(64) + 2816
    assert emu.emu_split_f64_rowcol(P, 100, 8, 8, 0, P, 8, P, P, 600, None) == 3           # workspace
    assert emu.emu_split_f64_rowcol(P, 100, 8, 8, 0, P, 8, 0, P, 1 << 20, None) == 1       # no v_out
    need = emu.emu_gemm_f64_rowcol_workspace_bytes(300, 200, 700)
    assert need > emu.emu_gemm_workspace_bytes(64, 300, 200, 700)
    assert emu.emu_gemm_f64_rowcol(300, 200, 700, P, 700, P, 200, P, 200, 6, P, need - 1, None) == 3
    assert emu.emu_gemm_f64_rowcol(4, 4, 4, P, 4, P, 4, P, 4, 11, P, 1 << 30, None) == 1      # nprod


def test_f64_tile_width_report(lib):
    # no GPU here: the launcher assumes 152 SMs; with EMU_F64_TILE unset a
    # large square result takes the 128 x 256 tile, a small one 128 x 128
    if os.environ.get("EMU_F64_TILE"):
        pytest.skip("EMU_F64_TILE forces a tile width")
    assert emu.emu_prodsum_f64_tile_columns(8192, 8192) == 256
    assert emu.emu_prodsum_f64_tile_columns(1024, 1024) == 128
    assert emu.emu_prodsum_f64_tile_columns(0, 8) == 0
    # 256-column tiles run on CTA pairs (256 rows) when there are two tile rows
    assert emu.emu_prodsum_f64_tile_rows(8192, 8192) == 256
    assert emu.emu_prodsum_f64_tile_rows(1024, 1024) == 128
    assert emu.emu_prodsum_f64_tile_rows(128, 65536) == 128
    assert emu.emu_prodsum_f64_tile_rows(8, 0) == 0
    # 8192^2: 1024 pair tiles on 76 pairs, 13.5 waves, one launch; 4096^2:
    # 256 pair tiles, 3.4 waves, the last 28 tiles as 112 128 x 128 tiles
    assert emu.emu_prodsum_f64_launches(8192, 8192) == 1
    assert emu.emu_prodsum_f64_launches(4096, 4096) == 2
    assert emu.emu_prodsum_f64_launches(1024, 1024) == 1
    assert emu.emu_prodsum_f64_launches(0, 1) == 0


def test_f32_launch_report(lib):
    # no GPU here: the launcher assumes 152 SMs (76 pairs per wave)
    if os.environ.get("EMU_F32_TILE") or os.environ.get("EMU_F32_PAIR"):
        pytest.skip("EMU_F32_TILE / EMU_F32_PAIR force a schedule")
    # 4096^2: 256 pair tiles, 3.4 waves, the last 28 as 112 128 x 128 quarters;
    # 8192^2: 1024 pair tiles, 13.5 waves, the last 36 as 144 quarters;
    # 16384^2: 53.9 waves, the last 68 pair tiles would need 272 quarters
    assert emu.emu_prodsum_f32_launches(4096, 4096) == 2
    assert emu.emu_prodsum_f32_launches(8192, 8192) == 2
    assert emu.emu_prodsum_f32_launches(16384, 16384) == 1
    assert emu.emu_prodsum_f32_launches(1024, 1024) == 1
    assert emu.emu_prodsum_f32_launches(0, 5) == 0
    # 256-column tiles, on CTA pairs where there are two tile rows
    assert emu.emu_prodsum_f32_tile_columns(16384, 16384) == 256
    assert emu.emu_prodsum_f32_tile_rows(16384, 16384) == 256
    assert emu.emu_prodsum_f32_tile_rows(128, 65536) == 128
    assert emu.emu_prodsum_f32_tile_columns(1024, 1024) in (64, 128)
    assert emu.emu_prodsum_f32_tile_rows(1024, 1024) == 128
    assert emu.emu_prodsum_f32_tile_rows(0, 4) == 0


def test_f32_schedule_rule(lib):
    """The FP32 schedule over a range of result sizes (152 SMs assumed, as
    without a GPU): a second launch of 128 x 128 quarters exactly when the
    pair tiles leave a partial last wave after at least one full one, its
    tiles fit one wave as quarters (4 per pair tile), and that is estimated
    at least 2 % faster (a quarter wave costs 0.5 / 0.85 of a pair wave)."""
    if os.environ.get("EMU_F32_TILE") or os.environ.get("EMU_F32_PAIR"):
        pytest.skip("EMU_F32_TILE / EMU_F32_PAIR force a schedule")
    seen = set()
    for M in (256, 1000, 2048, 3000, 4096, 5120, 6144, 8192, 10240, 12288, 16384):
        for N in (512, 2048, 4096, 8192, 12288, 16384):
            cols, rows = emu.emu_prodsum_f32_tile_columns(M, N), emu.emu_prodsum_f32_tile_rows(M, N)
            launches = emu.emu_prodsum_f32_launches(M, N)
            assert cols in (64, 128, 256) and rows in (128, 256) and launches in (1, 2)
            if rows == 256:
                assert cols == 256 and M > 128
            pairs = ((M + 127) // 128 + 1) // 2 * ((N + 255) // 256)
            full, left = divmod(pairs, 76)
            mixed = rows == 256 and full >= 1 and 0 < left and 4 * left <= 152 and \
                full + 0.5 / 0.85 <= 0.98 * (full + 1)
            assert launches == (2 if mixed else 1), (M, N, pairs)
            seen.add(launches)
    assert seen == {1, 2}

