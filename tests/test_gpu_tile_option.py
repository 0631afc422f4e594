"""The product-sums' tile shapes. FP32 (EMU_F32_TILE=128x256 / 128x128 /
128x64 forces one; unset, the library picks by tile count; 128 x 256 tiles
run as 256 x 256 tiles on CTA pairs unless EMU_F32_PAIR=0): every shape
issues the same MMAs in the same order for each output element, so C must
be bit-identical across shapes and within the FP32-mode bar of the oracle.
The switches are read once per process, so each shape runs in a child
process."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import hashlib, sys
sys.path.insert(0, {root!r})
sys.path.insert(0, {tests!r})
import numpy as np
import oracle, synth
import paper_2609_04663_gb300 as emu
from helpers import device, fp32_within_tolerance, gemm_f32_one_accumulator, to_dev
dev = device()
# 4000 x 4096: 256 pair tiles (3.4 waves), so by default the full waves run
# on pairs and the last 28 pair tiles as 128 x 128 quarters (the last tile
# row holds 32 of the 128 rows)
for M, N, K, seed in [(300, 333, 700, 1), (129, 257, 33, 3), (256, 512, 1024, 8), (1024, 1024, 512, 9),
                      (4000, 4096, 96, 10)]:
    A, B = synth.gemm_inputs("f32", M, N, K, seed)
    C, flags = gemm_f32_one_accumulator(to_dev(A, dev), to_dev(B, dev))
    assert flags == 0
    Cn = C.cpu().numpy()
    rows = list(range(M)) if M <= 1024 else [0, 1, 1999, 3840, 3999]
    ok, worst = fp32_within_tolerance(Cn[rows], oracle.gemm_f32(A[rows], B)[0], A[rows], B)
    assert ok, (M, N, K, worst)
    print("digest", M, N, K, hashlib.sha256(Cn.tobytes()).hexdigest())
"""


def _run(tile, pair=True):
    env = dict(os.environ)
    env.pop("EMU_F32_TILE", None)
    env.pop("EMU_F32_PAIR", None)
    if tile:
        env["EMU_F32_TILE"] = tile
    if not pair:
        env["EMU_F32_PAIR"] = "0"
    code = CHILD.format(root=ROOT, tests=os.path.join(ROOT, "tests"))
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    return [line for line in r.stdout.splitlines() if line.startswith("digest")]


def test_f32_tile_shapes_parity_and_bit_identity():
    ref = _run(None)
    assert len(ref) == 5
    for tile in ("128x256", "128x128", "128x64"):
        assert _run(tile) == ref, tile
    # 128 x 256 tiles with one CTA each instead of pairs (129 and 300 rows
    # leave the second CTA of the last pair wholly or partly below the matrix)
    assert _run("128x256", pair=False) == ref


CHILD64 = r"""
import hashlib, sys
sys.path.insert(0, {root!r})
sys.path.insert(0, {tests!r})
import numpy as np
import oracle, synth
import paper_2609_04663_gb300 as emu
from helpers import device, to_dev
dev = device()

def digest(tag, C):
    print("digest", tag, hashlib.sha256(C.tobytes()).hexdigest())

# whole-matrix levels, Algorithm 2: ragged tiles, tiny and multi-chunk K, every product count
# (with 256 x 256 tiles on CTA pairs: 300 rows leave the second CTA of the
# last pair below the matrix, 129 rows leave it one row, 100 rows need no pair)
for M, N, K, seed, nprod in [(300, 333, 700, 1, 21), (129, 257, 33, 3, 6), (256, 512, 1024, 8, 10),
                             (520, 130, 300, 5, 15), (100, 600, 500, 9, 6)]:
    A, B = synth.gemm_inputs("f64", M, N, K, seed)
    C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), nprod)
    assert emu.read_flags(ws) == 0
    Cn = C.cpu().numpy()
    assert np.array_equal(Cn, oracle.gemm_f64(A, B, nprod)[0]), (M, N, K, nprod)
    digest((M, N, K, nprod), Cn)
# a 4096 x 4096 result: 3.4 waves of 256 x 256 tiles on CTA pairs, so by
# default the full waves run as pairs and the last tiles as 128 x 128 parts
A, B = synth.gemm_inputs("f64", 4096, 4096, 264, 14)
C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), 10)
assert emu.read_flags(ws) == 0
Cn = C.cpu().numpy()
for r in (0, 1234, 3000, 4095):
    assert np.array_equal(Cn[r], oracle.gemm_f64(A, B, 10, rows=(r, r + 1))[0][0]), r
digest("mixed", Cn)
# positive entries: every running sum passes 2^24 units, so the carries into the low words run
A, B = synth.gemm_inputs("f64", 200, 300, 8192, 11)
A, B = np.abs(A), np.abs(B)
C, ws = emu.gemm_f64(to_dev(A, dev), to_dev(B, dev), 21)
assert emu.read_flags(ws) == 0
Cn = C.cpu().numpy()
for r in (0, 77, 199):
    assert np.array_equal(Cn[r], oracle.gemm_f64(A, B, 21, rows=(r, r + 1))[0][0]), r
digest("carry", Cn)
# levels per row / column (the TwoSum and per-element carry paths)
A, B = synth.gemm_inputs("f64", 260, 300, 1000, 12)
A = A * np.exp2(np.arange(260) % 7 - 3)[:, None]
C, ws = emu.gemm_f64_rowcol(to_dev(A, dev), to_dev(B, dev), 15)
assert emu.read_flags(ws) == 0
Cn = C.cpu().numpy()
assert np.array_equal(Cn, oracle.gemm_f64_rowcol(A, B, 15)[0])
digest("rowcol", Cn)
# merged tail: the head is the product-sum, the tail added last
A, B = synth.gemm_inputs("f64", 300, 400, 600, 13)
C, ws = emu.gemm_f64_merged(to_dev(A, dev), to_dev(B, dev), 21, 4)
assert emu.read_flags(ws) == 0
digest("merged", C.cpu().numpy())
"""


def _run64(tile):
    env = dict(os.environ)
    env.pop("EMU_F64_TILE", None)
    if tile:
        env["EMU_F64_TILE"] = tile
    code = CHILD64.format(root=ROOT, tests=os.path.join(ROOT, "tests"))
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    return [line for line in r.stdout.splitlines() if line.startswith("digest")]


def test_f64_tile_shapes_parity_and_bit_identity():
    """The FP64 product-sum's tile shapes (EMU_F64_TILE=128x128 / 128x256 /
    256x256, the last on CTA pairs): all form the same exact per-product sums
    and add them in Algorithm 2's order, so C must equal the oracle bit for bit
    with any shape, and with the default schedule that runs the last partial
    wave of 256-column tiles as 128 x 128 ones, through the plain, carry,
    per-row/column and merged-tail paths."""
    ref = _run64(None)
    assert len(ref) == 9
    for tile in ("256x256", "128x256", "128x128"):
        assert _run64(tile) == ref, tile
