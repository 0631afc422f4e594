"""The FP32 product-sum's tile shapes (EMU_F32_TILE=128x256 / 128x128 /
128x64 forces one; unset, the library picks by tile count): every shape
issues the same MMAs in the same order for each output element, so C must
be bit-identical across shapes and within the FP32-mode bar of the oracle.
The switch is read once per process, so each shape runs in a child process."""
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
from helpers import device, fp32_within_tolerance, to_dev
dev = device()
for M, N, K, seed in [(300, 333, 700, 1), (129, 257, 33, 3), (256, 512, 1024, 8), (1024, 1024, 512, 9)]:
    A, B = synth.gemm_inputs("f32", M, N, K, seed)
    C, ws = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    assert emu.read_flags(ws) == 0
    Cn = C.cpu().numpy()
    ok, worst = fp32_within_tolerance(Cn, oracle.gemm_f32(A, B)[0], A, B)
    assert ok, (M, N, K, worst)
    print("digest", M, N, K, hashlib.sha256(Cn.tobytes()).hexdigest())
"""


def _run(tile):
    env = dict(os.environ)
    env.pop("EMU_F32_TILE", None)
    if tile:
        env["EMU_F32_TILE"] = tile
    code = CHILD.format(root=ROOT, tests=os.path.join(ROOT, "tests"))
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    return [line for line in r.stdout.splitlines() if line.startswith("digest")]


def test_f32_tile_shapes_parity_and_bit_identity():
    ref = _run(None)
    assert len(ref) == 4
    for tile in ("128x256", "128x128", "128x64"):
        assert _run(tile) == ref, tile
