"""The FP32 product-sum's alternative tile (EMU_F32_TILE=128x128: 128 x 128
tiles, 64-wide K-blocks, 128-byte swizzle, two stages) against the oracle.
The switch is read once per process, so the case runs in a child process."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys
sys.path.insert(0, {root!r})
sys.path.insert(0, {tests!r})
import numpy as np
import oracle, synth
import paper_2609_04663_gb300 as emu
from helpers import device, fp32_within_tolerance, to_dev
dev = device()
for M, N, K, seed in [(300, 333, 700, 1), (129, 257, 33, 3), (256, 512, 1024, 8)]:
    A, B = synth.gemm_inputs("f32", M, N, K, seed)
    C, ws = emu.gemm_f32(to_dev(A, dev), to_dev(B, dev))
    assert emu.read_flags(ws) == 0
    ok, worst = fp32_within_tolerance(C.cpu().numpy(), oracle.gemm_f32(A, B)[0], A, B)
    assert ok, (M, N, K, worst)
print("tile-option-ok")
"""


def test_f32_tile_128x128_parity():
    env = dict(os.environ, EMU_F32_TILE="128x128")
    code = CHILD.format(root=ROOT, tests=os.path.join(ROOT, "tests"))
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "tile-option-ok" in r.stdout, r.stdout[-2000:] + r.stderr[-2000:]
