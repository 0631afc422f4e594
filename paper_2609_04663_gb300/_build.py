"""Compile the CUDA library ``_emu.so`` in-tree for sm_103a (GB300).

nvcc compiles each translation unit of ``csrc/`` in parallel with
``-gencode arch=compute_103a,code=sm_103a``, then links them into one shared
library.  No FTZ and no fast-math: the split kernels must round exactly as
the paper's equations say.
"""
from __future__ import annotations

import os
import shutil
import subprocess
import tempfile

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
SO = os.path.join(HERE, "_emu.so")
SOURCES = ["emu_api.cu", "split_f32.cu", "split_f64.cu", "split_fix.cu", "split_rc.cu", "prodsum_f32.cu", "gemm_f32_fused.cu", "prodsum_f64.cu", "prodsum_f64w.cu", "prodsum_tail.cu", "noalloc.cu", "host_api.cu", "epilogue.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-ftz=false", "-prec-div=true",
         "-prec-sqrt=true", "-fmad=true"]


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build the emulation library")


def _deps():
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cu", ".cuh"))]
    files.append(os.path.join(INCLUDE, "emu.h"))
    return files


def up_to_date() -> bool:
    if not os.path.exists(SO):
        return False
    t = os.path.getmtime(SO)
    return all(os.path.getmtime(f) <= t for f in _deps())


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and up_to_date():
        return SO
    nvcc = _nvcc()
    tmpdir = tempfile.mkdtemp(prefix="emu_build_", dir=HERE)
    try:
        procs, objs = [], []
        for src in SOURCES:
            obj = os.path.join(tmpdir, src.replace(".cu", ".o"))
            cmd = [nvcc, *ARCH, *FLAGS, "-I", INCLUDE, "-c", os.path.join(CSRC, src), "-o", obj]
            if verbose:
                cmd.insert(1, "-Xptxas=-v")
            procs.append((src, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)))
            objs.append(obj)
        errors = []
        for src, p in procs:
            out, _ = p.communicate()
            if verbose or p.returncode:
                print(out, end="")
            if p.returncode:
                errors.append(src)
        if errors:
            raise RuntimeError(f"nvcc failed for {errors}")
        tmp_so = os.path.join(tmpdir, "_emu.so")
        subprocess.run([nvcc, *ARCH, "-shared", "-o", tmp_so, *objs], check=True)
        os.replace(tmp_so, SO)
    finally:
        shutil.rmtree(tmpdir, ignore_errors=True)
    return SO


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
