"""bench.py's DRAM-traffic bookkeeping on the CPU: the source digest that keys
profiles/traffic.txt ignores comments and whitespace but not code, every
entry of the table parses and names a bench workload, and the entries were
taken on the current product-sum sources (so the bench reports them)."""
import importlib.util
import os
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_04663_gb300", "csrc")


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _copy_tree(tmp_path):
    """The kernel sources and the C-ABI header laid out as in the package,
    so that relative includes resolve."""
    dst = tmp_path / "pkg" / "csrc"
    shutil.copytree(CSRC, dst)
    shutil.copytree(os.path.join(ROOT, "include"), tmp_path / "include")
    return dst


def test_digest_ignores_comments_but_not_code(bench, tmp_path):
    dst = _copy_tree(tmp_path)
    f = dst / "prodsum_f32.cu"
    d0 = bench.code_digest(str(f))
    assert d0 == bench.code_digest(os.path.join(CSRC, "prodsum_f32.cu"))
    text = f.read_text()
    f.write_text("// a comment\n/* another\n   one */\n" + text.replace("\n", "\n  ", 3))
    assert bench.code_digest(str(f)) == d0
    f.write_text(text.replace("kRateQuarter = 0.85", "kRateQuarter = 0.86", 1))
    assert bench.code_digest(str(f)) != d0
    f.write_text(text)
    (dst / "common.cuh").write_text((dst / "common.cuh").read_text() + "\nstatic int emu_extra = 1;\n")
    assert bench.code_digest(str(f)) != d0                 # an included header changed


def test_traffic_table_entries(bench):
    entries = []
    with open(os.path.join(ROOT, "profiles", "traffic.txt")) as fh:
        for line in fh:
            if line.startswith("#") or not line.strip():
                continue
            kernel, name, digest, nbytes = line.split()
            entries.append((kernel, name, digest, float(nbytes)))
    assert entries
    kernels = {k for k, _, _, _ in entries}
    assert kernels <= {"prodsum_f32", "prodsum_f64", "prodsum_f64w"}
    for kernel, name, digest, nbytes in entries:
        base = name.rsplit("_np", 1)[0] if kernel != "prodsum_f32" else name
        bench.workload(base)                              # a known workload
        assert nbytes > 0 and len(digest) == 16
    # the headline workload has an entry, and every entry was captured on the
    # current sources of its kernel
    assert any(k == "prodsum_f32" and n == bench.DEFAULT_WORKLOAD for k, n, _, _ in entries)
    current = {k: bench.code_digest(os.path.join(CSRC, k + ".cu")) for k in kernels}
    stale = [(k, n) for k, n, d, _ in entries if d != current[k]]
    assert not stale, stale
    assert bench.kernel_traffic("prodsum_f32", bench.DEFAULT_WORKLOAD) is not None
