"""bench.py's multi-rank path on CPU with the gloo backend (world size 2):
the job time is the slowest rank's, the throughput counts every rank's work,
and under torchrun only rank 0 prints the JSON line."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist
    r, w, _ = bench.dist_init()
    t = bench.max_over_ranks(1.0 + r, w)                 # rank 1 is the slow one
    v = bench.job_throughput(1e12, steps=4, world=w, t_max_s=t)
    bench.barrier(w)
    out.put((r, w, t, v))
    dist.destroy_process_group()


def test_max_over_ranks_and_job_throughput_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r, w, t, v in res:
        assert w == 2 and t == 2.0                       # max over ranks
        assert v == pytest.approx(1e12 * 4 * 2 / 2.0 / 1e12)


def test_torchrun_reference_arm_prints_one_line():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference",
           "--workload", "fp32_n256", "--steps", "1", "--warmup", "0", "--gpus", "2", "--ref-seconds", "0.2"]
    env = dict(os.environ, OMP_NUM_THREADS="2")
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300, env=env)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"


def test_clock_sampler_keeps_the_timed_window():
    """Only samples stamped inside the timed region count; throttle reasons
    are those seen there."""
    import datetime
    import bench

    class FakeProc:
        def __init__(self, out):
            self.out = out

        def terminate(self):
            pass

        def communicate(self, timeout=None):
            return self.out, ""

    def line(t, mhz, power_cap):
        ts = datetime.datetime.fromtimestamp(t).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
        return f"{ts}, 0, {mhz}, 2070, 900.0, Not Active, Not Active, Not Active, {'Active' if power_cap else 'Not Active'}"

    t0 = 1_800_000_000.0
    out = "\n".join([line(t0 - 1.0, 300, True), line(t0 + 0.1, 1900, False), line(t0 + 0.2, 1950, False),
                     line(t0 + 5.0, 400, True)])
    s = bench.ClockSampler(0)
    s.proc = FakeProc(out)
    clk = s.stop((t0, t0 + 1.0))
    assert clk["samples"] == 2 and clk["sm_mhz"] == 1925 and clk["reasons"] == [] and clk["sm_max_mhz"] == 2070
    s.proc = FakeProc(out)
    assert s.stop((t0 + 10, t0 + 11))["samples"] == 4             # nothing inside: every sample
