#!/usr/bin/env python3
"""Throughput of the BF16 component-product GEMM emulation on GB300.

Metric: emulated GEMM TFLOP/s = 2 M N K / t per step, where a step is one
pass of the whole hot path on resident inputs: split A, split B (transposed)
and the tensor-core product-sum.  The headline workload is FP32 mode (6
products) at M = N = K = 16384, the top of the paper's square sweep; FP64
mode (4096^3 at 6, 10, 15 and 21 products, 8192^3 scaled inputs, the
large-K shape) and the rest of the FP32 sweep are reported under "variants".

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   (the CPU oracle on the host cores)

Multi-GPU (torchrun, one rank per GPU): every rank runs its own independent
GEMM of the same size (replicas, weak scaling); no data moves between ranks.
Rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import datetime
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "emulated GEMM TFLOP/s (2MNK/t) FP32-6p & FP64-6/10/15/21p; tensor-pipe % peak"
DEFAULT_WORKLOAD = "fp32_n16384"
L2_BYTES = 129 * 1024 * 1024


# ------------------------------------------------------------ distributed
def dist_init():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    """Max of a per-rank scalar (the slowest rank sets the job time)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(flop_per_rank_step: float, steps: int, world: int, t_max_s: float) -> float:
    """Whole-job TFLOP/s: the work of all ranks over the slowest rank's time."""
    return flop_per_rank_step * steps * world / t_max_s / 1e12


# ------------------------------------------------------------ clock sampler
class ClockSampler:
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50",
                 "-i", str(self.gpu)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self, window=None):
        """Median SM clock, max clock and throttle reasons of the samples taken
        inside window = (t0, t1) (epoch seconds; all samples if None or if the
        window caught none)."""
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.splitlines():
            f = [t.strip() for t in line.split(",")]
            if len(f) < 9:
                continue
            try:
                ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                rows.append((ts, float(f[2]), float(f[3]), f[5:9]))
            except ValueError:
                continue
        inside = [r for r in rows if window and window[0] <= r[0] <= window[1]]
        used = inside if inside else rows
        sm = [r[1] for r in used]
        mx = [r[2] for r in used]
        reasons = {name for r in used for name, val in zip(self.NAMES, r[3]) if val.lower().startswith("active")}
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm),
                "window": "timed region" if inside else "whole run (no sample inside the timed region)"}


# ------------------------------------------------------------ workloads
def workload(name: str):
    import synth
    kind, M, N, K, seed, phi, nprods = synth.WORKLOADS[name]
    return kind, M, N, K, seed, phi, nprods


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"bf16_sustained": p["bf16_tflops_sustained"], "bf16_burst": p["bf16_tflops"],
                "hbm": p["hbm_gbs"], "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"bf16_sustained": 1700.0, "bf16_burst": 1900.0, "hbm": 6800.0, "source": "fallback"}


def code_digest(path: str) -> str:
    """sha256 prefix of a CUDA source and of the project headers it includes
    (recursively), with comments and whitespace removed, so that a comment
    edit does not invalidate counters taken on the same code but a change to
    any code the kernel is built from does."""
    import re
    seen, parts = set(), []

    def walk(p):
        p = os.path.normpath(p)
        if p in seen or not os.path.exists(p):
            return
        seen.add(p)
        text = open(p).read()
        for inc in re.findall(r'^\s*#\s*include\s+"([^"]+)"', text, flags=re.M):
            walk(os.path.join(os.path.dirname(p), inc))
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        parts.append(os.path.basename(p) + ":" + re.sub(r"\s+", "", text))

    walk(path)
    return hashlib.sha256("\n".join(parts).encode()).hexdigest()[:16]


def kernel_traffic(kernel: str, workload_name: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the current code of the kernel (else None)."""
    src = os.path.join(ROOT, "paper_2609_04663_gb300", "csrc", kernel + ".cu")
    try:
        digest = code_digest(src)
        with open(os.path.join(ROOT, "profiles", "traffic.txt")) as f:
            for line in f:
                t = line.split()
                if len(t) >= 4 and not line.startswith("#") and t[0] == kernel and t[1] == workload_name \
                        and t[2] == digest:
                    return float(t[3])
    except OSError:
        pass
    return None


class Case:
    """Device-resident inputs, planes and output of one GEMM workload."""

    def __init__(self, name: str, rank: int, nprod: int | None = None, fused: bool = False,
                 merge_from: int | None = None, api: bool = False):
        import numpy as np
        import torch
        import synth
        import paper_2609_04663_gb300 as emu
        self.emu, self.torch = emu, torch
        self.name = name
        kind, M, N, K, seed, phi, nprods = workload(name)
        self.kind, self.M, self.N, self.K = kind, M, N, K
        self.mode = 32 if kind.startswith("f32") else 64
        self.nprod = nprod or nprods[0]
        # FP32 only: the whole path in one kernel (emu_gemm_f32_fused), no planes
        self.fused = fused and self.mode == 32
        # FP64 only: the tail diagonals from merge_from on in one FP32 sum (emu_gemm_f64_merged)
        self.merge_from = merge_from if self.mode == 64 else None
        # the whole GEMM through the public call (emu_gemm_f32 / emu_gemm_f64), timed as one region
        self.api = api and not self.fused and self.merge_from is None
        # each rank draws its own problem (replicas): offset the seed by the rank
        A, B = synth.gemm_inputs(kind, M, N, K, seed + 1000003 * rank, phi=phi)
        self.A_host, self.B_host = A, B
        dev = torch.device("cuda")
        self.A = torch.from_numpy(A).to(dev)
        self.B = torch.from_numpy(B).to(dev)
        self.ldk = emu.gemm_ldk(K)
        s = 3 if self.mode == 32 else 6
        self.Ap = torch.empty((s, M, self.ldk), dtype=torch.int16, device=dev)
        self.Bp = torch.empty((s, N, self.ldk), dtype=torch.int16, device=dev)
        self.v = torch.empty(12, dtype=torch.int32, device=dev)
        self.C = torch.empty((M, N), dtype=torch.float32 if self.mode == 32 else torch.float64, device=dev)
        self.ws = emu.workspace(max(emu.emu_split_workspace_bytes(self.mode),
                                    emu.emu_prodsum_workspace_bytes(self.mode, M, N)), dev)
        self.gemm_ws = None
        if self.merge_from is not None:
            self.gemm_ws = emu.workspace(emu.emu_gemm_f64_merged_workspace_bytes(M, N, K), dev)
        if self.api:
            self.gemm_ws = emu.workspace(emu.emu_gemm_workspace_bytes(self.mode, M, N, K), dev)
        # the product-sum kernel that runs: FP64 mode has 128 x 128 tiles and 256-column tiles
        # (128 x 256 on one SM, 256 x 256 on a pair of SMs), both kernels named after their file
        self.kernel = "prodsum_f32" if self.mode == 32 else \
            "prodsum_f64w" if emu.emu_prodsum_f64_tile_columns(M, N) == 256 else "prodsum_f64"
        # the kernel's own name (FP32: 256 x 256 tiles on CTA pairs have a kernel of their own)
        self.kernel_name = "prodsum_f32_pair_kernel" if self.mode == 32 and emu.emu_prodsum_f32_tile_rows(M, N) == 256 \
            else self.kernel + "_kernel"
        self.flop = 2.0 * M * N * K
        self.exec_flop = self.flop * (6 if self.mode == 32 else self.nprod)
        # kernels of ours per step: FP32 split of both operands = 1 launch; FP64 split of both =
        # 5 (level maxima of both, then a speculative pass and a verifier per operand);
        # product-sum = 1, or 2 when the library runs the last partial wave of 256-column
        # tiles as 128 x 128 tiles (it reports its schedule)
        self.launches = 1 if self.fused else 1 + emu.emu_prodsum_f32_launches(M, N) if self.mode == 32 else \
            5 + emu.emu_prodsum_f64_launches(M, N)
        if self.merge_from is not None:
            self.launches += 1                    # the tail kernel
        if self.api and self.mode == 32:
            self.launches = 2                     # both splits in one launch, then the product-sum
        del np

    def split(self, stream):
        emu, st = self.emu, stream.cuda_stream
        ws, n = self.ws.data_ptr(), self.ws.numel()
        if self.fused or self.merge_from is not None or self.api:
            return                                # the whole GEMM runs in prodsum()
        if self.mode == 32:
            r = emu.emu_split_f32_pair(self.M, self.N, self.K, self.A.data_ptr(), self.A.stride(0), self.B.data_ptr(),
                                       self.B.stride(0), self.Ap.data_ptr(), self.Bp.data_ptr(), self.ldk, ws, n, st)
        else:
            # only the d slices the product-sum reads (d = 3, 4, 5, 6 for nprod = 6, 10, 15, 21)
            d = {6: 3, 10: 4, 15: 5, 21: 6}[self.nprod]
            r = emu.emu_split_f64_pair(self.M, self.N, self.K, self.A.data_ptr(), self.A.stride(0), self.B.data_ptr(),
                                       self.B.stride(0), self.Ap.data_ptr(), self.Bp.data_ptr(), self.ldk, d,
                                       self.v.data_ptr(), self.v.data_ptr() + 24, ws, n, st)
        assert r == 0, r

    def prodsum(self, stream):
        emu, st = self.emu, stream.cuda_stream
        if self.api and self.mode == 32:
            r = emu.emu_gemm_f32(self.M, self.N, self.K, self.A.data_ptr(), self.K, self.B.data_ptr(), self.N,
                                 self.C.data_ptr(), self.N, self.gemm_ws.data_ptr(), self.gemm_ws.numel(), st)
        elif self.api:
            r = emu.emu_gemm_f64(self.M, self.N, self.K, self.A.data_ptr(), self.K, self.B.data_ptr(), self.N,
                                 self.C.data_ptr(), self.N, self.nprod, self.gemm_ws.data_ptr(), self.gemm_ws.numel(),
                                 st)
        elif self.merge_from is not None:
            r = emu.emu_gemm_f64_merged(self.M, self.N, self.K, self.A.data_ptr(), self.K, self.B.data_ptr(), self.N,
                                        self.C.data_ptr(), self.N, self.nprod, self.merge_from,
                                        self.gemm_ws.data_ptr(), self.gemm_ws.numel(), st)
        elif self.fused:
            r = emu.emu_gemm_f32_fused(self.M, self.N, self.K, self.A.data_ptr(), self.K, self.B.data_ptr(), self.N,
                                       self.C.data_ptr(), self.N, self.ws.data_ptr(), self.ws.numel(), st)
        elif self.mode == 32:
            r = emu.emu_prodsum_f32(self.M, self.N, self.K, self.Ap.data_ptr(), self.Bp.data_ptr(), self.ldk,
                                    self.C.data_ptr(), self.N, self.ws.data_ptr(), self.ws.numel(), st)
        else:
            r = emu.emu_prodsum_f64(self.M, self.N, self.K, self.Ap.data_ptr(), self.Bp.data_ptr(), self.ldk,
                                    self.v.data_ptr(), self.v.data_ptr() + 24, self.nprod, self.C.data_ptr(), self.N,
                                    self.ws.data_ptr(), self.ws.numel(), st)
        assert r == 0, r

    def split_bytes(self):
        """Algorithmic HBM bytes of the two splits: FP32 4 B read + 6 B written
        per entry; FP64 8 B (level-0 max) + 8 B (fused pass) read + 2 B written
        per slice formed (the d slices the product-sum reads)."""
        per = 10 if self.mode == 32 else 16 + 2 * {6: 3, 10: 4, 15: 5, 21: 6}[self.nprod]
        return per * (self.M * self.K + self.K * self.N)


def time_device(case: Case, steps: int, warmup: int, world: int, flush: bool):
    """Time `steps` whole-path steps with CUDA events on the launching stream."""
    torch = case.torch
    stream = torch.cuda.current_stream()
    scratch = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device="cuda") if flush else None
    for _ in range(warmup):
        case.split(stream)
        case.prodsum(stream)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    epoch0 = time.time()
    one_region = case.api or case.fused or case.merge_from is not None
    for i in range(steps):
        if flush:
            scratch.fill_(i & 0xFF)              # evict the previous step from L2 (not timed)
        ev[i][0].record(stream)
        if not one_region:
            case.split(stream)
            ev[i][1].record(stream)
        case.prodsum(stream)
        ev[i][2].record(stream)
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    window = (epoch0, time.time())
    split_ms = [0.0 if one_region else a.elapsed_time(b) for a, b, _ in ev]
    prod_ms = [a.elapsed_time(c) if one_region else b.elapsed_time(c) for a, b, c in ev]
    step_ms = [a.elapsed_time(c) for a, _, c in ev]
    return {"step_ms": step_ms, "split_ms": split_ms, "prodsum_ms": prod_ms, "wall_s": wall, "window": window}


def time_e2e(case: Case, steps: int, warmup: int, world: int):
    """Same metric through the public host-buffer C-ABI call (emu_gemm_*_host):
    A and B in pinned host memory, C back in pinned host memory; the library
    pipelines the copies with the split and the product-sum, and all of it is
    inside the timing."""
    torch, emu = case.torch, case.emu
    stream = torch.cuda.current_stream()
    A_h = torch.from_numpy(case.A_host).pin_memory()
    B_h = torch.from_numpy(case.B_host).pin_memory()
    C_h = torch.empty(case.C.shape, dtype=case.C.dtype).pin_memory()
    need = emu.emu_gemm_host_workspace_bytes(case.mode, case.M, case.N, case.K)
    ws = emu.workspace(need, "cuda")
    M, N, K = case.M, case.N, case.K

    def step():
        st = stream.cuda_stream
        if case.mode == 32:
            r = emu.emu_gemm_f32_host(M, N, K, A_h.data_ptr(), K, B_h.data_ptr(), N, C_h.data_ptr(), N,
                                      ws.data_ptr(), ws.numel(), st)
        else:
            r = emu.emu_gemm_f64_host(M, N, K, A_h.data_ptr(), K, B_h.data_ptr(), N, C_h.data_ptr(), N,
                                      case.nprod, ws.data_ptr(), ws.numel(), st)
        assert r == 0, r

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    barrier(world)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for _ in range(steps):
        step()
    end.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    t = max_over_ranks(start.elapsed_time(end) / 1e3, world)
    h2d = case.A_host.nbytes + case.B_host.nbytes
    d2h = C_h.numel() * C_h.element_size()
    flags = emu.read_flags(ws)
    del ws, A_h, B_h, C_h
    return {"value": job_throughput(case.flop, steps, world, t), "unit": "TFLOP/s",
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "api": "emu_gemm_f32_host" if case.mode == 32 else "emu_gemm_f64_host", "flags": flags}


# ------------------------------------------------------------ CPU oracle
class OracleSampler:
    """Times the CPU oracle (as it stands) on a bounded sample of a workload.

    One sample: the split of B (FP32: a block of B's rows, scaled to all K
    rows -- the FP32 split is elementwise; FP64: the whole of B, because its
    levels are global), the split of A (FP32: the sampled rows; FP64: the
    whole of A), each pro-rated to the sampled output rows, plus the
    product-sum of the sampled rows.  Value = 2 * rows * N * K / time."""

    def __init__(self, name: str, nprod: int | None = None):
        import synth
        kind, M, N, K, seed, phi, nprods = workload(name)
        self.name, self.kind, self.M, self.N, self.K = name, kind, M, N, K
        self.nprod = nprod or nprods[0]
        self.A, self.B = synth.gemm_inputs(kind, M, N, K, seed, phi=phi)
        self.rows = 2
        self.Bp = None

    def _split(self, X):
        import oracle
        return oracle.split_f32(X)[0] if self.kind.startswith("f32") else oracle.split_f64(X)[0]

    def sample(self, budget_s: float):
        import numpy as np
        import oracle
        M, N, K = self.M, self.N, self.K
        t0 = time.perf_counter()
        if self.kind.startswith("f32"):
            kb = min(K, 1024)
            self._split(self.B[:kb])
            t_b = (time.perf_counter() - t0) * K / kb
            if self.Bp is None:
                self.Bp = self._split(self.B)
        else:
            self.Bp = self._split(self.B)
            t_b = time.perf_counter() - t0
            t0 = time.perf_counter()
            self.Ap = self._split(self.A)
            t_a_full = time.perf_counter() - t0
        while True:
            sel = np.arange(self.rows)
            t0 = time.perf_counter()
            if self.kind.startswith("f32"):
                oracle.prodsum_f32(self._split(self.A[sel]), self.Bp)
            else:
                oracle.prodsum_f64(self.Ap[:, sel], self.Bp, self.nprod)
            t_rows = time.perf_counter() - t0
            if t_rows >= budget_s / 3 or self.rows >= M:
                break
            self.rows = min(M, self.rows * 2)
        share = self.rows / M
        t = t_rows + t_b * share + (0.0 if self.kind.startswith("f32") else t_a_full * share)
        cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
        return {"value": 2.0 * self.rows * N * K / t / 1e12, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                "sample": f"{self.rows} of {M} output rows of {self.name} (nprod "
                          f"{6 if self.kind.startswith('f32') else self.nprod}); operand splits timed and pro-rated to "
                          f"those rows; {t:.2f} s of CPU work"}


def oracle_sample(name: str, target_s: float = 15.0):
    return OracleSampler(name).sample(target_s)


# ------------------------------------------------------------ arms
def reference_arm(args, rank, world):
    if rank != 0:
        return 0
    name = args.workload
    kind, M, N, K, *_ = workload(name)
    sampler = OracleSampler(name)
    budget = min(args.ref_seconds, 120.0 / max(args.steps + args.warmup, 1))
    for _ in range(args.warmup):
        sampler.sample(budget)
    vals = []
    t_start = time.perf_counter()
    for _ in range(args.steps):
        vals.append(sampler.sample(budget))
    wall = time.perf_counter() - t_start
    v = statistics.mean(x["value"] for x in vals)
    cpu = dict(vals[-1])
    cpu["value"] = v
    line = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * wall / max(args.steps, 1),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32" if kind.startswith("f32") else "f64", "data": "synthetic",
        "config": {"workload": name, "M": M, "N": N, "K": K},
        "cpu_baseline": cpu,
        "e2e": {"value": v, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def capture_run(args, local):
    """--capture W[:P],W[:P],...: run each workload's split and product-sum
    --warmup + --steps times in one process and print, for each, the name of
    the product-sum kernel and the number of product-sum launches per step, so
    that one profiler run (its kernel filter on "prodsum") yields the counters
    of every workload in order.  Prints no JSON line."""
    import torch
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    for item in args.capture.split(","):
        name, _, nprod = item.partition(":")
        case = Case(name, 0, int(nprod) if nprod else None)
        stream = torch.cuda.current_stream()
        for _ in range(args.warmup + args.steps):
            case.split(stream)
            case.prodsum(stream)
        torch.cuda.synchronize()
        per_step = (case.emu.emu_prodsum_f32_launches if case.mode == 32 else
                    case.emu.emu_prodsum_f64_launches)(case.M, case.N)
        print(f"capture {name}" + (f"_np{case.nprod}" if case.mode == 64 else "") +
              f" {case.kernel} launches_per_step={per_step} steps={args.warmup + args.steps}", flush=True)
        del case
        torch.cuda.empty_cache()
    return 0


def gpu_arm(args, rank, world, local):
    import torch
    torch.cuda.set_device(local)
    import __graft_entry__
    __graft_entry__.build()
    pk = peaks()
    name = args.workload
    case = Case(name, rank, args.nprod, fused=args.fused, merge_from=args.merge_from)
    clocks = ClockSampler(local)
    clocks.start()
    res = time_device(case, args.steps, args.warmup, world, flush=False)
    clk = clocks.stop(res["window"])
    t_job = max_over_ranks(sum(res["step_ms"]) / 1e3, world)
    value = job_throughput(case.flop, args.steps, world, t_job)
    prod_ms = statistics.mean(res["prodsum_ms"])
    split_ms = statistics.mean(res["split_ms"])
    achieved = case.exec_flop / (prod_ms / 1e3) / 1e12
    # the timed region is well under the seconds-long loop of the sustained
    # figure, so the (higher) burst peak is the denominator
    roofline = {"bound": "tensor", "achieved": achieved, "peak": pk["bf16_burst"], "unit": "TFLOP/s",
                "frac": achieved / pk["bf16_burst"],
                "peak_source": f"{pk['source']} bf16 burst (cuBLAS 8192^3); sustained {pk['bf16_sustained']}",
                "kernel": "gemm_f32_fused_kernel" if case.fused else case.kernel_name,
                "traffic": None if case.fused or case.merge_from else
                           kernel_traffic(case.kernel, name if case.mode == 32 else f"{name}_np{case.nprod}")}
    flags = case.emu.read_flags(case.gemm_ws if case.gemm_ws is not None else case.ws)
    e2e = None if args.no_e2e else time_e2e(case, max(2, min(args.steps, 5)), 1, world)
    split_gbs = case.split_bytes() / (split_ms / 1e3) / 1e9
    line = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * t_job / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": name, "mode": f"fp{case.mode}" + ("_fused" if case.fused else "") +
                   (f"_merged{case.merge_from}" if case.merge_from else ""), "nprod": case.nprod if case.mode == 64 else 6,
                   "M": case.M, "N": case.N, "K": case.K, "parallelism": f"replicas{world}",
                   "l2": "inputs larger than L2 (no flush needed)"},
        "breakdown": {"split_ms": split_ms, "prodsum_ms": prod_ms, "split_gbs": split_gbs,
                      "split_frac_hbm": split_gbs / pk["hbm"], "executed_tflops": achieved,
                      "effective_prodsum_only_tflops": case.flop / (prod_ms / 1e3) / 1e12},
        "roofline": roofline, "clocks": clk, "e2e": e2e, "gpu_launches": case.launches * args.steps,
        "flags": flags,
    }
    del case
    torch.cuda.empty_cache()
    if not args.no_variants:
        line["variants"] = variants(args, rank, world, pk)
    if rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = oracle_sample(name, target_s=args.ref_seconds)
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def variants(args, rank, world, pk):
    """The other workloads, a few steps each, L2 flushed between steps."""
    out = {}
    # entries: (workload, FP64 product count | "fused" | (product count, merge_from)).
    # The default list covers every configuration of the paper's evaluation
    # that these workloads stand in for: FP32 256^3; the FP32 square sweep
    # 1024-8192 (16384 is the headline); FP64 4096^3 at 6/10/15/21 products;
    # FP64 8192^3 scaled inputs at 21 and 10 products; the large-K shape
    # 2048 x 2048 x 65536 in FP32 and at every FP64 product count.
    todo = [("fp32_n256", "api"), ("fp32_n1024", "api"), ("fp32_n2048", "api"), ("fp32_n4096", None),
            ("fp32_n8192", None), ("fp64_n4096", 6), ("fp64_n4096", 10), ("fp64_n4096", 15), ("fp64_n4096", 21),
            ("fp64_scaled_phi4_n8192", 21), ("fp64_scaled_phi4_n8192", 10), ("fp64_scaled_phi0.5_n8192", 21),
            ("fp64_scaled_phi2_n8192", 21), ("fp32_largek", None), ("fp64_largek", 6), ("fp64_largek", 10),
            ("fp64_largek", 15), ("fp64_largek", 21)]
    if args.all_variants:
        todo += [("fp32_n8192", "fused"), ("fp32_n16384", "fused"), ("fp64_n4096", (21, 4)), ("fp64_n4096", (15, 4)),
                 ("fp64_scaled_phi4_n8192", (21, 4)), ("fp64_scaled_phi0.5_n8192", (21, 4)),
                 ("fp32_cancel_n4096", None), ("fp64_cancel_n4096", 21)]
    torch = __import__("torch")
    for name, nprod in todo:
        fused, api = nprod == "fused", nprod == "api"
        merge_from = nprod[1] if isinstance(nprod, tuple) else None
        nprod = nprod[0] if isinstance(nprod, tuple) else None if fused or api else nprod
        case = Case(name, rank, nprod, fused=fused, merge_from=merge_from, api=api)
        # steps of a few microseconds vary by some microseconds: many more of them
        steps = 50 if case.flop < 2e11 else max(3, args.variant_steps)
        res = time_device(case, steps, 5 if case.flop < 2e11 else 2, world, flush=True)
        t = max_over_ranks(sum(res["step_ms"]) / 1e3, world)
        pm = statistics.mean(res["prodsum_ms"])
        key = f"{name}" + (f"_np{case.nprod}" if case.mode == 64 else "_fused" if fused else "_gemm" if api else "") + \
            (f"_merged{merge_from}" if merge_from else "")
        out[key] = {"tflops": job_throughput(case.flop, len(res["step_ms"]), world, t),
                    "ms_per_step": 1e3 * t / len(res["step_ms"]),
                    "prodsum_ms": pm, "split_ms": statistics.mean(res["split_ms"]),
                    "executed_tflops": case.exec_flop / (pm / 1e3) / 1e12,
                    "frac_of_bf16_peak": case.exec_flop / (pm / 1e3) / 1e12 / pk["bf16_burst"],
                    "kernel": case.kernel,
                    "traffic": None if fused or merge_from or api else
                               kernel_traffic(case.kernel, name if case.mode == 32 else f"{name}_np{case.nprod}"),
                    "flags": case.emu.read_flags(case.gemm_ws if case.gemm_ws is not None else case.ws)}
        del case
        torch.cuda.empty_cache()
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--nprod", type=int, default=None, help="FP64 product count (6, 10, 15, 21)")
    ap.add_argument("--fused", action="store_true",
                    help="FP32 workloads: time emu_gemm_f32_fused (split inside the product-sum) as the step")
    ap.add_argument("--merge-from", type=int, default=None,
                    help="FP64 workloads: time emu_gemm_f64_merged with the tail from this diagonal as the step")
    ap.add_argument("--variant-steps", type=int, default=5)
    ap.add_argument("--all-variants", action="store_true")
    ap.add_argument("--no-variants", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--ref-seconds", type=float, default=15.0)
    ap.add_argument("--capture", default=None,
                    help="W[:P],...: only run these workloads' steps for a profiler (see capture_run); no JSON")
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "ours":
        ap.error("--warmup must be at least 3")
    rank, world, local = dist_init()
    if args.impl == "reference":
        return reference_arm(args, rank, world)
    if args.capture:
        return capture_run(args, local)
    return gpu_arm(args, rank, world, local)


if __name__ == "__main__":
    sys.exit(main())
