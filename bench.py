"""Benchmark of C = A*B (CSR SpGEMM) on the GPU, one JSON line on stdout.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

A step is one full product -- symbolic pass (including its nnz read-back),
a fresh allocation of C's arrays, numeric pass and the final status read --
over device-resident inputs.  Between timed steps the L2 is flushed by
writing a buffer larger than it; each step is timed with CUDA events on the
stream the library runs on.  Throughput is GFLOP/s = 2 x products / time;
the effective HBM bandwidth uses the compulsory bytes (read A and B once,
write C once, at their stored widths).

The headline is the uniform 2^20 x 2^16 (16/row) times 2^16 x 2^16 (32/row)
product in fp32.  Without --workload, the line also carries `per_config`:
the same measurement (value, roofline, end to end, CPU oracle, clocks) for
each of the five named SpGEMM workloads, each timed for at least half a
second, and `sustained`: the headline product timed again over at least one
second with its own clock record.

Extra keys: `e2e` (the same product through the public Python API from
pinned host inputs to the host copy of C, copies inside the timed region),
`roofline` (the whole product -- symbolic + numeric, the span the throughput
target is set on -- against the measured copy bandwidth, with each pass's own
figure under `passes`; `traffic` is the DRAM bytes ncu recorded for the
current kernel sources, null when none match), `cpu_baseline` (the CPU oracle
on a bounded row sample, on this host's cores), `clocks` (nvidia-smi samples
during the timed region).

With an elementwise workload (``--workload ewise_* --op add|mul``) a step is
one elementwise operation C = A + B or C = A .* B and the value is its
effective bandwidth in GB/s of compulsory bytes; with ``--workload spmspv_*``
a step is one sparse matrix - sparse vector product y = A x (A resident by
columns, x the step's input), also in GB/s of compulsory bytes.

Under torchrun (N > 1) every rank runs its own replica of the workload on its
own GPU (no collective on the data path); rank 0 prints the line with the
maximum time over ranks.  `--impl reference` times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from synth import (EWISE_WORKLOADS, SPMSPV_WORKLOADS, WORKLOAD_ORDER, WORKLOADS, ewise_workload,  # noqa: E402
                   spmspv_workload, workload)

METRIC = "SpGEMM GFLOP/s (2×products) and effective HBM GB/s vs 8 TB/s, per config"
EWISE_METRIC = "SpAdd / Hadamard effective HBM GB/s (compulsory bytes: read A and B, write C)"
SPMSPV_METRIC = "SpMSpV effective HBM GB/s (compulsory bytes: read x, the columns of A it selects, write y)"
DEFAULT_WORKLOAD = "uniform_rect_1m"
NOMINAL_HBM_GBS = 8000.0

# Dominant kernel of each pass on the headline workload (the analysis,
# scatter and scan kernels move a few MB).
PASS_KERNELS = {"symbolic": "bmr_plan_kernel", "numeric": "bmr_numeric_kernel"}
PROFILES = os.path.join(ROOT, "profiles")


def source_digest(rel_path: str) -> str | None:
    """First 16 hex digits of the SHA-256 of a source file of this repository."""
    import hashlib
    path = os.path.join(ROOT, rel_path)
    if not os.path.exists(path):
        return None
    with open(path, "rb") as fh:
        return hashlib.sha256(fh.read()).hexdigest()[:16]


def recorded_traffic(workload: str, kernel: str) -> float | None:
    """DRAM bytes (read + write) of one full-size launch of `kernel` on
    `workload`, from a `traffic-record:` line of a profile summary under
    profiles/ (an ncu capture of a row cut, scaled by rows), or None when no
    record exists or the kernel's source changed since it was taken."""
    if not os.path.isdir(PROFILES):
        return None
    for name in sorted(os.listdir(PROFILES)):
        if not name.endswith(".md"):
            continue
        with open(os.path.join(PROFILES, name)) as fh:
            for line in fh:
                if not line.startswith("traffic-record:"):
                    continue
                kv = dict(x.split("=", 1) for x in line.split()[1:] if "=" in x)
                if kv.get("workload") != workload or kv.get("kernel") != kernel:
                    continue
                if source_digest(kv.get("source", "")) != kv.get("sha256"):
                    return None  # stale: the kernel changed since the capture
                return float(kv["dram_bytes"]) * float(kv["of"]) / float(kv["rows"])
    return None


def products_per_row(A, B) -> np.ndarray:
    lenB = np.diff(B.rowptr)
    ub = np.zeros(A.nrows, dtype=np.int64)
    if A.nnz:
        np.add.at(ub, np.repeat(np.arange(A.nrows), np.diff(A.rowptr)), lenB[A.colidx])
    return ub


def csr_bytes(nrows: int, nnz: int, value_bytes: int) -> int:
    return 8 * (nrows + 1) + (4 + value_bytes) * nnz


def measured_peaks() -> dict:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as fh:
            d = json.load(fh)
        return {"hbm_gbs": float(d["hbm_gbs"]), "source": "measured"}
    return {"hbm_gbs": 6800.0, "source": "fallback"}


class ClockSampler:
    """Samples SM clocks and throttle reasons with nvidia-smi while running.

    Samples carry nvidia-smi's own timestamps; `stop(t0, t1)` keeps those taken
    inside the wall-clock window [t0, t1] (widened to 0.5 s around it when the
    window is shorter than the sampling period)."""

    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int, period_ms: int = 25):
        self.index = index
        self.period_ms = period_ms
        self.proc = None
        self.lines: list[tuple[float, str]] = []
        self._t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", str(self.period_ms)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return self
        self._t = threading.Thread(target=self._read, daemon=True)
        self._t.start()
        time.sleep(0.3)  # let the first samples arrive before the timed region
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def stop(self, t0: float, t1: float) -> dict | None:
        if not self.proc:
            return None
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self._t:
            self._t.join(timeout=2)
        pad = 0.0 if (t1 - t0) > 4 * self.period_ms / 1e3 else 0.5
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, smax, reasons = [], [], set()
        for when, ln in self.lines:
            if not (t0 - pad <= when <= t1 + pad):
                continue
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm), "window_s": round(t1 - t0, 3)}


def oracle_sample(A, B, target_s: float, rng, cores: int) -> tuple[np.ndarray, float]:
    """A seeded uniform row sample on which the oracle runs for about target_s
    seconds (grown from 1024 rows by 4x until a run takes a quarter of the
    target, then scaled), and the time of its last sizing run."""
    from oracle import oracle_spgemm
    n = min(A.nrows, 1024)
    while True:
        rows = np.sort(rng.choice(A.nrows, size=n, replace=False))
        t0 = time.perf_counter()
        oracle_spgemm(A, B, rows=rows, threads=cores)
        dt = time.perf_counter() - t0
        if dt >= 0.25 * target_s or n >= A.nrows:
            break
        n = min(A.nrows, n * 4)
    want = int(n * target_s / max(dt, 1e-6))
    return np.sort(rng.choice(A.nrows, size=min(A.nrows, max(n, want)), replace=False)), dt


def cpu_baseline(A, B, ub: np.ndarray, target_s: float, seed: int = 0) -> dict:
    """The CPU oracle on a seeded row sample sized to about target_s seconds."""
    from oracle import oracle_spgemm
    cores = os.cpu_count() or 1
    rng = np.random.default_rng(seed)
    rows, _ = oracle_sample(A, B, target_s, rng, cores)
    nrows = rows.size
    t0 = time.perf_counter()
    oracle_spgemm(A, B, rows=rows, threads=cores)
    dt = time.perf_counter() - t0
    prods = int(ub[rows].sum())
    return {"value": round(2.0 * prods / dt / 1e9, 4), "unit": "GFLOP/s", "cores": cores, "kind": "oracle",
            "sample": f"{nrows} of {A.nrows} rows (seeded uniform sample, {prods} products), "
                      f"{dt:.1f} s, std::map per row, {cores} threads"}


def roofline_obj(nbytes: int, seconds: float, peaks: dict, traffic) -> dict:
    """Compulsory bytes over the measured mean duration, against the measured copy bandwidth."""
    achieved = nbytes / seconds / 1e9
    return {"bound": "hbm", "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": round(achieved / peaks["hbm_gbs"], 4), "peak_source": peaks["source"],
            "algorithmic_bytes": int(nbytes), "mean_ms": round(seconds * 1e3, 4), "traffic": traffic}


def numeric_kernels(info: dict) -> str:
    """Which numeric kernels a plan launches (from ws_spgemm_plan_info)."""
    names = []
    for key, kern in (("direct_rows", "direct_rows_kernel"), ("bitmap_rows", "bmr_numeric/bitmap_rows_kernel"),
                      ("hash_rows", "hash_rows_kernel"), ("sorted_rows", "sort_rows_kernel"),
                      ("rcd_rows", "rcd_numeric_kernel"), ("wb_rows", "wb_kernel"), ("dense_rows", "dense_rows_kernel")):
        if info.get(key):
            names.append(kern)
    return ", ".join(names) or "none"


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    pg = None
    if world > 1:
        import torch.distributed as dist
        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
        pg = dist
    return world, rank, local, pg


def reduce_max(x: float, world: int, pg, device) -> float:
    if world == 1:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int, pg) -> None:
    if world > 1:
        pg.barrier()


def is_ewise(args) -> bool:
    return args.workload in EWISE_WORKLOADS


def load_workload(args):
    """The named workload, optionally cut to the first --rows rows of A."""
    if is_ewise(args):
        return ewise_workload(args.workload)
    A, B = workload(args.workload)
    if args.rows and args.rows < A.nrows:
        from synth import row_subset
        A = row_subset(A, np.arange(args.rows))  # B stays the full right operand
    return A, B


def run_reference(args, world, rank) -> None:
    """CPU oracle arm: each step computes a bounded row sample on the host cores."""
    if rank != 0:
        return
    if is_ewise(args):
        run_reference_ewise(args)
        return
    from oracle import oracle_spgemm
    A, B = load_workload(args)
    ub = products_per_row(A, B)
    cores = os.cpu_count() or 1
    rng = np.random.default_rng(1234)
    rows, _ = oracle_sample(A, B, args.ref_step_s, rng, cores)  # one step ~ ref_step_s seconds
    nrows = rows.size
    prods = int(ub[rows].sum())
    for _ in range(args.warmup):
        oracle_spgemm(A, B, rows=rows, threads=cores)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle_spgemm(A, B, rows=rows, threads=cores)
        times.append(time.perf_counter() - t0)
    total = sum(times)
    value = 2.0 * prods * args.steps / total / 1e9
    sample = f"{nrows} of {A.nrows} rows per step (seeded uniform sample, {prods} products), {cores} threads"
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GFLOP/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * total / args.steps, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": str(A.vals.dtype).replace("float", "f"),
        "data": "synthetic", "config": {"workload": args.workload, "description": WORKLOADS[args.workload]},
        "cpu_baseline": {"value": round(value, 4), "unit": "GFLOP/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "GFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def ewise_bytes(A, B, nnz_c: int) -> int:
    s = A.vals.dtype.itemsize
    return csr_bytes(A.nrows, A.nnz, s) + csr_bytes(B.nrows, B.nnz, s) + csr_bytes(A.nrows, nnz_c, s)


def ewise_oracle_timed(A, B, op: str, steps: int) -> tuple[float, int]:
    """Seconds per oracle run (the whole operation: the elementwise oracle is
    vectorised numpy and finishes the full input in seconds) and nnz(C)."""
    from oracle import oracle_ewise
    times, nnz = [], 0
    for _ in range(steps):
        t0 = time.perf_counter()
        nnz = oracle_ewise(A, B, op).nnz
        times.append(time.perf_counter() - t0)
    return statistics.mean(times), nnz


def run_reference_ewise(args) -> None:
    A, B = load_workload(args)
    if args.warmup > 0:
        ewise_oracle_timed(A, B, args.op, args.warmup)
    dt, nnz = ewise_oracle_timed(A, B, args.op, max(args.steps, 1))
    value = ewise_bytes(A, B, nnz) / dt / 1e9
    sample = f"whole operation ({A.nnz} + {B.nnz} entries), numpy on one core"
    line = {
        "impl": "reference", "metric": EWISE_METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * dt, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": args.workload, "op": args.op, "description": EWISE_WORKLOADS[args.workload]},
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": 1, "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def spmspv_bytes(At, x_idx, nnz_y: int) -> int:
    """Compulsory bytes of y = A x: x, the column pointers and entries of the
    columns x selects, and y."""
    s = At.vals.dtype.itemsize
    cols = np.asarray(x_idx, dtype=np.int64)
    products = int((At.rowptr[cols + 1] - At.rowptr[cols]).sum())
    return (4 + s) * cols.size + 16 * cols.size + (4 + s) * products + (4 + s) * nnz_y


def run_spmspv(args, world, rank, local, pg) -> None:
    import torch
    from oracle import oracle_spmspv
    from paper_2606_20855_gb300 import _abi
    from paper_2606_20855_gb300.spgemm import DeviceCSR, SpMSpV
    from synth import transpose_csr

    A, xi, xv = spmspv_workload(args.workload)
    if args.impl == "reference":
        if rank != 0:
            return
        for _ in range(max(args.warmup, 0)):
            oracle_spmspv(A, xi, xv)
        times = []
        for _ in range(max(args.steps, 1)):
            t0 = time.perf_counter()
            y = oracle_spmspv(A, xi, xv)
            times.append(time.perf_counter() - t0)
        At = transpose_csr(A)
        dt = statistics.mean(times)
        value = spmspv_bytes(At, xi, y.nnz) / dt / 1e9
        line = {"impl": "reference", "metric": SPMSPV_METRIC, "value": round(value, 4), "unit": "GB/s",
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * dt, 3),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": {"workload": args.workload, "description": SPMSPV_WORKLOADS[args.workload]},
                "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
                                 "sample": "whole product, numpy on one core"},
                "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return
    _abi.load()
    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    At = transpose_csr(A)
    dAt = DeviceCSR.from_host(At, device)
    dxi = torch.from_numpy(xi).to(device)
    dxv = torch.from_numpy(xv).to(device)
    stream = torch.cuda.current_stream(device)
    l2 = torch.cuda.get_device_properties(device).L2_cache_size
    flush = torch.empty(max(2 * l2, 256 << 20) // 4, dtype=torch.int32, device=device)
    op = SpMSpV(dAt)
    for _ in range(args.warmup):
        yi, _ = op(dxi, dxv)
    nnz_y = int(yi.numel())
    algo = spmspv_bytes(At, xi, nnz_y)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    clocks = ClockSampler(local).start() if rank == 0 else None
    barrier(world, pg)
    torch.cuda.synchronize(device)
    t_wall0 = time.time()
    for i in range(args.steps):
        flush.fill_(i)  # write > L2 between timed steps (not timed)
        ev[i][0].record(stream)
        op(dxi, dxv)
        ev[i][1].record(stream)
    torch.cuda.synchronize(device)
    t_wall1 = time.time()
    barrier(world, pg)
    clk = clocks.stop(t_wall0, t_wall1) if clocks else None
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_s = reduce_max(sum(step_ms) / 1e3, world, pg, device)
    launches = op.plan_info()["numeric_launches"]
    e2e = None
    if args.e2e_steps > 0:
        hxi, hxv = torch.from_numpy(xi).pin_memory(), torch.from_numpy(xv).pin_memory()
        hyi = torch.empty(nnz_y, dtype=torch.int32).pin_memory()
        hyv = torch.empty(nnz_y, dtype=torch.float64).pin_memory()

        def e2e_step():
            yi2, yv2 = op(hxi.to(device, non_blocking=True), hxv.to(device, non_blocking=True))
            hyi.copy_(yi2, non_blocking=True)
            hyv.copy_(yv2, non_blocking=True)
            torch.cuda.synchronize(device)

        e2e_step()
        barrier(world, pg)
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            e2e_step()
        e2e_s = reduce_max(time.perf_counter() - t0, world, pg, device)
        e2e = {"value": round(algo * args.e2e_steps * world / e2e_s / 1e9, 3), "unit": "GB/s",
               "h2d_bytes_per_step": int(hxi.numel() * 4 + hxv.numel() * 8),
               "d2h_bytes_per_step": int(nnz_y * 12), "steps": args.e2e_steps,
               "note": "A stays resident (the operator); x is the step's input"}
    op.close()
    if rank != 0:
        return
    peaks = measured_peaks()
    value = algo * args.steps * world / total_s / 1e9
    base = None
    if args.cpu_baseline_s > 0:
        t0 = time.perf_counter()
        oracle_spmspv(A, xi, xv)
        dt = time.perf_counter() - t0
        base = {"value": round(algo / dt / 1e9, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
                "sample": f"whole product, {dt:.1f} s, numpy on one core"}
    line = {
        "metric": SPMSPV_METRIC, "value": round(value, 3), "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(1e3 * total_s / args.steps, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": args.workload, "description": SPMSPV_WORKLOADS[args.workload], "m": A.nrows,
                   "n": A.ncols, "nnz_a": int(A.colidx.size), "nnz_x": int(xi.size), "nnz_y": nnz_y,
                   "l2": "flushed between timed steps (write of a buffer > L2)",
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "phases_ms": {"step_min": round(min(step_ms), 4), "step_median": round(statistics.median(step_ms), 4)},
        "roofline": dict(roofline_obj(algo, statistics.mean(step_ms) / 1e3, peaks, None),
                         kernel="whole product (offsets, scan, scatter, tile counts, scan, write; read-back included)"),
        "gpu_launches": int(launches * args.steps),
        "clocks": clk, "e2e": e2e, "cpu_baseline": base,
    }
    print(json.dumps(line), flush=True)


def run_outer(args, world, rank, local, pg, A, B, dA, dB, ub, flush, stream, device) -> None:
    """The outer-product SpGEMM (k blocks, partial products, sparse-addition merge), timed whole."""
    import torch
    from paper_2606_20855_gb300.spgemm import spgemm_outer
    products = int(ub.sum())
    C = None
    for _ in range(args.warmup):
        C = spgemm_outer(dA, dB, args.parts)
    torch.cuda.synchronize(device)
    nnz = C.nnz if C is not None else 0
    stats = {}
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    clocks = ClockSampler(local).start() if rank == 0 else None
    barrier(world, pg)
    torch.cuda.synchronize(device)
    t_wall0 = time.time()
    for i in range(args.steps):
        flush.fill_(i)
        ev[i][0].record(stream)
        C = spgemm_outer(dA, dB, args.parts, stats=stats)
        ev[i][1].record(stream)
    torch.cuda.synchronize(device)
    t_wall1 = time.time()
    barrier(world, pg)
    clk = clocks.stop(t_wall0, t_wall1) if clocks else None
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_s = reduce_max(sum(step_ms) / 1e3, world, pg, device)
    if rank != 0:
        return
    s = A.vals.dtype.itemsize
    algo = csr_bytes(A.nrows, A.nnz, s) + csr_bytes(B.nrows, B.nnz, s) + csr_bytes(A.nrows, nnz, s)
    peaks = measured_peaks()
    value = 2.0 * products * args.steps * world / total_s / 1e9
    line = {
        "metric": METRIC, "value": round(value, 3), "unit": "GFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(1e3 * total_s / args.steps, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64" if s == 8 else "f32", "data": "synthetic",
        "config": {"workload": args.workload, "description": WORKLOADS[args.workload], "algo": "outer",
                   "parts": args.parts, "m": A.nrows, "k": A.ncols, "n": B.ncols, "nnz_c": int(nnz),
                   "products": products, "l2": "flushed between timed steps (write of a buffer > L2)",
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "effective_hbm_gbs": round(algo * args.steps * world / total_s / 1e9, 1),
        "phases_ms": {"step_min": round(min(step_ms), 4), "step_median": round(statistics.median(step_ms), 4)},
        "roofline": dict(roofline_obj(algo, statistics.mean(step_ms) / 1e3, peaks, None),
                         kernel=f"whole outer-product SpGEMM ({args.parts} k blocks inside the library: "
                                "column-block extraction, partial products, pairwise sparse additions; "
                                "read-backs included)"),
        "gpu_launches": int(stats.get("launches", 0)),
        "clocks": clk, "e2e": None, "cpu_baseline": None,
    }
    print(json.dumps(line), flush=True)


def time_steps(op, steps, flush, stream, device, world, pg, rank, local):
    """Times `steps` operations (symbolic with its read-back, a fresh C,
    numeric), the L2 flushed before each; returns per-step, symbolic and
    numeric milliseconds, the clock record and the max-over-ranks total."""
    import torch
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    clocks = ClockSampler(local).start() if rank == 0 else None
    barrier(world, pg)
    torch.cuda.synchronize(device)
    t_wall0 = time.time()
    for i in range(steps):
        flush.fill_(i)  # write > L2 between timed steps (not timed)
        e0, e1, e2 = ev[i]
        e0.record(stream)
        op.symbolic()
        e1.record(stream)
        C = op.numeric()  # C's arrays allocated inside the timed span
        e2.record(stream)
        op.wait()
        del C
    torch.cuda.synchronize(device)
    t_wall1 = time.time()
    barrier(world, pg)
    clk = clocks.stop(t_wall0, t_wall1) if clocks else None
    step_ms = [a.elapsed_time(c) for a, _, c in ev]
    sym_ms = [a.elapsed_time(b) for a, b, _ in ev]
    num_ms = [b.elapsed_time(c) for _, b, c in ev]
    total_s = reduce_max(sum(step_ms) / 1e3, world, pg, device)
    return step_ms, sym_ms, num_ms, clk, total_s


def e2e_measure(A, B, make_op, same, device, steps, world, pg, nnz, algo_bytes, ew, products):
    """The operation through the public Python API from pinned host inputs to
    the host copy of C, copies inside the timed region."""
    import torch
    from paper_2606_20855_gb300.spgemm import DeviceCSR
    hA = [torch.from_numpy(a).pin_memory() for a in (A.rowptr, A.colidx, A.vals)]
    hB = hA if same else [torch.from_numpy(a).pin_memory() for a in (B.rowptr, B.colidx, B.vals)]
    h_col = torch.empty(nnz, dtype=torch.int32).pin_memory()
    h_val = torch.empty(nnz, dtype=hA[2].dtype).pin_memory()
    h_rp = torch.empty(A.nrows + 1, dtype=torch.int64).pin_memory()

    def e2e_step():
        tA = DeviceCSR(A.nrows, A.ncols, *[t.to(device, non_blocking=True) for t in hA])
        tB = tA if same else DeviceCSR(B.nrows, B.ncols, *[t.to(device, non_blocking=True) for t in hB])
        with make_op(tA, tB) as op2:
            op2.symbolic()
            C = op2.numeric()
            h_rp.copy_(C.rowptr, non_blocking=True)
            h_col.copy_(C.colidx, non_blocking=True)
            h_val.copy_(C.vals, non_blocking=True)
            op2.wait()
        torch.cuda.synchronize(device)

    e2e_step()
    barrier(world, pg)
    # Each step timed on its own (host clock around a synchronised step): the
    # host-link copies now and then take several times their usual time, so
    # the value uses the median step; mean and slowest are reported beside it.
    step_s = []
    for _ in range(steps):
        t0 = time.perf_counter()
        e2e_step()
        step_s.append(time.perf_counter() - t0)
    med_s = reduce_max(statistics.median(step_s), world, pg, device)
    mean_s = reduce_max(statistics.fmean(step_s), world, pg, device)
    max_s = reduce_max(max(step_s), world, pg, device)
    h2d = sum(t.numel() * t.element_size() for t in hA) + (0 if same else sum(t.numel() * t.element_size() for t in hB))
    d2h = h_rp.numel() * 8 + h_col.numel() * 4 + h_val.numel() * h_val.element_size()
    work = algo_bytes if ew else 2.0 * float(products)
    # The host link alone: the device-to-host copy of C's arrays from a device
    # buffer to the same pinned buffers (copy engines), timed by itself.
    dcol = torch.empty(max(nnz, 1), dtype=torch.int32, device=device)
    dval = torch.empty(max(nnz, 1), dtype=h_val.dtype, device=device)
    torch.cuda.synchronize(device)
    t0 = time.perf_counter()
    h_col.copy_(dcol[:nnz], non_blocking=True)
    h_val.copy_(dval[:nnz], non_blocking=True)
    torch.cuda.synchronize(device)
    copy_s = time.perf_counter() - t0
    del dcol, dval
    link_gbs = (h_col.numel() * 4 + h_val.numel() * h_val.element_size()) / max(copy_s, 1e-9) / 1e9
    return {"value": round(work * world / med_s / 1e9, 3), "unit": "GB/s" if ew else "GFLOP/s",
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": steps,
            "ms_per_step": round(1e3 * med_s, 3), "statistic": "median step",
            "ms_per_step_mean": round(1e3 * mean_s, 3), "ms_per_step_max": round(1e3 * max_s, 3),
            "host_link": {"d2h_gbs": round(link_gbs, 1),
                          "c_copy_ms": round(1e3 * copy_s, 3),
                          "c_copy_share_of_step": round(copy_s / med_s, 3),
                          "note": "device-to-host copy of C's arrays alone, pinned host memory"}}


def measure(args, name, A, B, steps, warmup, e2e_steps, cpu_s, world, rank, local, pg, min_region_s=0.0,
            with_traffic=False):
    """One workload: the timed steps, the roofline of the whole operation and
    of each pass, end to end and the CPU oracle.  With min_region_s > 0 the
    step count grows until the timed region lasts at least that long."""
    import torch
    from paper_2606_20855_gb300.spgemm import DeviceCSR, Ewise, SpGEMM

    device = torch.device(f"cuda:{local}")
    stream = torch.cuda.current_stream(device)
    same = B is A
    ew = name in EWISE_WORKLOADS
    ub = np.zeros(A.nrows, dtype=np.int64) if ew else products_per_row(A, B)
    products = int(ub.sum())
    make_op = (lambda x, y: Ewise(x, y, args.op)) if ew else SpGEMM
    s = 8 if A.vals.dtype == np.float64 else 4

    dA = DeviceCSR.from_host(A, device)
    dB = dA if same else DeviceCSR.from_host(B, device)
    l2 = torch.cuda.get_device_properties(device).L2_cache_size
    flush = torch.empty(max(2 * l2, 256 << 20) // 4, dtype=torch.int32, device=device)
    op = make_op(dA, dB)
    t0 = time.perf_counter()
    for _ in range(max(warmup, 1) if min_region_s > 0 else warmup):
        op.symbolic()
        C = op.numeric()
        op.wait()
        del C
    torch.cuda.synchronize(device)
    if min_region_s > 0:  # size the timed region from the warm-up's wall time (slowest rank)
        per = reduce_max((time.perf_counter() - t0) / max(warmup, 1), world, pg, device)
        steps = max(steps, min(20000, int(np.ceil(1.2 * min_region_s / max(per, 1e-6)))))
    nnz = op.nnz
    info = op.plan_info()
    algo_bytes = csr_bytes(A.nrows, A.nnz, s) + csr_bytes(B.nrows, B.nnz, s) + csr_bytes(A.nrows, nnz, s)
    # symbolic pass: read the structure of A and B once, write C.rowptr
    sym_bytes = csr_bytes(A.nrows, A.nnz, 0) + csr_bytes(B.nrows, B.nnz, 0) + 8 * (A.nrows + 1)
    step_ms, sym_ms, num_ms, clk, total_s = time_steps(op, steps, flush, stream, device, world, pg, rank, local)
    launches_per_step = info["symbolic_launches"] + info["numeric_launches"]
    op.close()
    del op, flush
    e2e = None
    if e2e_steps > 0:
        e2e = e2e_measure(A, B, make_op, same, device, e2e_steps, world, pg, nnz, algo_bytes, ew, products)
    del dA, dB
    torch.cuda.empty_cache()
    if rank != 0:
        return None
    peaks = measured_peaks()
    eff_gbs = algo_bytes * steps * world / total_s / 1e9
    value = eff_gbs if ew else 2.0 * products * steps * world / total_s / 1e9
    base = None
    if cpu_s > 0:
        if ew:
            dt, _ = ewise_oracle_timed(A, B, args.op, 1)
            base = {"value": round(algo_bytes / dt / 1e9, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
                    "sample": f"whole operation, {dt:.1f} s, numpy on one core"}
        else:
            base = cpu_baseline(A, B, ub, cpu_s)
    traffic = {"symbolic": None, "numeric": None}
    if with_traffic and not ew and not args.rows:
        traffic = {k: recorded_traffic(name, kern) for k, kern in PASS_KERNELS.items()}
    whole_traffic = (None if traffic["symbolic"] is None or traffic["numeric"] is None
                     else traffic["symbolic"] + traffic["numeric"])
    return {
        "workload": name if not args.rows else f"{name}[:{A.nrows} rows]",
        "description": EWISE_WORKLOADS[name] if ew else WORKLOADS[name],
        "value": round(value, 3), "unit": "GB/s" if ew else "GFLOP/s",
        "ms_per_step": round(1e3 * total_s / steps, 4), "steps": steps, "warmup": warmup,
        "dtype": "f64" if s == 8 else "f32",
        "m": A.nrows, "k": A.ncols, "n": B.ncols, "nnz_a": A.nnz, "nnz_b": B.nnz, "nnz_c": int(nnz),
        **({"op": args.op} if ew else {"products": products}),
        "effective_hbm_gbs": round(eff_gbs, 1),
        "frac_of_8tbs": round(eff_gbs / NOMINAL_HBM_GBS, 4),
        "phases_ms": {"symbolic_median": round(statistics.median(sym_ms), 4),
                      "numeric_median": round(statistics.median(num_ms), 4),
                      "step_min": round(min(step_ms), 4), "step_median": round(statistics.median(step_ms), 4)},
        "roofline": dict(roofline_obj(algo_bytes, statistics.mean(step_ms) / 1e3, peaks, whole_traffic),
                         kernel=("whole operation" if ew else "whole product") +
                                ": symbolic pass (nnz read-back included) + numeric pass",
                         passes={
                             "symbolic": dict(roofline_obj(sym_bytes, statistics.mean(sym_ms) / 1e3, peaks,
                                                           traffic["symbolic"]),
                                              kernel="symbolic pass (compulsory bytes: structure of A and B "
                                                     "read once, C.rowptr written)"),
                             "numeric": dict(roofline_obj(algo_bytes, statistics.mean(num_ms) / 1e3, peaks,
                                                          traffic["numeric"]),
                                             kernel="numeric pass: " + ("ew_merge_kernel" if ew else
                                                                            numeric_kernels(info))),
                         }),
        "gpu_launches": int(launches_per_step * steps),
        "plan": info,
        "clocks": clk,
        "e2e": e2e,
        "cpu_baseline": base,
        "_total_s": total_s,
    }


def run_ours(args, world, rank, local, pg) -> None:
    import torch
    from paper_2606_20855_gb300 import _abi

    _abi.load()
    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    A, B = load_workload(args)
    ew = is_ewise(args)
    if args.algo == "outer" and not ew:
        from paper_2606_20855_gb300.spgemm import DeviceCSR
        s_dev = torch.cuda.current_stream(device)
        l2 = torch.cuda.get_device_properties(device).L2_cache_size
        flush = torch.empty(max(2 * l2, 256 << 20) // 4, dtype=torch.int32, device=device)
        dA = DeviceCSR.from_host(A, device)
        dB = dA if B is A else DeviceCSR.from_host(B, device)
        run_outer(args, world, rank, local, pg, A, B, dA, dB, products_per_row(A, B), flush, s_dev, device)
        return
    head = measure(args, args.workload, A, B, args.steps, args.warmup, args.e2e_steps, args.cpu_baseline_s,
                   world, rank, local, pg, with_traffic=True)
    # The headline product again over at least one second, with its own clock record.
    sustained = None
    if not ew and not args.rows and args.sustained_s > 0:
        sus = measure(args, args.workload, A, B, args.steps, args.warmup, 0, 0, world, rank, local, pg,
                      min_region_s=args.sustained_s)
        if rank == 0:
            sustained = {"steps": sus["steps"], "ms_per_step": sus["ms_per_step"], "value": sus["value"],
                         "unit": sus["unit"], "timed_region_s": round(sus["_total_s"], 3), "clocks": sus["clocks"]}
    # Every named SpGEMM workload (the five configurations of the headline metric), on a single GPU.
    per_config = None
    if args.per_config and not ew and not args.rows and world == 1:
        per_config = {}
        for name in WORKLOAD_ORDER:
            if name == args.workload:
                e = head
            else:
                A2, B2 = workload(name)
                e = measure(args, name, A2, B2, args.steps, args.warmup, args.e2e_steps, args.per_config_cpu_s,
                            world, rank, local, pg, min_region_s=args.per_config_s)
                del A2, B2
            if rank == 0:
                per_config[name] = {k: e[k] for k in ("value", "unit", "ms_per_step", "steps", "dtype", "products",
                                                      "nnz_c", "effective_hbm_gbs", "frac_of_8tbs", "phases_ms",
                                                      "roofline", "gpu_launches", "clocks", "e2e", "cpu_baseline")}
    if rank != 0:
        return
    line = {
        "metric": EWISE_METRIC if ew else METRIC,
        "value": head["value"],
        "unit": head["unit"],
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": head["ms_per_step"],
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": head["dtype"],
        "data": "synthetic",
        "config": {
            "workload": head["workload"], "description": head["description"],
            "m": head["m"], "k": head["k"], "n": head["n"], "nnz_a": head["nnz_a"], "nnz_b": head["nnz_b"],
            "nnz_c": head["nnz_c"], **({"op": args.op} if ew else {"products": head["products"]}),
            "l2": "flushed between timed steps (write of a buffer > L2)",
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
        },
        "effective_hbm_gbs": head["effective_hbm_gbs"],
        "frac_of_8tbs": head["frac_of_8tbs"],
        "phases_ms": head["phases_ms"],
        "roofline": head["roofline"],
        "gpu_launches": head["gpu_launches"],
        "plan": head["plan"],
        "clocks": head["clocks"],
        "e2e": head["e2e"],
        "cpu_baseline": head["cpu_baseline"],
    }
    if sustained is not None:
        line["sustained"] = sustained
    if per_config is not None:
        line["per_config"] = per_config
    print(json.dumps(line), flush=True)


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=list(WORKLOADS) + list(EWISE_WORKLOADS) + list(SPMSPV_WORKLOADS),
                    default=DEFAULT_WORKLOAD)
    ap.add_argument("--op", choices=["add", "mul"], default="add", help="elementwise workloads: C = A + B or A .* B")
    ap.add_argument("--algo", choices=["gustavson", "outer"], default="gustavson",
                    help="SpGEMM workloads: row-wise (default) or the outer-product variant")
    ap.add_argument("--parts", type=int, default=4, help="k blocks of the outer-product variant")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--cpu-baseline-s", type=float, default=12.0, help="seconds of CPU oracle work (0 = skip)")
    ap.add_argument("--ref-step-s", type=float, default=2.0, help="seconds per reference-arm step")
    ap.add_argument("--rows", type=int, default=0,
                    help="use only the first ROWS rows of A (a smaller case of the same workload, for profiling)")
    ap.add_argument("--per-config", dest="per_config", action="store_true", default=None,
                    help="also measure every named SpGEMM workload (default: on without --workload)")
    ap.add_argument("--no-per-config", dest="per_config", action="store_false")
    ap.add_argument("--per-config-s", type=float, default=0.5, help="least seconds of timed steps per workload")
    ap.add_argument("--per-config-cpu-s", type=float, default=3.0, help="seconds of CPU oracle work per workload")
    ap.add_argument("--sustained-s", type=float, default=1.0,
                    help="least seconds of the headline's second timed region (0 = skip)")
    args = ap.parse_args(argv)
    if args.per_config is None:
        args.per_config = args.workload == DEFAULT_WORKLOAD and "--workload" not in (argv or sys.argv[1:])
    world, rank, local, pg = dist_setup()
    try:
        if args.workload in SPMSPV_WORKLOADS:
            run_spmspv(args, world, rank, local, pg)
        elif args.impl == "reference":
            run_reference(args, world, rank)
        else:
            run_ours(args, world, rank, local, pg)
    finally:
        if pg is not None:
            pg.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
