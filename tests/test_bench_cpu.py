"""bench.py host logic on the CPU: the reference (oracle) arm, its JSON line, and
the multi-rank path (torchrun with world size 2 over gloo: rank 0 prints one
line, the other rank exits cleanly; max-over-ranks reduction)."""
from __future__ import annotations

import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _json_lines(out: str):
    return [json.loads(ln) for ln in out.splitlines() if ln.startswith("{")]


def test_reference_arm_json_line():
    cmd = [sys.executable, "bench.py", "--impl", "reference", "--workload", "uniform_2k", "--steps", "2",
           "--warmup", "1", "--ref-step-s", "0.2"]
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert res.returncode == 0, res.stderr
    lines = _json_lines(res.stdout)
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 1
    assert d["value"] > 0 and d["unit"] == "GFLOP/s" and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["config"]["workload"] == "uniform_2k"


@pytest.mark.slow
def test_reference_arm_two_ranks_gloo():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference",
           "--gpus", "2", "--workload", "uniform_2k", "--steps", "1", "--warmup", "0", "--ref-step-s", "0.2"]
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300, env=env)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = _json_lines(res.stdout)
    assert len(lines) == 1 and lines[0]["impl"] == "reference" and lines[0]["n_gpus"] == 2


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo")
    try:
        bench.barrier(world, dist)
        q.put((rank, bench.reduce_max(float(rank + 1) * 1.5, world, dist, "cpu")))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert out == {0: 3.0, 1: 3.0}


def test_traffic_records_follow_the_kernel_source(tmp_path, monkeypatch):
    """roofline.traffic comes from a `traffic-record:` line of a profile
    summary, scaled from the captured rows to the full workload, and is None
    once the kernel source no longer matches the recorded digest."""
    sys.path.insert(0, ROOT)
    import bench

    src = tmp_path / "kern.cu"
    src.write_text("// kernel v1\n")
    prof = tmp_path / "profiles"
    prof.mkdir()
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "PROFILES", str(prof))
    digest = bench.source_digest("kern.cu")
    assert digest is not None and len(digest) == 16
    (prof / "k.md").write_text(
        "# capture\n\ntraffic-record: workload=w kernel=k_kernel rows=100 of=400 dram_bytes=2.5e6 "
        f"source=kern.cu sha256={digest}\n")
    assert bench.recorded_traffic("w", "k_kernel") == 1e7
    assert bench.recorded_traffic("w", "other_kernel") is None
    assert bench.recorded_traffic("other", "k_kernel") is None
    src.write_text("// kernel v2\n")  # the kernel changed after the capture
    assert bench.recorded_traffic("w", "k_kernel") is None
