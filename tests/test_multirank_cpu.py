"""The N > 1 host paths of bench.py, exercised as world-size-2 `gloo` ranks on the CPU:
the job's time is the slowest rank's (max over ranks), and under torchrun the reference
arm runs and prints on rank 0 only while the other ranks exit without work."""
from __future__ import annotations

import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        out.put((rank, bench.max_over_ranks(10.0 + 5.0 * rank)))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = dict(out.get(timeout=10) for _ in range(2))
    assert got == {0: 15.0, 1: 15.0}


def test_max_over_ranks_without_group_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5) == 3.5


def test_reference_arm_under_torchrun_prints_on_rank0_only():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "1", "--cpu-seconds", "1"]
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, res.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference"
    assert line["n_gpus"] == 2 and line["unit"] == "vehicle-ticks/s" and line["value"] > 0
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["cpu_baseline"]["kind"] == "oracle"


def test_append_reference_arm_prints_one_line():
    """The cache-append workload's reference arm: the fp64 append oracle on the host cores
    (one backbone layer here to keep the CPU suite short)."""
    cmd = [sys.executable, "bench.py", "--impl", "reference", "--workload", "append_b1_l224", "--layers", "1",
           "--steps", "1", "--warmup", "1", "--cpu-seconds", "1"]
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, res.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["unit"] == "vehicle-appends/s" and line["value"] > 0
    assert line["config"]["workload"] == "append_b1_l224" and line["config"]["layers"] == 1
    assert line["cpu_baseline"]["kind"] == "oracle"


def test_clip_reference_arm_prints_one_line():
    """The staleness-masked clip workload's reference arm (two expert layers here)."""
    cmd = [sys.executable, "bench.py", "--impl", "reference", "--workload", "clip_j40_delta1", "--layers", "2",
           "--steps", "1", "--warmup", "1", "--cpu-seconds", "1"]
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, res.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["unit"] == "frame-blocks/s" and line["value"] > 0
    assert line["config"]["frames"] == 40 and line["config"]["delta"] == 1


def test_gpus_flag_without_torchrun_starts_the_ranks_itself():
    """`bench.py --gpus 2` outside torchrun starts two ranks with the rank environment
    torchrun would give them; the reference arm then prints one line, from rank 0."""
    env = {k: v for k, v in os.environ.items() if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK")}
    cmd = [sys.executable, "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "1",
           "--cpu-seconds", "1"]
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, res.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["config"]["parallelism"] == "replicas x2"
    assert line["config"]["workload"] == "bf16_b128_ragged" and line["config"]["B"] == 128


def test_cpu_baseline_sample_spans_the_length_order():
    sys.path.insert(0, ROOT)
    import numpy as np
    import bench
    lengths = np.array([300, 70, 2048, 900, 64, 1500, 1200, 400, 999, 1800])
    picks = bench.baseline_vehicles(lengths)
    assert len(picks) == 8 and len(set(picks)) == 8
    assert int(np.argmin(lengths)) in picks and int(np.argmax(lengths)) in picks
    assert bench.baseline_vehicles([224]) == [0]


def test_paper_layout_reference_arm_prints_one_line():
    """The ten-token workload's reference arm: its fp64 oracle (one expert layer here)."""
    cmd = [sys.executable, "bench.py", "--impl", "reference", "--workload", "paper_b1_l224", "--layers", "1",
           "--steps", "1", "--warmup", "1", "--cpu-seconds", "1"]
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, res.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["config"]["workload"] == "paper_b1_l224" and line["config"]["tokens_per_vehicle"] == 10
