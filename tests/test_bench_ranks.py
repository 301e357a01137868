"""The benchmark's multi-rank host logic on CPU: gloo process groups of two
ranks (the GPU path uses the same helpers over NCCL)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms, e2e = bench.reduce_max([1.0 + rank, 5.0 - rank], dist, torch.device("cpu"))
    out[rank] = (ms, e2e, bench.job_throughput(2.0, world, ms))
    dist.barrier()
    dist.destroy_process_group()


def test_reduce_max_and_job_throughput_two_gloo_ranks():
    port = _free_port()
    out = mp.get_context("spawn").Manager().dict()
    mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
    for rank in range(2):
        ms, e2e, value = out[rank]
        assert ms == 2.0 and e2e == 5.0          # the slowest rank's time, on every rank
        assert value == pytest.approx(2.0 * 2 / 2e-3)


def test_single_process_is_identity():
    assert bench.reduce_max([3.0, 4.0], None, None) == [3.0, 4.0]
    assert bench.job_throughput(1.0, 1, 1.0) == pytest.approx(1000.0)


def test_reference_arm_under_torchrun_prints_one_line_from_rank0():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0", "--ref-step-s", "0.5"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
