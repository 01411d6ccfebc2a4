"""Multi-rank host logic on CPU (gloo, world size 2): the replica helpers that
the GPU arm runs over NCCL, and the reference arm of bench.py under torchrun
(rank 0 alone works and prints; the other rank exits 0)."""
from __future__ import annotations

import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2608_01784_gb300 import replicas as R

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank: int, world: int, port: int, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    ri = R.rank_info()
    R.init(ri.world, "gloo")
    try:
        R.barrier(ri.world)
        # slowest rank decides the time
        ms = R.max_over_ranks(1.5 + ri.rank, ri.world)
        out.put((ri.rank, ri.world, ri.local_rank, R.rank_seed(7, ri.rank), ms,
                 R.whole_job_rate(1024, ri.world, ms)))
    finally:
        R.finalize(ri.world)


def test_replicas_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [g[0] for g in got] == [0, 1]
    assert all(g[1] == 2 for g in got)
    assert [g[2] for g in got] == [0, 1]
    assert [g[3] for g in got] == [7, 8]          # distinct batches per rank
    assert all(g[4] == 2.5 for g in got)          # max over ranks, on every rank
    assert all(g[5] == pytest.approx(2 * 1024 / 2.5e-3) for g in got)


def test_single_rank_helpers():
    assert R.rank_info({}) == R.RankInfo(0, 1, 0)
    assert R.max_over_ranks(3.25, 1) == 3.25
    assert R.rank_seed(5, 0) == 5
    assert R.whole_job_rate(10, 1, 1.0) == pytest.approx(1e4)


def test_reference_arm_torchrun_world2():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
           "--nproc-per-node", "2", "--master-addr", "127.0.0.1",
           "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "1",
           "--config", "tiny_fp32"]
    env = dict(os.environ, OMP_NUM_THREADS="2")
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [json.loads(l) for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1                         # rank 0 only
    line = lines[0]
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["value"] > 0 and line["e2e"]["h2d_bytes_per_step"] == 0
    assert line["cpu_baseline"]["kind"] == "oracle"
