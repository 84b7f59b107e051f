"""The bench's multi-rank path on the CPU: two gloo ranks, no GPU.

The pruning stage shards by request with no exchange, so N GPUs run N independent
replicas; the only collectives are the timing max over ranks and the barriers. These
tests run that host logic with world_size 2 over gloo (127.0.0.1), and the reference
arm under torchrun, where rank 0 alone works and prints.
"""
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

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        # rank r took 5 * (r + 1) ms for 10 steps of 100 units: the job's rate uses the slowest rank
        rate, ms_step = bench.whole_job_rate(100, 10, 5.0 * (rank + 1), world)
        bench.barrier(world)
        out.put((rank, rate, ms_step))
    finally:
        dist.destroy_process_group()


def test_whole_job_rate_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
        assert p.exitcode == 0
    results = sorted(out.get(timeout=10) for _ in range(2))
    for rank, rate, ms_step in results:
        assert ms_step == pytest.approx(1.0)                       # the slowest rank: 10 ms / 10 steps
        assert rate == pytest.approx(100 * 10 * 2 / 10e-3)         # both ranks' units over that time


def test_whole_job_rate_single_process():
    sys.path.insert(0, ROOT)
    import bench

    rate, ms_step = bench.whole_job_rate(7, 4, 2.0, 1)
    assert ms_step == pytest.approx(0.5) and rate == pytest.approx(7 * 4 / 2e-3)


def test_reference_arm_under_torchrun_two_ranks():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--config", "tiny", "--steps", "1", "--warmup", "3"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    res = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, res.stdout  # rank 0 alone prints
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["cpu_baseline"]["kind"] == "oracle"
