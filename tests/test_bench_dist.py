"""The multi-rank path of bench.py on CPU: two gloo ranks (no GPU, no NCCL).

The benchmark shards over images with no exchange in the data path; its only collectives are the
timing barrier and the max over ranks of the measured times, and the reference arm runs on rank 0
alone.  Both are exercised here with world size 2."""
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


def _rank(rank, world, port, out_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = [10.0 + rank, 5.0 - rank, 7.0 + 2 * rank]   # elapsed, e2e, graph on this rank
        got = bench.max_over_ranks(dist, mine, torch.device("cpu"))
        dist.barrier()
        with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
            json.dump(got, f)
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo(tmp_path):
    world = 2
    mp.spawn(_rank, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    res = [json.load(open(tmp_path / f"r{r}.json")) for r in range(world)]
    assert res[0] == res[1] == [11.0, 5.0, 9.0]     # every rank sees the slowest rank's times


def test_max_over_ranks_without_group():
    assert bench.max_over_ranks(None, [1, 2.5], None) == [1.0, 2.5]


def test_job_throughput_is_weak_scaling():
    one = bench.job_images_per_s(1, 10.0)
    assert one == pytest.approx(bench.BATCH / 0.01)
    assert bench.job_images_per_s(4, 10.0) == pytest.approx(4 * one)


def test_reference_arm_under_torchrun_two_ranks():
    """`--impl reference` under torchrun: rank 0 times the oracle and prints one JSON line, the
    other rank exits 0 without work."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--steps", "1",
           "--warmup", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="2")
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
