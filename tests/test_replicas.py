"""The N > 1 path of bench.py (replicas only: one independent solve per GPU, no data-path
collective) on CPU: two gloo ranks take the slowest replica's time and report the
whole-job aggregate; the reference arm runs on rank 0 alone."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

from conftest import ROOT


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, outdir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    import bench
    ms = bench.max_over_ranks(100.0 + 50.0 * rank, dist, "cpu")   # rank 1 is the slow replica
    dist.barrier()
    with open(os.path.join(outdir, "rank%d.json" % rank), "w") as f:
        json.dump([ms, bench.whole_job_rate(world, 3.0e12, ms)], f)
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_replica(tmp_path):
    world = 2
    mp.spawn(_rank, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)  # spawn, not fork
    res = {}
    for r in range(world):
        with open(tmp_path / ("rank%d.json" % r)) as f:
            res[r] = tuple(json.load(f))
    assert res[0] == res[1]                       # every rank agrees
    ms, rate = res[0]
    assert ms == 150.0                            # the max over ranks
    assert rate == pytest.approx(2 * 3.0e12 / 0.150, rel=1e-15)


def test_single_process_needs_no_collective():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(12.5, None, "cpu") == 12.5
    assert bench.whole_job_rate(1, 1.0e9, 500.0) == 2.0e9


def _run_reference(rank, world):
    env = dict(os.environ, RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                           "--config", "normal_d1024_s8", "--steps", "1", "--warmup", "0", "--gpus", str(world)],
                          capture_output=True, text=True, env=env, timeout=600)


def test_reference_arm_runs_on_rank_zero_only():
    r = _run_reference(1, 2)
    assert r.returncode == 0 and r.stdout.strip() == ""
    r = _run_reference(0, 2)
    assert r.returncode == 0
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["value"] > 0
