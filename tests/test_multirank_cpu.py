"""The N > 1 path of bench.py on the CPU: world_size 2 over gloo.

The GPU path has no data-path collective (each rank runs an independent
replica of the workload); the only exchange is the max over ranks of the
timed regions, and the whole-job value adds every rank's units.  The
reference arm runs on rank 0 only; other ranks exit without work.
"""

import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    # rank r's timed regions: ms = 10 + 5 r, e2e = 30 - r
    got = bench.max_over_ranks([10.0 + 5 * rank, 30.0 - rank], "cpu")
    dist.barrier()
    dist.destroy_process_group()
    with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
        json.dump(got, f)


def test_max_over_ranks_gloo(tmp_path):
    import torch.multiprocessing as mp
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, str(tmp_path)), nprocs=2, start_method="spawn")
    for r in range(2):
        got = json.load(open(tmp_path / f"r{r}.json"))
        assert got == [15.0, 30.0]      # every rank gets the slowest rank's times


def test_whole_job_value_adds_ranks():
    sys.path.insert(0, ROOT)
    import bench
    one = bench.whole_job_value(1, 6, 100, 15, 128, 50.0)
    assert one == pytest.approx(6 * 100 * 15 * 128 / 0.05)
    assert bench.whole_job_value(4, 6, 100, 15, 128, 50.0) == pytest.approx(4 * one)


def test_reference_arm_other_ranks_exit_without_work():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--workload", "small", "--steps", "1", "--warmup", "0"],
                       env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0
    assert r.stdout.strip() == ""
