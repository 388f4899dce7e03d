"""The multi-rank path of bench.py on CPU: two gloo ranks, launched the way the
benchmark launches one process per GPU.  The layer shards along the batch
(independent images), so ranks exchange only the timing: a barrier around the
timed region and the maximum over ranks of its duration."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    import bench
    import torch.distributed as dist
    w, r, local = bench.dist_setup()
    assert (w, r, local) == (world, rank, rank)
    assert dist.get_backend() == "gloo"
    bench.barrier(w)
    t_local = 1.0 + 0.5 * rank  # the slower rank sets the job time
    t_max = bench.max_over_ranks(t_local, w)
    rate = bench.whole_job_rate(units_per_rank_step=100.0, world=w, steps=10, t_max=t_max)
    bench.barrier(w)
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump({"t_max": t_max, "rate": rate}, f)
    dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_slowest_time(tmp_path):
    world = 2
    mp.spawn(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    got = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    for g in got:
        assert g["t_max"] == pytest.approx(1.5)
        # whole job: both ranks' 10 steps of 100 units in the slowest rank's 1.5 s
        assert g["rate"] == pytest.approx(2 * 100 * 10 / 1.5)


def test_reference_arm_runs_on_rank_zero_only():
    """Under a multi-rank launch the oracle arm does its work on rank 0; other ranks exit 0 silently."""
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", MASTER_ADDR="127.0.0.1", MASTER_PORT="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""


def test_whole_job_rate_is_weak_scaling():
    import bench
    # N ranks, each with its own shard of the same size, in the same time: N times the units per second
    one = bench.whole_job_rate(2.0e9, 1, 50, 0.01)
    assert bench.whole_job_rate(2.0e9, 4, 50, 0.01) == pytest.approx(4 * one)
    # a slower rank lowers the whole-job rate
    assert bench.whole_job_rate(2.0e9, 4, 50, 0.02) == pytest.approx(2 * one)
