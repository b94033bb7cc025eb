"""The multi-rank path of the benchmark on CPU: two gloo ranks, 127.0.0.1.

With N GPUs every rank runs its own replica of the workload (the path shards
by sequence and exchanges nothing); the job's time is the slowest rank's and
its throughput counts every rank's queries.  No GPU is needed: the reduction
and the whole-job formula are host logic."""

import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, times, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        t = bench.max_over_ranks(times[rank], world, "cpu")
        out[rank] = (t, bench.job_throughput(world, 16, 30, t), bench.rank_seed(7, rank))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time_and_count_every_rank():
    mgr = mp.Manager()
    out = mgr.dict()
    times = [12.5, 17.25]  # ms of K = 30 steps on each rank
    mp.spawn(_rank_main, args=(2, _free_port(), times, out), nprocs=2, join=True)
    for r in range(2):
        t, value, seed = out[r]
        assert t == pytest.approx(17.25)
        # 2 ranks x 16 queries x 30 steps in 17.25 ms
        assert value == pytest.approx(2 * 16 * 30 / 17.25e-3)
    assert out[0][2] != out[1][2]  # each rank decodes its own data


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks(3.0, 1, "cpu") == 3.0
    assert bench.job_throughput(1, 8, 10, 2.0) == pytest.approx(8 * 10 / 2e-3)


def test_both_bench_arms_report_the_same_config():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2607_24331_gb300 import synth as S

    for cfg in (1, 4):
        c = bench.workload_config(S.workload(cfg), 2)
        assert c["workload"] == S.workload(cfg).name and c["parallelism"] == "replicas x2"
        assert set(c) == {"workload", "batch", "context", "layers", "step", "l2", "parallelism"}
