"""The multi-replica path of bench.py on two CPU ranks (gloo): each rank
times its own replica; the job's time is the slowest rank's, its value
counts the tokens of every rank, and the reference arm runs on rank 0 only
(the other ranks return without work). No GPU: the aggregation is the same
code bench.py runs under torchrun with NCCL, given a CPU device."""

import os
import sys
import tempfile

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, init_file, out_dir):
    sys.path.insert(0, ROOT)
    import bench

    dist.init_process_group("gloo", init_method=f"file://{init_file}", rank=rank, world_size=world)
    try:
        dist.barrier()
        local_ms = 10.0 + 5.0 * rank  # rank 1 is the slower replica
        ms = bench.max_over_ranks(local_ms, "cpu", world)
        value = bench.job_tokens_per_s(16384, world, ms)

        class Args:
            steps = 1
            warmup = 0

        ref = bench.run_reference(Args(), rank, world) if rank != 0 else None
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(f"{ms} {value} {ref}\n")
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_rank_aggregation_and_rank0_only_reference():
    world = 2
    with tempfile.TemporaryDirectory() as d:
        init_file = os.path.join(d, "rendezvous")
        mp.start_processes(_worker, args=(world, init_file, d), nprocs=world, start_method="spawn", join=True)
        res = [open(os.path.join(d, f"rank{r}.txt")).read().split() for r in range(world)]
    for r in range(world):
        ms, value, ref = float(res[r][0]), float(res[r][1]), res[r][2]
        assert ms == 15.0  # the slowest rank's time, on every rank
        assert value == pytest.approx(2 * 16384 / 0.015)  # tokens of both replicas
    assert res[1][2] == "None"  # a non-zero rank of the reference arm does no work


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(7.5, "cpu", 1) == 7.5
    assert bench.job_tokens_per_s(1000, 1, 2.0) == pytest.approx(5e5)
