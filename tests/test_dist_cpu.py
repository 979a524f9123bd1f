"""The multi-process path of bench.py on CPU: world_size 2 over gloo.

The method has no exchange step (requests are independent, weights
replicated), so N GPUs run N replicas: the ranks meet only at the barrier
around the timed region and in the max of their times, and rank 0 alone
prints.  These tests run that plumbing as two CPU processes.
"""
import os
import socket
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update({"RANK": str(rank), "LOCAL_RANK": str(rank), "WORLD_SIZE": str(world),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                       "LSP_DIST_BACKEND": "gloo"})
    sys.path.insert(0, ROOT)
    import bench
    dist = bench.Dist()
    try:
        assert dist.world == world and dist.rank == rank and dist.pg is not None
        dist.barrier()
        # each rank's time differs; every rank must see the slowest
        t = dist.max(1.5 * (rank + 1))
        # the reference arm: only rank 0 does work under torchrun
        ran = bench.run_reference(None, dist) if rank != 0 else "skipped"
        dist.barrier()
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(f"{t} {ran}\n")
    finally:
        dist.close()


@pytest.mark.timeout(180)
def test_replicas_barrier_and_max_over_two_gloo_ranks(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    for r in range(world):
        t, ran = open(tmp_path / f"rank{r}.txt").read().split()
        assert float(t) == 3.0                        # max over ranks, seen by every rank
        assert ran == ("None" if r else "skipped")    # rank 1 returned without work


def test_whole_job_throughput_is_the_sum_over_replicas():
    """value = world x C x B / (max-over-ranks ms): weak scaling over replicas."""
    sys.path.insert(0, ROOT)
    import bench
    assert bench.job_throughput(1, 16, 16, 1.25) == pytest.approx(256 / 1.25e-3)
    assert bench.job_throughput(4, 16, 16, 1.25) == pytest.approx(4 * 256 / 1.25e-3)
