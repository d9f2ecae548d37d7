"""The multi-GPU path of bench.py is independent replicas: the only
cross-rank step is the max-reduction of the timing.  Checked here with two
gloo ranks on CPU (no GPU)."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench

        seconds = [2.0, 5.0][rank]                 # rank 1 is the slower replica
        rate, slowest = bench.whole_job_rate(seconds, local_queries=100, world=world, device="cpu")
        results[rank] = (rate, slowest)
        bench.barrier(world)
    finally:
        dist.destroy_process_group()


def test_two_replicas_report_the_whole_job_over_the_slowest_rank():
    world = 2
    port = _free_port()
    with mp.Manager() as manager:
        results = manager.dict()
        mp.spawn(_rank, args=(world, port, results), nprocs=world, join=True)
        for rank in range(world):
            rate, slowest = results[rank]
            assert slowest == pytest.approx(5.0)
            assert rate == pytest.approx(200 / 5.0)


def test_single_rank_needs_no_process_group():
    import bench

    assert bench.whole_job_rate(4.0, 80, world=1) == (20.0, 4.0)
