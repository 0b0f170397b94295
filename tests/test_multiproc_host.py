"""Host logic of the multi-GPU bench path with two gloo ranks on CPU.

Sequences are independent, so ranks shard the batch (each rank draws its own
seeded batch) and exchange nothing on the data path; only the timing is
reduced (max over ranks) and the whole-job value sums all ranks' rounds.
"""

import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench

    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, lr, w = bench.dist_env()
        assert (r, lr, w) == (rank, rank, world)
        # each rank's batch is its own: different seeds, different draws
        seed = bench.shard_seed(42, rank)
        seeds = [None] * world
        dist.all_gather_object(seeds, seed)
        assert len(set(seeds)) == world
        # the slowest rank decides the time; the value counts every rank's rounds
        my_secs = 1.0 + rank
        bench.barrier(world)
        t = bench.max_over_ranks(my_secs, world)
        assert t == float(world)
        results[rank] = bench.aggregate_value(10, world, t)
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_rank_host_logic():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    results = mgr.dict()
    mp.spawn(_worker, args=(world, port, results), nprocs=world, join=True)
    assert results[0] == results[1] == 10 * world / 2.0
