"""The benchmark's multi-rank host path on the CPU (two gloo ranks).

The Ember step has no cross-GPU exchange here: every rank holds its own
table and state (independent replicas).  What several ranks share is host
logic: the rendezvous, the barrier around the timed region and the
max-over-ranks step time.  This runs it with world_size 2 on gloo.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(world),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    w, r, local = bench.dist_setup()
    assert (w, r, local) == (world, rank, rank)
    bench.barrier(w)
    ms = bench.allreduce_max(w, 1.0 + 2.5 * rank)  # rank 1 is the slower one
    bench.barrier(w)
    import torch.distributed as dist
    dist.destroy_process_group()
    out[rank] = ms


def test_two_rank_barrier_and_max_time():
    world, port = 2, _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
        assert dict(out) == {0: 3.5, 1: 3.5}


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.allreduce_max(1, 2.0) == 2.0
    bench.barrier(1)
