"""The bench's multi-rank bookkeeping on CPU: two gloo ranks take the max of
their times and report the whole job's throughput (replicas, no exchange)."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    t = bench.reduce_max(1.0 + rank, world, "cpu")          # rank 1 is the slow one
    v = bench.aggregate(per_rank_units=80.0, max_seconds=t, world=world)
    bench.barrier(world)
    out[rank] = (t, v)
    dist.destroy_process_group()


def test_two_gloo_ranks_take_max_time_and_sum_units():
    world, port = 2, _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, port, out), nprocs=world, start_method="spawn")
    assert out[0] == out[1] == (2.0, 80.0)
