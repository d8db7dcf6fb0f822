"""The multi-GPU path of the benchmark is replicas only (each rank runs the whole
decode step on its own GPU; the path does not shard).  Its host side -- the
max-over-ranks time and the whole-job sum of work -- runs here on CPU with the
gloo backend and world size 2."""
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


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    t_local = 1.0 + rank          # rank 1 is the slower replica
    units_local = 100.0 * (rank + 1)
    t, u = bench.replica_totals(t_local, units_local, dist, torch.device("cpu"))
    dist.barrier()
    out[rank] = (t, u)
    dist.destroy_process_group()


def test_replica_totals_gloo_world2():
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
    for rank in range(2):
        t, u = out[rank]
        assert t == 2.0                      # the job lasts as long as its slowest replica
        assert u == 300.0                    # whole-job work is the sum over replicas


def test_replica_totals_single_process():
    import bench
    assert bench.replica_totals(0.5, 42.0) == (0.5, 42.0)
