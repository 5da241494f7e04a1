"""Replica timing aggregation across ranks on CPU (gloo, world size 2): every
rank runs an independent replica, the job's time is the slowest rank's and
the throughput counts every rank's units (the benchmark's rule)."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, secs, units, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ws, r, local = bench.dist_env()
        assert (ws, r, local) == (world, rank, rank)
        t = torch.tensor([secs[rank]], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        u = torch.tensor([units[rank]], dtype=torch.float64)
        dist.all_reduce(u, op=dist.ReduceOp.SUM)
        dist.barrier()
        out[rank] = (float(u.item()) / float(t.item()), float(t.item()))
    finally:
        dist.destroy_process_group()


def test_replica_aggregation_gloo():
    world = 2
    secs = [1.5, 2.0]
    units = [3.0e12, 3.0e12]
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, _free_port(), secs, units, out), nprocs=world, join=True)
        res = dict(out)
    want = bench.aggregate(secs, units)
    for r in range(world):
        assert res[r][0] == pytest.approx(want[0]) and res[r][1] == pytest.approx(want[1])
    assert want == (6.0e12 / 2.0, 2.0)
