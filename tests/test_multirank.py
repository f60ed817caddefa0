"""The N>1 measurement path of bench.py on CPU: two gloo ranks, the slowest rank's time and
the whole-job throughput (every rank runs its own canvases, no data-path collective)."""
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
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, w, local = bench.dist_env()
    assert (r, w, local) == (rank, world, rank)

    def reduce_max(x):
        t = torch.tensor([x], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    ms_local = 100.0 + 50.0 * rank          # rank 1 is the slow one
    ms_total, ms_step, value = bench.aggregate_timing(ms_local, 20, world, reduce_max)
    out[rank] = (ms_total, ms_step, value)
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_aggregation_gloo():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        ms_total, ms_step, value = res[rank]
        assert ms_total == 150.0                       # max over ranks
        assert ms_step == pytest.approx(7.5)
        assert value == pytest.approx(world * 20 / 0.150)   # whole-job steps/s
