"""The multi-rank logic of bench.py (independent replicas, one search per rank) on two
CPU processes with the gloo backend: the job rate is all ranks' units over the slowest
rank's time, and ranks agree on it."""
import os
import socket

import pytest
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
    secs = [2.0, 5.0][rank]                  # rank 1 is the slow one
    out[rank] = (bench.max_over_ranks(secs, world), bench.job_throughput(200, secs, world))
    bench.barrier(world)
    dist.destroy_process_group()


def test_replica_throughput_two_ranks_gloo():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
            assert p.exitcode == 0
        res = dict(out)
    for r in range(2):
        slowest, rate = res[r]
        assert slowest == 5.0
        assert rate == pytest.approx(200 * 2 / 5.0)
