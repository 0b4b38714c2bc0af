"""bench.py's multi-GPU path is replicas: every rank decodes the whole sentence set and the
job rate is (units of all ranks) / (slowest rank's time).  The cross-rank reduction it uses is
checked here with two gloo ranks on the CPU."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    tokens = 1000.0 * (rank + 1)             # rank 0: 1000 tokens in 2 s; rank 1: 2000 in 4 s
    seconds = 2.0 * (rank + 1)
    out[rank] = (bench.over_ranks(seconds, "max", dist), bench.over_ranks(tokens, "sum", dist),
                 bench.job_rate(tokens, seconds, dist))
    dist.barrier()
    dist.destroy_process_group()


def test_replica_job_rate_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        for r in range(2):
            assert out[r] == (4.0, 3000.0, 750.0)


def test_single_process_is_identity():
    import bench
    assert bench.over_ranks(3.5, "max") == 3.5
    assert bench.job_rate(100.0, 4.0) == 25.0
