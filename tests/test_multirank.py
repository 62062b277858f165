"""Multi-GPU host logic on CPU: two gloo ranks, each with its own independent
copy of the workload (weak scaling), combined by max-of-time / sum-of-work.
No GPU and no collective on the data path."""
import os
import socket

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2608_16336_gb300 import workloads as W

    w = W.config(1, replicas=range(3), requests=50, seed_block=rank)
    seconds = 1.0 + rank            # rank 1 is the slow one
    units = 1000.0 * (rank + 1)
    events = 10.0 * (rank + 1)
    t, u, e = bench.aggregate(seconds, units, events)
    bench.barrier()
    out.put((rank, t, u, e, int(w.arrival_us[:50].sum()), bench.dist_env()[:2]))
    dist.destroy_process_group()


def test_two_ranks_weak_scaling_aggregation():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    for rank, t, u, e, _, env in res:
        assert t == 2.0            # max over ranks
        assert u == 3000.0         # sum over ranks
        assert e == 30.0
        assert env == (2, rank)
    assert res[0][4] != res[1][4]  # each rank simulates its own, independent traces


def test_single_process_aggregate_is_identity():
    import bench

    assert bench.aggregate(1.5, 10.0, 3.0) == (1.5, 10.0, 3.0)
