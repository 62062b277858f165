"""Multi-GPU host logic on CPU: two gloo ranks split one workload's replica
range by predicted work (requests x instances x load), each builds exactly
its own replicas' traces, and the timings combine by max-of-time /
sum-of-work.  No GPU and no collective on the data path."""
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

    ws, rk, _ = bench.dist_env()
    # the 3,840-replica sweep: replicas carry different loads, so the split is by work, not by count
    lo, hi = W.partition(W.predicted_work(2, requests=40), ws)[rk]
    w = W.config(2, replicas=range(lo, hi), requests=40)
    seconds = 1.0 + rank            # rank 1 is the slow one
    units = 1000.0 * (rank + 1)
    events = 10.0 * (rank + 1)
    t, u, e = bench.aggregate(seconds, units, events)
    bench.barrier()
    out.put((rank, t, u, e, (lo, hi), int(w.num_replicas), int(w.arrival_us.astype(np.int64).sum()), (ws, rk)))
    dist.destroy_process_group()


def test_two_ranks_partition_and_aggregation():
    from paper_2608_16336_gb300 import workloads as W

    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=180) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    for rank, t, u, e, _, _, _, env in res:
        assert t == 2.0            # max over ranks
        assert u == 3000.0         # sum over ranks
        assert e == 30.0
        assert env == (2, rank)
    # the two ranges tile 0..3839 exactly once, and each rank built exactly its own replicas
    (lo0, hi0), (lo1, hi1) = res[0][4], res[1][4]
    assert lo0 == 0 and hi0 == lo1 and hi1 == 3840
    assert res[0][5] == hi0 - lo0 and res[1][5] == hi1 - lo1
    # the traces a rank built are those of the full workload's same replicas
    full = W.config(2, requests=40)
    for rank, *_rest in res:
        lo, hi = res[rank][4]
        assert res[rank][6] == int(full.arrival_us[full.offsets[lo]:full.offsets[hi]].astype(np.int64).sum())
    # balanced by predicted work: the halves differ by less than one replica's weight
    wts = W.predicted_work(2, requests=40)
    assert abs(wts[lo0:hi0].sum() - wts[lo1:hi1].sum()) <= wts.max()


@pytest.mark.parametrize("parts", [1, 2, 3, 7, 8])
def test_partition_covers_every_replica_once(parts):
    from paper_2608_16336_gb300 import workloads as W

    for cid in range(5):
        wts = W.predicted_work(cid)
        if len(wts) < parts:
            with pytest.raises(ValueError):
                W.partition(wts, parts)
            continue
        ranges = W.partition(wts, parts)
        assert len(ranges) == parts
        assert ranges[0][0] == 0 and ranges[-1][1] == len(wts)
        for (a, b), (c, d) in zip(ranges, ranges[1:]):
            assert b == c
        assert all(b > a for a, b in ranges)
        share = [wts[a:b].sum() for a, b in ranges]
        assert max(share) - min(share) <= 2 * wts.max() + 1e-6


def test_partition_by_weight_not_count():
    from paper_2608_16336_gb300 import workloads as W

    # one heavy replica followed by light ones: the heavy one gets a range of its own
    assert W.partition([10.0, 1.0, 1.0, 1.0, 1.0, 1.0, 1.0, 1.0, 1.0, 1.0, 1.0], 2) == [(0, 1), (1, 11)]
    assert W.partition([1.0] * 8, 4) == [(0, 2), (2, 4), (4, 6), (6, 8)]


def test_single_process_aggregate_is_identity():
    import bench

    assert bench.aggregate(1.5, 10.0, 3.0) == (1.5, 10.0, 3.0)
