"""Randomised GPU-vs-oracle sweep: many small clusters with random shapes and
policies (instances 1-70, block size, batch size, tier count and headroom,
migration on or off, auto-scaling thresholds, drain schedules, iteration-time
coefficients), each compared bit-exactly on every per-request result, the
migration / signal log and every per-replica counter.  Seeded: every run
draws the same cases."""
import numpy as np
import pytest

from paper_2608_16336_gb300 import workloads as W
from tests import parity

pytestmark = pytest.mark.gpu

NEVER = 0xFFFFFFFF


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def random_workload(seed: int):
    rng = np.random.default_rng(50_000 + seed)
    n = int(rng.choice([1, 2, 3, 5, 8, 16, 31, 33, 64, 70]))
    t_blk = int(rng.choice([1, 2, 3, 4, 8, 16, 64]))
    # a third of the cases starve for KV blocks, so preemption is frequent
    m = int(rng.integers(8, 40)) if rng.random() < 0.33 else int(rng.integers(40, 400))
    bmax = int(rng.choice([1, 2, 3, 7, 16, 64]))
    k = int(rng.integers(1, 17))
    h0 = int(rng.integers(0, max(1, m // 2)))
    heads = [h0 >> i for i in range(k)]
    cap = m * t_blk
    reps = int(rng.integers(1, 9))
    traces = []
    for _ in range(reps):
        q = int(rng.integers(0, 300))
        gaps = rng.choice([0, 0, 1, 3, 50, 200, 900], size=q)
        a = np.cumsum(gaps).astype(np.uint32)
        p = rng.integers(1, max(2, min(cap, 65535) // 2), size=q).astype(np.int64)
        o = rng.integers(1, 40, size=q).astype(np.int64)
        o = np.maximum(np.minimum(o, min(cap, 65536) - p), 1)
        traces.append((a, p.astype(np.uint16), o.astype(np.uint16), rng.integers(0, k, size=q).astype(np.uint8)))
    den = int(rng.integers(1, 5))
    out_num = int(rng.integers(-8 * den, 2 * den))
    policy = dict(iter_base_us=int(rng.integers(1, 200)), iter_us_per_prefill_token=int(rng.integers(0, 5)),
                  iter_us_per_decode_seq=int(rng.integers(0, 8)), migrate_blocks_per_iter=int(rng.integers(1, 9)),
                  migrate_interval_us=int(rng.integers(20, 600)), enable_migration=int(rng.integers(0, 4) > 0),
                  autoscale=int(rng.integers(0, 2)), scale_out_num=out_num,
                  scale_in_num=out_num + int(rng.integers(1, 10 * den)), scale_den=den)
    w = W.custom(n, m, [k], [heads], [0] * reps, traces, tokens_per_block=t_blk, max_batch=bmax, **policy)
    if rng.integers(0, 2):
        d = np.full((reps, n), NEVER, np.uint32)
        for r in range(reps):
            arr = traces[r][0].astype(np.int64)
            span = int(arr[-1]) + 1 if arr.size else 1000
            pick = rng.random(n) < 0.3
            d[r, pick] = rng.integers(0, span, size=int(pick.sum()))
        w.drain_start_us = d
    return w


@pytest.mark.parametrize("chunk", range(12))
def test_random_clusters(chunk):
    for seed in range(chunk * 25, chunk * 25 + 25):
        w = random_workload(seed)
        if w.total_requests == 0:
            continue
        try:
            parity.check_parity(w, event_log_capacity=1 << 14)
        except AssertionError as e:
            raise AssertionError("random case %d: %s" % (seed, e)) from e


@pytest.mark.parametrize("chunk", range(4))
def test_random_clusters_with_headroom_changes(chunk):
    """The same random clusters run in random-size chunks of steps, with the
    headroom table replaced at random between chunks (sim_set_headroom, the
    adaptive-headroom mechanism); the oracle given the same schedule must
    agree bit for bit."""
    from oracle import oracle as O
    from paper_2608_16336_gb300 import mtsim

    total_changes = 0
    for seed in range(chunk * 25, chunk * 25 + 25):
        w = random_workload(1000 + seed)
        if w.total_requests == 0:
            continue
        rng = np.random.default_rng(90_000 + seed)
        k, m = w.tables_k[0], w.blocks_per_instance
        steps = int(rng.integers(1, 400))
        cap = 1 << 14
        sched = []
        sim = mtsim.Simulator(w, event_log_capacity=cap)
        try:
            sim.load()
            j = 0
            while sim.run(steps) > 0:
                j += 1
                if rng.random() < 0.7:
                    tab = np.zeros_like(sim._th)
                    tab[0, :k] = rng.integers(0, max(1, m // 2), size=k)
                    sim.set_headroom(tab)
                    sched.append((j * steps, [int(x) for x in tab[0, :k]]))
            res, st, ev = sim.metrics()
            events = [sim.events_of(ev, st, r) for r in range(w.num_replicas)]
        finally:
            sim.close()
        total_changes += len(sched)
        ref = O.run_workload(w, range(w.num_replicas), nthreads=8, log_capacity=cap,
                             headroom_schedules={r: sched for r in range(w.num_replicas)})
        try:
            for r in range(w.num_replicas):
                parity.compare_replica(w, r, res, st, events, ref[r])
        except AssertionError as e:
            raise AssertionError("random case %d (%d changes): %s" % (1000 + seed, len(sched), e)) from e
    assert total_changes >= 25, total_changes  # the tables really changed mid-run
