"""GPU path vs CPU oracle, bit-exact, with draining instances and the
auto-scaling signal (Sec. 3.4-3.6): per-request results, the migration log
(scale-out / scale-in records included) and every per-replica counter."""
import numpy as np
import pytest

from paper_2608_16336_gb300 import mtsim
from paper_2608_16336_gb300 import workloads as W
from tests import parity
from tests._tiny import tiny_case

pytestmark = pytest.mark.gpu

NEVER = 0xFFFFFFFF


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def drain_schedule(w, seed, *, p_instance=0.3):
    """Per replica: no draining, some instances draining from a time drawn
    from the trace's arrivals, the ticks or uniformly (so that equal times
    occur), half the instances draining from t = 0, or every instance
    draining (the dispatch fallback)."""
    rng = np.random.default_rng(seed)
    R, N = w.num_replicas, w.num_instances
    d = np.full((R, N), NEVER, np.uint32)
    for r in range(R):
        arr = w.arrival_us[w.replica_slice(r)].astype(np.int64)
        if arr.size == 0:
            continue
        span = int(arr[-1]) + 1
        ticks = np.arange(1, span // w.migrate_interval_us + 2, dtype=np.int64) * w.migrate_interval_us
        times = np.concatenate([arr, ticks, rng.integers(0, span, size=arr.size)])
        u = rng.random()
        if u < 0.15:
            d[r] = rng.choice(times, size=N)
        elif u < 0.25:
            d[r, : N // 2] = 0
        elif u < 0.35:
            continue
        else:
            pick = rng.random(N) < p_instance
            d[r, pick] = rng.choice(times, size=int(pick.sum()))
    return d


def _with(w, seed, autoscale=1, **policy):
    w.autoscale = autoscale
    for k, v in policy.items():
        setattr(w, k, v)
    w.drain_start_us = drain_schedule(w, seed)
    return w


def _kinds(events):
    return set(int(k) for e in events for k in e[:, 5])


def test_workload0_drain_and_autoscale():
    w = W.config(0)
    w.autoscale = 1
    arr = w.arrival_us
    w.drain_start_us = np.array([[NEVER, int(arr[len(arr) // 3]), NEVER, 10 * w.migrate_interval_us]], np.uint32)
    _, st, ev = parity.check_parity(w, event_log_capacity=1 << 15)
    assert {mtsim.SIM_EV_SCALE_IN, mtsim.SIM_EV_QUEUED} <= _kinds(ev)


def test_workload1_slice_drain_and_autoscale():
    w = _with(W.config(1, replicas=range(67), requests=3000), seed=1)
    _, st, ev = parity.check_parity(w, event_log_capacity=1 << 14)
    assert (st["scale_in_signals"] + st["scale_out_signals"]).sum() > 0


def test_workload1_full_requests_drain_sample():
    w = _with(W.config(1, replicas=[3, 700]), seed=2)
    parity.check_parity(w, event_log_capacity=1 << 16)


def test_workload2_drain_and_autoscale():
    reps = [((k * 3 + d) * 2 + ld) * 64 + (k + 2 * d + ld) % 64 for k in range(10) for d in range(3) for ld in range(2)]
    w = _with(W.config(2, replicas=reps, requests=2000), seed=3)
    parity.check_parity(w, event_log_capacity=1 << 14)


def test_workload3_many_instances_drain_and_autoscale():
    # 128 instances: four per lane, running-request records in HBM
    w = _with(W.config(3, replicas=[0, 1, 2], requests=20000), seed=4)
    parity.check_parity(w, event_log_capacity=1 << 16)


def test_autoscale_ticks_without_migration():
    w = _with(W.config(1, replicas=range(24), requests=3000), seed=5, enable_migration=0)
    _, st, ev = parity.check_parity(w, event_log_capacity=1 << 14)
    assert (st["migrations"] == 0).all() and (st["migration_starts"] == 0).all()
    assert st["scale_in_signals"].sum() + st["scale_out_signals"].sum() > 0


@pytest.mark.parametrize("thresholds", [(-1, 3, 2), (1, 6, 1), (-9, -1, 4)])
@pytest.mark.parametrize("n,m,t_blk,bmax,k", [(2, 12, 4, 3, 2), (5, 30, 3, 4, 3), (33, 20, 2, 5, 4)])
def test_tiny_clusters_drain(n, m, t_blk, bmax, k, thresholds):
    traces = []
    for s in range(40):
        _, _, _, tr, _ = tiny_case(7000 + 100 * n + s, max_requests=40)
        a, p, o, tier = tr
        cap = m * t_blk
        p = np.minimum(p, cap // 2).astype(np.uint16)
        o = np.maximum(np.minimum(o, cap - p), 1).astype(np.uint16)
        traces.append((a, p, o, (tier % k).astype(np.uint8)))
    h = [max(0, m // 4 >> i) for i in range(k)]
    out_num, in_num, den = thresholds
    w = W.custom(n, m, [k], [h], [0] * len(traces), traces, tokens_per_block=t_blk, max_batch=bmax,
                 iter_base_us=60, iter_us_per_prefill_token=2, iter_us_per_decode_seq=3, migrate_blocks_per_iter=2,
                 migrate_interval_us=150, autoscale=1, scale_out_num=out_num, scale_in_num=in_num, scale_den=den)
    w.drain_start_us = drain_schedule(w, seed=n * 31 + m, p_instance=0.5)
    parity.check_parity(w)


def test_chunked_run_with_drain_equals_oracle():
    w = _with(W.config(1, replicas=range(8), requests=1500), seed=6)
    parity.check_parity(w, max_steps=97)


def test_device_drain_schedule_and_removal():
    torch = pytest.importorskip("torch")
    w = _with(W.config(1, replicas=range(8), requests=1500), seed=7)
    ref = parity.run_gpu(w)
    sim = mtsim.Simulator(w)
    try:
        sim.load()                           # host schedule from the workload
        d = torch.from_numpy(w.drain_start_us.view(np.int32)).cuda()
        mtsim.sim_set_drain(sim.handle, d.data_ptr(), 1)
        sim.reset()                          # the device copy takes effect here
        assert sim.run() == 0
        res, st, _ = sim.metrics()
        np.testing.assert_array_equal(res, ref[0])
        np.testing.assert_array_equal(st, ref[1])
        mtsim.sim_set_drain(sim.handle, None, 0)
        sim.reset()
        assert sim.run() == 0
        res2, st2, _ = sim.metrics()
    finally:
        sim.close()
    w.drain_start_us = None
    plain = parity.run_gpu(w)
    np.testing.assert_array_equal(res2, plain[0])
    np.testing.assert_array_equal(st2, plain[1])
