"""GPU path vs CPU oracle, bit-exact: per-request dispatch instance, final
instance, first-token and finish times, migration and preemption counts, the
migration log and every per-replica counter, on the same seeded inputs."""
import numpy as np
import pytest

from paper_2608_16336_gb300 import mtsim
from paper_2608_16336_gb300 import workloads as W
from tests import parity
from tests._tiny import tiny_case

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


# ------------------------------------------------------------ workloads --
def test_workload0_full():
    w = W.config(0)
    parity.check_parity(w, event_log_capacity=1 << 15)


def test_workload1_slice_ragged():
    # 67 replicas: not a multiple of the warps per block or of the grid
    w = W.config(1, replicas=range(67), requests=4000)
    parity.check_parity(w)


def test_workload1_full_requests_sample():
    w = W.config(1, replicas=[0, 511, 1023])
    parity.check_parity(w, event_log_capacity=1 << 15)


def test_workload2_sweep_sample():
    # every K = 1..10, every tier distribution and both loads
    reps = [((k * 3 + d) * 2 + ld) * 64 + (k + d + ld) % 64 for k in range(10) for d in range(3) for ld in range(2)]
    w = W.config(2, replicas=reps, requests=2500)
    parity.check_parity(w)


def test_workload3_bursty_many_instances():
    w = W.config(3, replicas=[0, 1], requests=30000)
    # Gamma gaps with CV = 3 put several arrivals on one microsecond
    for r in range(w.num_replicas):
        a = w.arrival_us[w.replica_slice(r)]
        _, counts = np.unique(a, return_counts=True)
        assert counts.max() > 4
    parity.check_parity(w, event_log_capacity=1 << 16)


def test_workload4_sample():
    w = W.config(4, replicas=[0, 7, 16383], requests=6000)
    parity.check_parity(w)


# ---------------------------------------------------------- edge cases --
def _batch_of_tiny(seed0, count, n, m, t_blk, bmax, k, **policy):
    traces = []
    for s in range(count):
        _, _, _, tr, _ = tiny_case(seed0 + s, max_requests=40)
        a, p, o, tier = tr
        cap = m * t_blk
        p = np.minimum(p, cap // 2).astype(np.uint16)
        o = np.maximum(np.minimum(o, cap - p), 1).astype(np.uint16)
        traces.append((a, p, o, (tier % k).astype(np.uint8)))
    h = [max(0, m // 4 >> i) for i in range(k)]
    return W.custom(n, m, [k], [h], [0] * count, traces, tokens_per_block=t_blk, max_batch=bmax, **policy)


@pytest.mark.parametrize("n,m,t_blk,bmax,k", [(1, 10, 4, 2, 1), (3, 12, 4, 3, 3), (5, 30, 3, 4, 2),
                                               (33, 20, 2, 5, 4), (70, 16, 5, 64, 16)])
def test_tiny_clusters(n, m, t_blk, bmax, k):
    w = _batch_of_tiny(100 * n, 50, n, m, t_blk, bmax, k, iter_base_us=60, iter_us_per_prefill_token=2,
                       iter_us_per_decode_seq=3, migrate_blocks_per_iter=2, migrate_interval_us=150)
    parity.check_parity(w)


def test_empty_and_single_request_replicas():
    one = (np.array([5], np.uint32), np.array([100], np.uint16), np.array([20], np.uint16), np.array([1], np.uint8))
    empty = tuple(np.zeros(0, dt) for dt in (np.uint32, np.uint16, np.uint16, np.uint8))
    w = W.custom(4, 1024, [2], [[256, 128]], [0, 0, 0, 0], [empty, one, empty, one])
    res, st, ev = parity.check_parity(w)
    assert int(st["steps"][0]) == 0 and int(st["steps"][2]) == 0
    assert int(res["first_token_us"][0]) - 5 == 4000 + 20 * 100


def test_many_simultaneous_arrivals():
    rng = np.random.default_rng(3)
    traces = []
    for burst in (31, 32, 33, 64, 65, 200):
        q = burst + 20
        a = np.concatenate([np.full(burst, 1000), 1000 + np.cumsum(rng.integers(0, 3, 20))]).astype(np.uint32)
        traces.append((a, rng.integers(16, 600, q).astype(np.uint16), rng.integers(1, 50, q).astype(np.uint16),
                       rng.integers(0, 4, q).astype(np.uint8)))
    w = W.custom(8, 512, [4], [[128, 64, 32, 16]], [0] * len(traces), traces)
    parity.check_parity(w)


def test_largest_shapes():
    """N = 256 instances (8 per lane), K = 16 tiers, batch 64."""
    T, N, M = 16, 256, 2048
    rate = W._load_rate(0.9, N, M, T, 64, W.LEN_DEFAULT)
    p = W._params(11, 6000, 16, W.tier_probs("uniform", 16), rate, W.LEN_DEFAULT)
    off, a, pl, ol, tr = W.generate([p])
    w = W.custom(N, M, [16], [W.headroom_decay_table(2048, 16)], [0], [(a, pl, ol, tr)])
    parity.check_parity(w)


def test_non_power_of_two_block_size_and_no_migration():
    w = W.config(1, replicas=range(5), requests=3000)
    w.tokens_per_block = 12
    parity.check_parity(w)
    w.enable_migration = 0
    parity.check_parity(w)


def test_memory_pressure_preemption_and_aborts():
    w = W.config(1, replicas=range(6), requests=2500)
    w.blocks_per_instance = 300
    w.tables_h = [[64, 32, 16, 8]]
    w.prompt_len = np.minimum(w.prompt_len, 2400).astype(np.uint16)
    res, st, ev = parity.check_parity(w, event_log_capacity=1 << 15)
    assert int(st["preemptions"].sum()) > 0 and int(st["migration_aborts"].sum()) > 0


def test_event_log_overflow_truncates():
    w = W.config(0, requests=600)
    res, st, ev = parity.check_parity(w, event_log_capacity=7)
    assert int(st["log_events"][0]) > 7 and ev[0].shape[0] == 7


# ---------------------------------------------------------- determinism --
def test_chunked_run_equals_single_run():
    w = W.config(1, replicas=range(9), requests=3000)
    full = parity.run_gpu(w)
    for chunk in (37, 1000):
        part = parity.run_gpu(w, max_steps=chunk)
        assert (full[0] == part[0]).all() and (full[1] == part[1]).all()
        for x, y in zip(full[2], part[2]):
            assert (x == y).all()
    small = W.config(1, replicas=range(2), requests=200)
    a, b = parity.run_gpu(small), parity.run_gpu(small, max_steps=1)
    assert (a[0] == b[0]).all() and (a[1] == b[1]).all()


def test_replica_independent_of_batch():
    w = W.config(1, replicas=range(12), requests=3000)
    batch = parity.run_gpu(w)
    alone = parity.run_gpu(w.subset([7]))
    sl = w.replica_slice(7)
    assert (batch[0][sl] == alone[0]).all()
    assert (batch[1][7] == alone[1][0]).all()
    assert (batch[2][7] == alone[2][0]).all()


def test_host_and_device_loading_agree_and_reset_repeats():
    w = W.config(2, replicas=[5, 900, 3000], requests=2000)
    a = parity.run_gpu(w, on_device=True)
    b = parity.run_gpu(w, on_device=False, torch_allocator=False)
    assert (a[0] == b[0]).all() and (a[1] == b[1]).all()
    from paper_2608_16336_gb300 import mtsim

    sim = mtsim.Simulator(w)
    sim.load()
    sim.run()
    r1 = sim.metrics()
    sim.reset()
    sim.run()
    r2 = sim.metrics()
    sim.close()
    assert (r1[0] == r2[0]).all() and (r1[1] == r2[1]).all() and (r1[2] == r2[2]).all()


def test_malformed_trace_rejected():
    from paper_2608_16336_gb300 import mtsim

    good = (np.array([1, 2], np.uint32), np.array([4, 4], np.uint16), np.array([4, 4], np.uint16),
            np.array([0, 1], np.uint8))
    bads = [
        (np.array([2, 1], np.uint32),) + good[1:],
        good[:3] + (np.array([0, 2], np.uint8),),
        (good[0], np.array([0, 4], np.uint16)) + good[2:],
        (good[0], np.array([60000, 4], np.uint16)) + good[2:],
    ]
    for tr in bads:
        w = W.custom(2, 64, [2], [[8, 4]], [0], [tr])
        sim = mtsim.Simulator(w)
        with pytest.raises(mtsim.SimError) as e:
            sim.load(on_device=False)
        assert e.value.code == mtsim.SIM_ERR_TRACE
        with pytest.raises(mtsim.SimError) as e:
            sim.run()
        assert e.value.code == mtsim.SIM_ERR_STATE
        sim.close()


def test_migration_threshold_equality():
    """Freeness difference exactly theta at a tick (theta = 0, equal
    instances) migrates; theta = 1/1000 does not (Sec. 3.5's >=)."""
    tr = (np.array([0, 1], np.uint32), np.array([1, 1], np.uint16), np.array([600, 600], np.uint16),
          np.array([0, 0], np.uint8))
    for num, den in ((0, 1), (1, 1000)):
        w = W.custom(2, 10, [1], [[0]], [0, 0], [tr, tr], tokens_per_block=64, theta_num=num, theta_den=den)
        _, st, _ = parity.check_parity(w)
        assert (st["migration_starts"] > 0).all() == (num == 0)


def test_replica_start_order_changes_nothing():
    """Starting the replicas in another order (sim_set_order) gives the same
    results bit for bit, with more replicas than the GPU holds at once (so
    the reordered counter feeds several waves); a non-permutation is
    rejected and leaves the previous order."""
    w = W.config(4, replicas=range(3000), requests=300)
    want = parity.run_gpu(w, event_log_capacity=1024)
    perm = np.random.default_rng(7).permutation(w.num_replicas)
    sim = mtsim.Simulator(w, event_log_capacity=1024)
    try:
        with pytest.raises(mtsim.SimError) as e:
            sim.set_order(np.zeros(w.num_replicas, np.int32))
        assert e.value.code == mtsim.SIM_ERR_ARG
        sim.set_order(perm)
        sim.load()
        assert sim.launch_info()["grid_blocks"] * 2 < w.num_replicas
        assert sim.run() == 0
        res, st, ev = sim.metrics()
        events = [sim.events_of(ev, st, r) for r in range(w.num_replicas)]
        sim.set_order(None)
    finally:
        sim.close()
    assert (res == want[0]).all() and (st == want[1]).all()
    for a, b in zip(events, want[2]):
        np.testing.assert_array_equal(a, b)


# ----------------------------------------------------------- full size --
def test_workload1_full_size_sampled():
    """The 1,024-replica workload at full size, in the launch configuration
    the benchmark times: sampled replicas bit-exact, properties for all."""
    w = W.config(1)
    res, st, events = parity.run_gpu(w, event_log_capacity=1 << 14)
    parity.check_properties(w, res, st)
    reps = [0, 1, 333, 777, 1022, 1023]
    ref = parity.run_oracle(w, reps, event_log_capacity=1 << 14)
    for r in reps:
        parity.compare_replica(w, r, res, st, events, ref[r])


def test_workload2_full_size_sampled():
    """The 3,840-replica sweep at full size: sampled replicas (K = 1, 5 and
    10, each tier distribution, both loads) bit-exact, properties for all."""
    w = W.config(2)
    res, st, events = parity.run_gpu(w, event_log_capacity=1 << 14)
    parity.check_properties(w, res, st)
    reps = [((k * 3 + d) * 2 + ld) * 64 + 17 * k % 64 for k in (0, 4, 9) for d in range(3) for ld in range(2)]
    ref = parity.run_oracle(w, reps, event_log_capacity=1 << 14)
    for r in reps:
        parity.compare_replica(w, r, res, st, events, ref[r])


def test_workload3_full_size_sampled():
    """The 256-replica, 128-instance bursty workload at full size (200,000
    requests per replica): first, middle and last replica bit-exact,
    properties for all."""
    w = W.config(3)
    res, st, events = parity.run_gpu(w, event_log_capacity=1 << 14)
    parity.check_properties(w, res, st)
    reps = [0, 128, 255]
    ref = parity.run_oracle(w, reps, event_log_capacity=1 << 14)
    for r in reps:
        parity.compare_replica(w, r, res, st, events, ref[r])


def test_workload4_full_size_sampled():
    """The 16,384-replica workload at full size (64 instances, 50,000 requests
    per replica) in the benchmark's launch: the same kernel variant and grid
    and a migration log sized, as the benchmark sizes it, to hold every
    record.  Eight sampled replicas (first, last, spread) bit-exact on every
    result, every log record and every counter; properties for all."""
    import bench
    import torch

    w = W.config(4)
    order = np.argsort(-W.predicted_work(4), kind="stable").astype(np.int32)  # the benchmark's start order
    sim, cap, st0 = bench.sized_simulator(mtsim, w, bench.initial_log_capacity(w), torch.cuda.current_stream(),
                                          order)
    try:
        assert sim.launch_info()["instances_per_lane"] == 2 and not sim.launch_info()["slots_in_shared"]
        res, st, ev = sim.metrics()
        assert int(st["log_events"].max()) <= cap
        reps = [0, 1, 2730, 5461, 8191, 10922, 13653, 16383]
        events = {r: sim.events_of(ev, st, r) for r in reps}
        del ev
    finally:
        sim.close()
    parity.check_properties(w, res, st)
    ref = parity.run_oracle(w, reps, event_log_capacity=cap)
    for r in reps:
        parity.compare_replica(w, r, res, st, events, ref[r])


def test_workload4_full_requests_sample():
    """Replicas of the 16,384-replica workload with their full 50,000-request
    traces, bit-exact."""
    w = W.config(4, replicas=[0, 8191, 16383])
    parity.check_parity(w, event_log_capacity=1 << 14)


def test_partitioned_runs_equal_the_whole():
    """Replicas split into ranges by predicted work, as the multi-GPU
    benchmark splits them across ranks, and simulated range by range give
    the whole run's results bit for bit (replicas never interact)."""
    reps = list(range(0, 3840, 32))  # 120 replicas of the sweep: every K, distribution and load
    whole = W.config(2, replicas=reps, requests=800)
    want = parity.run_gpu(whole, event_log_capacity=2048)
    work = W.predicted_work(2, requests=800)[reps]
    for lo, hi in W.partition(work, 3):
        part = W.config(2, replicas=reps[lo:hi], requests=800)
        got = parity.run_gpu(part, event_log_capacity=2048)
        a, b = int(whole.offsets[lo]), int(whole.offsets[hi])
        assert (got[0] == want[0][a:b]).all()
        assert (got[1] == want[1][lo:hi]).all()
        for r in range(hi - lo):
            np.testing.assert_array_equal(got[2][r], want[2][lo + r])
