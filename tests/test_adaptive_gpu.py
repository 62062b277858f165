"""Adaptive headroom on the GPU (the controller of adaptive.py driving
sim_set_headroom between sim_run epochs) against the oracle run with the
same headroom schedule: bit-exact on every result, log record and counter."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_16336_gb300 import adaptive
from paper_2608_16336_gb300 import workloads as W
from tests import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def _check(w, slo, epoch_steps, cap=4096):
    res, st, events, sched = adaptive.run(w, slo, epoch_steps=epoch_steps, event_log_capacity=cap)
    v = adaptive.per_replica_tables(w)
    ref = O.run_workload(v, range(v.num_replicas), nthreads=8, log_capacity=cap, headroom_schedules=sched)
    for r in range(v.num_replicas):
        parity.compare_replica(v, r, res, st, events, ref[r])
    return sched


def test_adaptive_headroom_matches_oracle():
    w = W.config(1, replicas=range(12), requests=3000)
    sched = _check(w, [40_000, 150_000, 100_000, 200_000], epoch_steps=4000)
    changes = [(r, j, tab) for r, s in sched.items() for j, tab in s]
    assert len(changes) > 12  # the rule fired, for every replica on average
    h0 = W.headroom_decay_table(512, 4)
    ups = sum(1 for r, s in sched.items() for _, tab in s if tab[0] > h0[0])
    downs = sum(1 for r, s in sched.items() for _, tab in s if tab[3] < h0[3])
    assert ups > 0 and downs > 0


def test_adaptive_headroom_many_tiers_and_chunks():
    # the 3,840-replica sweep: K = 1..10, two loads; small epochs, many changes
    reps = [((k * 3 + d) * 2 + ld) * 64 + (k + d) % 64 for k in (0, 4, 9) for d in range(3) for ld in range(2)]
    w = W.config(2, replicas=reps, requests=1500)
    sched = _check(w, [30_000 * (p + 1) for p in range(10)], epoch_steps=997)
    assert sum(len(s) for s in sched.values()) > 0


def test_set_headroom_rejects_bad_tables():
    from paper_2608_16336_gb300 import mtsim

    w = adaptive.per_replica_tables(W.config(1, replicas=range(3), requests=200))
    sim = mtsim.Simulator(w, event_log_capacity=64)
    try:
        sim.load()
        good = np.array(sim._th)
        bad = good.copy()
        bad[1, 2] = -1
        with pytest.raises(mtsim.SimError) as e:
            sim.set_headroom(bad)
        assert e.value.code == mtsim.SIM_ERR_ARG
        huge = good.copy()
        huge[0, 0] = 1 << 19
        with pytest.raises(mtsim.SimError):
            sim.set_headroom(huge)
        assert (sim._th == good).all()  # nothing changed
        sim.set_headroom(good)          # the same tables: the run is the plain one
        assert sim.run() == 0
        res, st, _ = sim.metrics()
    finally:
        sim.close()
    want = parity.run_gpu(w, event_log_capacity=64)
    assert (res == want[0]).all() and (st == want[1]).all()
