"""bench.py's host-side arithmetic: the algorithmic bytes of a run (the
scope table's per-unit figures times the run's exact counters), the
migration-log capacity rule and the replica start order."""
import numpy as np

import bench
from paper_2608_16336_gb300 import mtsim
from paper_2608_16336_gb300 import workloads as W


def _stats(rows):
    st = np.zeros(len(rows), mtsim.STATS_DTYPE)
    for r, (member, iters, logs) in enumerate(rows):
        st[r]["member_iterations"] = member
        st[r]["iterations"] = iters
        st[r]["log_events"] = logs
    return st


def test_algorithmic_bytes_terms():
    st = _stats([(1000, 40, 7), (500, 20, 3)])
    q = 100
    a = bench.algorithmic_bytes(q, st)
    touched = (40 + 20) + q + 2 * (7 + 3)
    assert a["touched_instance_steps"] == touched
    assert a["member_iterations"] == 1500 and a["iterations"] == 60 and a["log_records"] == 10
    # 9 B trace + 14 B result per request, 8 B per member-iteration, 64 B per
    # touched instance-step, 16 B per log record
    assert a["total"] == q * 23 + 1500 * 8 + touched * 64 + 10 * 16


def test_initial_log_capacity():
    w = W.config(1, replicas=range(3), requests=1000)
    assert bench.initial_log_capacity(w) == 1504            # 1.5 x requests, a multiple of 16
    w = W.config(1, replicas=range(2), requests=10)
    assert bench.initial_log_capacity(w) == 1024            # never below 1,024
    assert bench.initial_log_capacity(w) % 16 == 0


def test_start_order_by_predicted_work():
    wts = W.predicted_work(2)
    order = np.argsort(-wts, kind="stable")
    assert sorted(order.tolist()) == list(range(len(wts)))
    assert (np.diff(wts[order]) <= 0).all()                 # heaviest first
    # equal weights keep trace order (the 16,384-replica workload's order is the identity)
    assert (np.argsort(-W.predicted_work(4), kind="stable") == np.arange(16384)).all()
    # within a weight class, trace order
    for v in np.unique(wts):
        sel = order[wts[order] == v]
        assert (np.diff(sel) > 0).all()
