"""Adaptive headroom (Sec. 6, "Adaptive headroom allocation"): a controller
that adjusts each replica's per-tier headroom H_p while the simulation runs,
raising it for a tier whose requests miss their latency target and lowering
it when the tier's latency leaves the headroom unused.

The paper names only the direction of the adjustment.  The rule here is a
stated reading, in integers:

* The run proceeds in epochs of ``epoch_steps`` steps per replica
  (``sim_run`` with that step limit).  A replica stopped by the limit has
  processed exactly that many steps, so the tables chosen after epoch j take
  effect at step index (j + 1) * epoch_steps.
* After each epoch, for each replica and tier p, the requests of tier p that
  finished during the epoch give n_p and the sum S_p of their TTFT (the
  differences of the cumulative per-tier statistics that ``sim_latency_stats``
  computes on the device).
* If n_p > 0 and S_p > slo_p * n_p (mean TTFT above the tier's target):
  H_p <- min(h_max, H_p + max(1, floor(H_p / 4))).
* Else if n_p > 0 and 2 * S_p <= slo_p * n_p (mean TTFT at most half the
  target: the headroom is not needed): H_p <- H_p - floor(H_p / 4).
* Otherwise H_p is unchanged.

Every replica adapts its own table.  All simulation work runs in the C ABI's
kernels; this module only reads the statistics and writes the tables.
"""
from __future__ import annotations

import copy

import numpy as np

from . import mtsim


def per_replica_tables(w):
    """A copy of workload ``w`` in which every replica has a headroom table of
    its own (so that each can adapt independently); traces are shared."""
    v = copy.copy(w)
    v.tables_k = [w.replica_k(r) for r in range(w.num_replicas)]
    v.tables_h = [list(w.replica_h(r)) for r in range(w.num_replicas)]
    v.replica_table = np.arange(w.num_replicas, dtype=np.int32)
    return v


def next_tables(h, k_of, n_ttft, s_ttft, slo_us, h_max: int):
    """One step of the rule.  h: int64 [R, KT] tables in force; k_of: [R] tier
    counts; n_ttft, s_ttft: int64 [R, KT] count and TTFT sum of the requests
    that finished during the epoch; slo_us: [KT] per-tier TTFT targets."""
    h = np.asarray(h, np.int64)
    n = np.asarray(n_ttft, np.int64)
    s = np.asarray(s_ttft, np.int64)
    slo = np.asarray(slo_us, np.int64)[None, : h.shape[1]]
    present = np.arange(h.shape[1])[None, :] < np.asarray(k_of)[:, None]
    up = present & (n > 0) & (s > slo * n)
    down = present & (n > 0) & ~up & (2 * s <= slo * n)
    out = h.copy()
    out[up] = np.minimum(h_max, h[up] + np.maximum(1, h[up] // 4))
    out[down] = h[down] - h[down] // 4
    return out


def run(w, slo_us, *, epoch_steps: int, h_max: int | None = None, event_log_capacity: int = 4096,
        stream=None):
    """Simulates ``w`` (every replica with its own table) under the rule above.
    Returns (results, stats, events, schedules): the usual outputs of
    ``Simulator.metrics`` and, per replica, the list of (step, table) changes
    that were applied (the input the oracle needs to reproduce the run)."""
    v = per_replica_tables(w)
    R = v.num_replicas
    kmax = max(v.tables_k)
    slo = list(slo_us) + [slo_us[-1]] * (kmax - len(slo_us))
    h_max = v.blocks_per_instance if h_max is None else int(h_max)
    sim = mtsim.Simulator(v, event_log_capacity=event_log_capacity, stream=stream)
    try:
        sim.load()
        h = np.zeros((R, kmax), np.int64)
        for r in range(R):
            h[r, : v.tables_k[r]] = v.tables_h[r]
        k_of = np.asarray(v.tables_k)
        prev_n = np.zeros((R, kmax), np.int64)
        prev_s = np.zeros((R, kmax), np.int64)
        schedules = {r: [] for r in range(R)}
        epoch = 0
        while True:
            left = sim.run(epoch_steps)
            epoch += 1
            if left == 0:
                break
            lat = sim.latency_stats()[:, :, mtsim.SIM_LAT_TTFT]
            n = lat["count"].astype(np.int64)
            s = lat["sum_us"].astype(np.int64)
            new = next_tables(h, k_of, n - prev_n, s - prev_s, slo, h_max)
            prev_n, prev_s = n, s
            if (new != h).any():
                sim.set_headroom(new.astype(np.int32))
                for r in np.nonzero((new != h).any(axis=1))[0]:
                    schedules[int(r)].append((epoch * epoch_steps, [int(x) for x in new[r, : k_of[r]]]))
                h = new
        res, st, ev = sim.metrics()
        events = [sim.events_of(ev, st, r) for r in range(R)]
    finally:
        sim.close()
    return res, st, events, schedules
