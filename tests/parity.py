"""Helpers that run a workload on the GPU through the C ABI and compare it,
field by field, with the CPU oracle on the same seeded inputs."""
import numpy as np

from oracle import oracle as O
from paper_2608_16336_gb300 import mtsim

STAT_FIELDS = ("steps", "iterations", "member_iterations", "events", "migrations", "preemptions",
               "migration_starts", "migration_aborts", "log_events", "finished", "scale_out_signals",
               "scale_in_signals")


def run_gpu(w, *, event_log_capacity=4096, max_steps=None, on_device=True, torch_allocator=True):
    sim = mtsim.Simulator(w, event_log_capacity=event_log_capacity, torch_allocator=torch_allocator)
    try:
        sim.load(on_device=on_device)
        if max_steps is None:
            left = sim.run()
            assert left == 0, "%d replicas unfinished" % left
        else:
            while sim.run(max_steps) > 0:
                pass
        res, st, ev = sim.metrics()
        events = [sim.events_of(ev, st, r) for r in range(w.num_replicas)]
    finally:
        sim.close()
    return res, st, events


def run_oracle(w, replicas, *, event_log_capacity=4096, nthreads=8):
    return O.run_workload(w, replicas, nthreads=nthreads, log_capacity=event_log_capacity)


def _as_i64_instance(x):
    x = x.astype(np.int64)
    x[x == mtsim.SIM_NONE16] = -1
    return x


def compare_replica(w, r, res, st, events, ref):
    sl = w.replica_slice(r)
    g = res[sl]
    where = "replica %d" % r
    assert ref.stats["status"] == 0, (where, ref.stats)
    assert int(st["status"][r]) == 0, (where, int(st["status"][r]))
    np.testing.assert_array_equal(_as_i64_instance(g["dispatch_instance"]), ref.dispatch_instance, err_msg=where)
    np.testing.assert_array_equal(g["first_token_us"], ref.first_token_us, err_msg=where)
    np.testing.assert_array_equal(g["finish_us"], ref.finish_us, err_msg=where)
    np.testing.assert_array_equal(_as_i64_instance(g["final_instance"]), ref.final_instance, err_msg=where)
    np.testing.assert_array_equal(g["n_migrations"].astype(np.int64), ref.n_migrations.astype(np.int64) & 0xFFFF,
                                  err_msg=where)
    np.testing.assert_array_equal(g["n_preemptions"].astype(np.int64), ref.n_preemptions.astype(np.int64) & 0xFFFF,
                                  err_msg=where)
    np.testing.assert_array_equal(events[r], ref.events(), err_msg=where)
    for f in STAT_FIELDS:
        assert int(st[f][r]) == int(ref.stats[f]), (where, f, int(st[f][r]), ref.stats[f])
    assert int(st["last_time_us"][r]) == int(ref.stats["last_time"]), where


def check_parity(w, replicas=None, **kw):
    cap = kw.pop("event_log_capacity", 4096)
    res, st, events = run_gpu(w, event_log_capacity=cap, **kw)
    reps = list(range(w.num_replicas)) if replicas is None else list(replicas)
    ref = run_oracle(w, reps, event_log_capacity=cap)
    for r in reps:
        compare_replica(w, r, res, st, events, ref[r])
    return res, st, events


def check_properties(w, res, st, chunk=1 << 24):
    """Checks that hold for every replica at any size: every request finished
    once, on a valid instance, no earlier than the iteration-time model allows.
    Large traces are checked ``chunk`` records at a time."""
    assert (st["status"] == 0).all()
    assert (st["finished"].astype(np.int64) == np.diff(w.offsets)).all()
    for a in range(0, w.total_requests, chunk):
        b = min(a + chunk, w.total_requests)
        g = res[a:b]
        first = g["first_token_us"].astype(np.int64)
        fin = g["finish_us"].astype(np.int64)
        arr = w.arrival_us[a:b].astype(np.int64)
        assert (first != mtsim.SIM_NONE32).all() and (fin != mtsim.SIM_NONE32).all()
        assert (first - arr >= w.iter_base_us + w.iter_us_per_prefill_token * w.prompt_len[a:b].astype(np.int64)).all()
        assert (fin - first >= (w.output_len[a:b].astype(np.int64) - 1) * (w.iter_base_us + w.iter_us_per_decode_seq)).all()
        assert (g["dispatch_instance"] < w.num_instances).all()
        assert (g["final_instance"] < w.num_instances).all()
