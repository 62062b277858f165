"""Pins of the oracle's headroom schedule, the mechanism behind adaptive
headroom (Sec. 6, "Adaptive headroom allocation": H_p adjusted while the
system runs).  A schedule is a list of (step, table): before the step of
that index is processed, the table in force becomes ``table``.

* Re-setting the table in force changes nothing; a change at step 0 is
  running with that table from the start; changes after the last step do
  nothing.
* Exact agreement with the independent brute force (``tiny_ref``, Fractions)
  on tiny clusters with random schedules that change H mid-run.
* A change of H at a known step moves the dispatch it should move.
"""
import numpy as np

from oracle import oracle as O
from tests import test_oracle_pins as pins
from tests._tiny import tiny_case


def _run(n, m, headroom, trace, policy, schedule=None, so_path=None):
    cfg = O.make_config(n, m, headroom, check_invariants=1, headroom_schedule=schedule, **policy)
    return O.run_trace(cfg, *trace, so_path=so_path)


def _same_result(a, b):
    assert a.stats == b.stats
    for f in ("dispatch_instance", "final_instance", "first_token_us", "finish_us", "n_migrations", "n_preemptions"):
        np.testing.assert_array_equal(getattr(a, f), getattr(b, f))
    np.testing.assert_array_equal(a.events(), b.events())


def test_resetting_the_same_table_changes_nothing():
    for seed in range(40):
        n, m, headroom, trace, policy = tiny_case(5000 + seed)
        base = _run(n, m, headroom, trace, policy)
        steps = int(base.stats["steps"])
        sched = [(s, headroom) for s in (0, 1, steps // 3, steps // 2, steps - 1, steps + 5) if s >= 0]
        _same_result(base, _run(n, m, headroom, trace, policy, sched))


def test_change_at_step_zero_is_the_new_table():
    for seed in range(40):
        n, m, headroom, trace, policy = tiny_case(6000 + seed)
        other = [h + 3 * (k + 1) for k, h in enumerate(headroom)]
        _same_result(_run(n, m, other, trace, policy), _run(n, m, headroom, trace, policy, [(0, other)]))
        # a change after the last step does nothing
        base = _run(n, m, headroom, trace, policy)
        _same_result(base, _run(n, m, headroom, trace, policy, [(int(base.stats["steps"]) + 1, other)]))


def _schedule_for(seed, headroom, steps, m):
    rng = np.random.default_rng(seed)
    sched = []
    for s in sorted(rng.integers(0, max(steps, 1) + 2, size=int(rng.integers(1, 5)))):
        sched.append((int(s), [int(x) for x in rng.integers(0, max(2, m // 2), size=len(headroom))]))
    return sched


def check_tiny_schedule_agreement(seeds, so_path=None):
    for seed in seeds:
        n, m, headroom, trace, policy = tiny_case(7000 + seed)
        steps = int(_run(n, m, headroom, trace, policy, so_path=so_path).stats["steps"])
        sched = _schedule_for(seed, headroom, steps, m)
        res = _run(n, m, headroom, trace, policy, sched, so_path=so_path)
        p = policy
        sim = pins.tiny_ref.TinySim(
            n, m, headroom, list(zip(*trace)), t_blk=p["tokens_per_block"], bmax=p["max_batch"],
            base=p["iter_base_us"], a=p["iter_us_per_prefill_token"], b=p["iter_us_per_decode_seq"],
            s_blocks=p["migrate_blocks_per_iter"], migration=bool(p["enable_migration"]),
            interval=p["migrate_interval_us"], theta=pins.Fraction(p["theta_num"], p["theta_den"]),
            headroom_schedule=sched).run()
        pins._same(res, sim)


def test_tiny_schedule_brute_force_agreement():
    check_tiny_schedule_agreement(range(300))


def check_dispatch_follows_the_change(so_path=None):
    """Two instances, M = 100, T = 16, tiers {0, 1}.  At t = 0 a tier-0
    request (3 blocks) goes to instance 0 and a tier-1 request (10 blocks) to
    instance 1; both start their prefills.  At t = 100 (the second step) a
    tier-0 request arrives: F_0 = 100 - 3 - H_0 against F_1 = 100 - 10 - H_1
    (one running request each), so it goes to instance 0 while H_0 < 7 + H_1.
    Raising H_0 to 20 before the second step sends it to instance 1; raising
    it one step later does not."""
    trace = (np.array([0, 0, 100], np.uint32), np.array([48, 160, 16], np.uint16),
             np.array([500, 500, 2], np.uint16), np.array([0, 1, 0], np.uint8))
    pol = dict(tokens_per_block=16, enable_migration=0)
    base = _run(2, 100, [0, 0], trace, pol, so_path=so_path)
    assert list(base.dispatch_instance) == [0, 1, 0]
    steps_before_third = 1  # step 0: both arrive at t = 0; step 1: the arrival at t = 100
    moved = _run(2, 100, [0, 0], trace, pol, [(steps_before_third, [20, 0])], so_path=so_path)
    assert list(moved.dispatch_instance) == [0, 1, 1]
    late = _run(2, 100, [0, 0], trace, pol, [(steps_before_third + 1, [20, 0])], so_path=so_path)
    assert list(late.dispatch_instance) == [0, 1, 0]


def test_dispatch_follows_the_change():
    check_dispatch_follows_the_change()
