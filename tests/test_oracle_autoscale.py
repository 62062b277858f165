"""Pins of the oracle's draining and auto-scaling rules (Sec. 3.4-3.6).

* A closed-form timeline whose mean normal-priority freeness crosses both
  thresholds, including a tick where it equals the scale-in threshold
  exactly (no signal: the comparison is strict).
* Reductions: instances draining from t = 0 behave as if absent; a cluster in
  which every instance drains dispatches exactly like one without draining
  and migrates nothing; the signal is an output and changes no schedule.
* Exact brute force (``tiny_ref``: the literal minus-infinity sentinel and
  ``Fraction`` means) on hundreds of tiny clusters with random drain
  schedules and thresholds.
* No request that arrives after an instance's drain start is dispatched to it
  while another instance is not draining.
"""
from fractions import Fraction

import numpy as np
import pytest

from oracle import oracle as O
from oracle import tiny_ref
from paper_2608_16336_gb300 import workloads as W
from tests._tiny import tiny_case_drain

NEVER = O.NONE32


def _run(n, m, headroom, trace, *, drain=None, log_capacity=1 << 16, **policy):
    cfg = O.make_config(n, m, headroom, check_invariants=1, drain_start_us=drain, **policy)
    return O.run_trace(cfg, *trace, log_capacity=log_capacity)


def _signals(res):
    ev = res.events()
    out = [int(e[0]) for e in ev if e[5] == O.EV_SCALE_OUT]
    inn = [int(e[0]) for e in ev if e[5] == O.EV_SCALE_IN]
    return out, inn


def _same_requests(a, b, shift=0):
    assert a.stats["status"] == O.STATUS_DONE and b.stats["status"] == O.STATUS_DONE
    assert list(a.dispatch_instance) == list(b.dispatch_instance + shift)
    assert list(a.final_instance) == list(b.final_instance + shift)
    assert list(a.first_token_us) == list(b.first_token_us)
    assert list(a.finish_us) == list(b.finish_us)
    assert list(a.n_migrations) == list(b.n_migrations)
    assert list(a.n_preemptions) == list(b.n_preemptions)


# ------------------------------------------------------------ closed form --
# Two instances of M = 16 blocks (T = 16), batch 1, one tier with no headroom,
# migration off; four requests at t = 0 with P = 200 (13 blocks), O = 50.
# Dispatch (Sec. 3.4): r0 -> 0; r1 -> 1 (F 16 > 3); r2, r3 -> 0 (ties 3 = 3 go
# to the lowest index; queued requests behind the head add no usage).  Both
# instances run their first request from t = 0: prefill 4000 + 20 * 200 =
# 8000 us, then decodes of 4000 + 30 = 4030 us, so the j-th decode ends at
# 8000 + 4030 j and the request finishes at 8000 + 49 * 4030 = 205,470; r2 then
# runs on instance 0 from 205,470 (finish 410,940) and r3 from 410,940
# (finish 616,410).  At a tick, a running request that has produced g tokens
# holds ceil((200 + g) / 16) blocks; the head of line needs 13.
P, OUT, M, T = 200, 50, 16, 16
STEP = 4000 + 30


def _expected_mean(t):
    """Mean F_normal at tick t, from the timeline above (Sec. 3.6)."""
    def running_blocks(start):
        first = start + 4000 + 20 * P
        g = 1 + (t - first) // STEP if t >= first else 0
        return -(-(P + g) // T)

    f = []
    fin0 = 8000 + 49 * STEP
    if t < fin0:
        # instance 0: r0 running, r2 at the head of line; instance 1: r1 running
        f.append(Fraction(M - running_blocks(0) - 13, 1))
        f.append(Fraction(M - running_blocks(0), 1))
    else:
        start2 = fin0
        fin2 = start2 + 8000 + 49 * STEP
        if t < fin2:
            f.append(Fraction(M - running_blocks(start2) - 13, 1))   # r3 at the head of line
        else:
            f.append(Fraction(M - running_blocks(fin2), 1))
        f.append(Fraction(M, 1))                                     # instance 1 empty
    return sum(f) / len(f)


def test_autoscale_closed_form_timeline():
    trace = (np.zeros(4, np.uint32), np.full(4, P, np.uint16), np.full(4, OUT, np.uint16), np.zeros(4, np.uint8))
    res = _run(2, M, [0], trace, max_batch=1, enable_migration=0, autoscale=1)
    assert list(res.dispatch_instance) == [0, 1, 0, 0]
    assert list(res.finish_us) == [205_470, 205_470, 410_940, 616_410]
    ticks = range(50_000, 616_410, 50_000)
    want_out = [t for t in ticks if _expected_mean(t) < Fraction(-1, 2)]
    want_in = [t for t in ticks if _expected_mean(t) > Fraction(3, 2)]
    # the same numbers, derived by hand: means -4.5, -4.5, -5.5, -6.5 (out),
    # then 2.5, 2.5, 2, 1.5 (equal to the threshold: no signal), 9.5, 9, 8.5, 8
    assert want_out == [50_000, 100_000, 150_000, 200_000]
    assert want_in == [250_000, 300_000, 350_000, 450_000, 500_000, 550_000, 600_000]
    assert _expected_mean(400_000) == Fraction(3, 2)
    got_out, got_in = _signals(res)
    assert (got_out, got_in) == (want_out, want_in)
    assert res.stats["scale_out_signals"] == 4 and res.stats["scale_in_signals"] == 7
    # the ticks are steps of their own: 1 arrival time, 150 distinct
    # iteration-end times (r0 and r1 run in lockstep on the two instances,
    # then r2 and r3 one after the other, 50 iterations each) and 12 ticks
    assert res.stats["steps"] == 1 + 50 + 50 + 50 + 12


def test_thresholds_are_parameters():
    trace = (np.zeros(4, np.uint32), np.full(4, P, np.uint16), np.full(4, OUT, np.uint16), np.zeros(4, np.uint8))
    # scale-in at >= 3/2 - epsilon: 1.5 > 29/20 now signals at 400,000 too
    res = _run(2, M, [0], trace, max_batch=1, enable_migration=0, autoscale=1, scale_in_num=29, scale_den=20,
               scale_out_num=-10)
    out, inn = _signals(res)
    assert 400_000 in inn and out == [50_000, 100_000, 150_000, 200_000]


# ------------------------------------------------------------- reductions --
def _w0_trace(q=600):
    w = W.config(0, requests=q)
    sl = w.replica_slice(0)
    return w, (w.arrival_us[sl], w.prompt_len[sl], w.output_len[sl], w.tier[sl])


@pytest.mark.parametrize("autoscale", [0, 1])
def test_draining_from_start_is_a_smaller_cluster(autoscale):
    """Instances that drain from t = 0 never receive a request, hold nothing,
    and are left out of the mean: the cluster behaves as the others alone."""
    w, tr = _w0_trace()
    h = w.tables_h[0]
    small = _run(2, w.blocks_per_instance, h, tr, autoscale=autoscale)
    hi = _run(4, w.blocks_per_instance, h, tr, drain=[NEVER, NEVER, 0, 0], autoscale=autoscale)
    lo = _run(4, w.blocks_per_instance, h, tr, drain=[0, 0, NEVER, NEVER], autoscale=autoscale)
    _same_requests(hi, small)
    _same_requests(lo, small, shift=2)
    for r in (hi, lo):
        assert r.stats["steps"] == small.stats["steps"]
        assert r.stats["scale_out_signals"] == small.stats["scale_out_signals"]
        assert r.stats["scale_in_signals"] == small.stats["scale_in_signals"]
        assert r.stats["migrations"] == small.stats["migrations"]
    if autoscale:
        assert small.stats["scale_in_signals"] > 0


def test_all_draining_dispatches_as_without_draining():
    """When every instance drains, dispatch falls back to the least loaded
    (ordinary freeness) and no instance can receive a migration: the schedule
    is that of the same cluster without migration."""
    w, tr = _w0_trace()
    h = w.tables_h[0]
    ref = _run(4, w.blocks_per_instance, h, tr, enable_migration=0)
    alld = _run(4, w.blocks_per_instance, h, tr, drain=[0, 0, 0, 0])
    _same_requests(alld, ref)
    assert alld.stats["migrations"] == 0 and alld.stats["migration_starts"] == 0
    assert len(set(ref.dispatch_instance.tolist())) == 4


def test_signal_changes_no_schedule():
    w, tr = _w0_trace()
    h = w.tables_h[0]
    for mig in (0, 1):
        a = _run(4, w.blocks_per_instance, h, tr, enable_migration=mig)
        b = _run(4, w.blocks_per_instance, h, tr, enable_migration=mig, autoscale=1)
        _same_requests(b, a)
        assert b.stats["scale_in_signals"] + b.stats["scale_out_signals"] > 0
        if mig:
            assert b.stats["steps"] == a.stats["steps"]
        else:
            assert b.stats["steps"] > a.stats["steps"]   # ticks are events of their own


def test_no_dispatch_to_draining_instance():
    w, tr = _w0_trace(1500)
    h = w.tables_h[0]
    t_mid = int(tr[0][len(tr[0]) // 3])
    drain = np.array([NEVER, t_mid, NEVER, t_mid // 2], np.uint32)
    res = _run(4, w.blocks_per_instance, h, tr, drain=drain, autoscale=1)
    assert res.stats["status"] == O.STATUS_DONE
    arr = tr[0].astype(np.int64)
    for i in (1, 3):
        late = arr >= int(drain[i])
        assert late.any() and not (res.dispatch_instance[late] == i).any()
        assert (res.dispatch_instance[~late] == i).any()
    # the draining instances are migration sources, never destinations, once draining
    ev = res.events()
    mig = ev[np.isin(ev[:, 5], [O.EV_QUEUED, O.EV_START])]
    for t, _r, s, d, _b, _k in mig:
        assert not t >= int(drain[d])
    assert any(t >= int(drain[s]) for t, _r, s, d, _b, _k in mig)


# ------------------------------------------------------------ brute force --
def _tiny_pair(seed, so_path=None):
    n, m, headroom, trace, policy, drain = tiny_case_drain(seed)
    cfg = O.make_config(n, m, headroom, check_invariants=1, drain_start_us=drain, **policy)
    res = O.run_trace(cfg, *trace, so_path=so_path)
    p = policy
    sim = tiny_ref.TinySim(
        n, m, headroom, list(zip(*trace)), t_blk=p["tokens_per_block"], bmax=p["max_batch"], base=p["iter_base_us"],
        a=p["iter_us_per_prefill_token"], b=p["iter_us_per_decode_seq"], s_blocks=p["migrate_blocks_per_iter"],
        migration=bool(p["enable_migration"]), interval=p["migrate_interval_us"],
        theta=Fraction(p["theta_num"], p["theta_den"]), drain=[int(x) for x in drain], autoscale=True,
        scale_out=Fraction(p["scale_out_num"], p["scale_den"]), scale_in=Fraction(p["scale_in_num"], p["scale_den"]))
    return res, sim.run(), drain


def check_tiny_drain_agreement(seeds, so_path=None):
    for seed in seeds:
        res, sim, _ = _tiny_pair(seed, so_path)
        assert res.stats["status"] == O.STATUS_DONE, (seed, res.stats)
        assert list(res.dispatch_instance) == sim.out["dispatch"], seed
        assert list(res.final_instance) == sim.out["final"], seed
        assert list(res.first_token_us) == sim.out["first"], seed
        assert list(res.finish_us) == sim.out["finish"], seed
        assert list(res.n_migrations) == sim.out["mig"], seed
        assert list(res.n_preemptions) == sim.out["pre"], seed
        assert [tuple(int(x) for x in e) for e in res.events()] == [tuple(e) for e in sim.log], seed
        assert res.stats["steps"] == sim.steps, seed
        assert res.stats["scale_out_signals"] == sim.signals["out"], seed
        assert res.stats["scale_in_signals"] == sim.signals["in"], seed


def test_tiny_drain_brute_force_agreement():
    check_tiny_drain_agreement(range(400))


def test_tiny_drain_cases_exercise_every_rule():
    """The tiny drain cases must reach both signals, migrations out of a
    draining instance and the all-draining dispatch fallback."""
    kinds, drain_src, fallback = set(), 0, 0
    for seed in range(400):
        res, _sim, drain = _tiny_pair(seed)
        ev = res.events()
        kinds |= set(int(k) for k in ev[:, 5])
        drain_src += sum(1 for e in ev if e[5] in (O.EV_QUEUED, O.EV_START) and e[0] >= drain[e[2]])
        arr = np.asarray(_tiny_case_arrivals(seed), np.int64)
        fallback += int(sum(1 for a in arr if (a >= drain.astype(np.int64)).all()))
    assert {O.EV_SCALE_OUT, O.EV_SCALE_IN, O.EV_QUEUED, O.EV_START} <= kinds
    assert drain_src > 0 and fallback > 0


def _tiny_case_arrivals(seed):
    return tiny_case_drain(seed)[3][0]


def test_autoscale_arguments_are_validated():
    trace = (np.zeros(1, np.uint32), np.full(1, 16, np.uint16), np.full(1, 4, np.uint16), np.zeros(1, np.uint8))
    for bad in (dict(scale_den=0), dict(scale_den=65), dict(scale_out_num=3, scale_in_num=3),
                dict(scale_in_num=5000), dict(autoscale=2)):
        kw = dict(dict(autoscale=1), **bad)
        res = _run(2, 64, [0], trace, **kw)
        assert res.stats["status"] == -1, bad
