"""Pins of the CPU oracle against what the paper and the mathematics fix.

* Sec. 3.3 Fig. 3 / Eq. 3: the exponential headroom schedule's printed values.
* Sec. 3.2 Fig. 2 / Eq. 1-2 and Sec. 3.3 Eq. 4: the worked virtual-usage bar.
* Closed forms of the iteration-time model for one and two requests.
* Exact brute force (``tiny_ref``, Fractions) on hundreds of tiny clusters.
* The K = 2 reduction to the original binary Llumnix headroom (Sec. 3.3).
* K = 1: the headroom is one constant added whenever the instance holds a
  request, and with H0 = 0 the schedule is plain freeness-balanced vLLM.
* Invariants (KV-block conservation, tier isolation, per-tier counts).
* The paper's qualitative per-tier TTFT ordering (Sec. 5.1).
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import oracle as O
from oracle import tiny_ref
from paper_2608_16336_gb300 import workloads as W
from tests._tiny import tiny_case

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ------------------------------------------------------------- headroom --
def test_headroom_schedule_matches_figure():
    g = _golden("headroom_schedule.json")
    m = 10 ** 7  # large M so flooring to whole blocks is below the figure's rounding
    h = W.headroom_exp_table(m, g["num_tiers"], g["h_max"], g["lambda"])
    pct = [100.0 * x / m for x in h]
    for got, want in zip(pct, g["percent_of_capacity"]):
        assert abs(got - want) <= g["percent_rounding"] + 1e-9, (pct, g)
    assert abs(sum(pct) - g["total_percent"]) <= g["total_rounding"]
    # tier 0 gets the most, each later tier less (Eq. 3, lambda > 0)
    assert all(a > b for a, b in zip(h, h[1:]))


def test_integer_decay_table():
    assert W.headroom_decay_table(256, 2) == [256, 128]
    assert W.headroom_decay_table(512, 4) == [512, 256, 128, 64]
    assert W.headroom_decay_table(1024, 10)[-1] == 2
    # floor(H0 * 0.5^k) written as a float product agrees with the shift
    for h0 in (1, 7, 512, 1000, 65535):
        assert W.headroom_decay_table(h0, 12) == [int(math.floor(h0 * 0.5 ** k)) for k in range(12)]


# ------------------------------------------------------------- freeness --
def test_virtual_usage_worked_example():
    g = _golden("virtual_usage_example.json")
    # one running tier-0 request holding phys blocks; the HoL request is tier 1
    cfg = O.make_config(1, g["capacity_blocks"], [g["tier_headroom_blocks"], 0])
    num, den = O.freeness(cfg, [g["phys_running_blocks"]], g["hol_demand_blocks"], [1, 1])
    assert den == 1
    assert g["capacity_blocks"] - num == g["virtual_usage_blocks"]
    assert num == g["freeness_times_batch"] == g["free_blocks"]


def test_freeness_terms_individually():
    cfg = O.make_config(1, 1000, [100, 40, 7])
    # nothing present: F = M / 1
    assert O.freeness(cfg, [], 0, [0, 0, 0]) == (1000, 1)
    # headroom once per present tier, not per request (Eq. 4)
    assert O.freeness(cfg, [10, 20, 30], 0, [3, 0, 0]) == (1000 - 60 - 100, 3)
    assert O.freeness(cfg, [10, 20, 30], 0, [1, 1, 1]) == (1000 - 60 - 147, 3)
    # HoL demand counts, the rest of the queue does not (Eq. 2)
    assert O.freeness(cfg, [10], 25, [1, 5, 0]) == (1000 - 10 - 25 - 140, 1)
    # inbound migration copy is occupied memory
    assert O.freeness(cfg, [10], 0, [1, 0, 0], reserved_in=64) == (1000 - 10 - 100 - 64, 1)
    # F goes negative when headroom plus demand exceed M (Sec. 3.2)
    n, d = O.freeness(cfg, [900], 80, [1, 0, 1])
    assert n < 0 and d == 1


# ---------------------------------------------------------- closed forms --
def _single(n, P, Ob, arrival=1000, migration=1, m=1024):
    cfg = O.make_config(n, m, [256, 128], enable_migration=migration, check_invariants=1)
    res = O.run_trace(cfg, np.array([arrival], np.uint32), np.array([P], np.uint16), np.array([Ob], np.uint16),
                      np.array([1], np.uint8))
    assert res.stats["status"] == O.STATUS_DONE
    return res


@pytest.mark.parametrize("n", [1, 4])
@pytest.mark.parametrize("migration", [0, 1])
@pytest.mark.parametrize("P,Ob", [(16, 8), (553, 221), (4096, 2048), (1, 1), (17, 2)])
def test_single_request_closed_form(n, migration, P, Ob):
    res = _single(n, P, Ob, migration=migration)
    ttft = int(res.first_token_us[0]) - 1000
    e2e = int(res.finish_us[0]) - 1000
    assert ttft == 4000 + 20 * P
    assert e2e == ttft + (Ob - 1) * (4000 + 30)
    assert res.dispatch_instance[0] == 0          # all instances equally free: lowest index
    assert res.n_preemptions[0] == 0


def test_two_simultaneous_requests_closed_form():
    P1, O1, P2, O2 = 100, 5, 300, 9
    cfg = O.make_config(1, 1024, [0], check_invariants=1)
    res = O.run_trace(cfg, np.array([0, 0], np.uint32), np.array([P1, P2], np.uint16),
                      np.array([O1, O2], np.uint16), np.array([0, 0], np.uint8))
    t1 = 4000 + 20 * (P1 + P2)
    assert list(res.first_token_us) == [t1, t1]
    # decode iterations with both alive until the shorter finishes
    f1 = t1 + (O1 - 1) * (4000 + 30 * 2)
    f2 = f1 + (O2 - O1) * (4000 + 30 * 1)
    assert list(res.finish_us) == [f1, f2]
    assert res.stats["iterations"] == O2
    assert res.stats["steps"] == O2 + 1            # the arrival time plus one per iteration end


def check_threshold_equality(so_path=None):
    """Sec. 3.5 migrates when max F - min F >= theta: equality triggers.  Two
    instances each run one long request that holds one KV block (T = 64,
    P = 1), so at the 50 ms tick both have F = (10 - 1) / 1: a difference of
    exactly 0.  With theta = 0 the tick pairs them (source: least free, lowest
    index = 0; destination: 1) and starts a staged copy of request 0, which
    commits at instance 0's next iteration end, 4,020 + 12 * 4,030 us.  With
    theta = 1/1000 nothing moves at the tick."""
    tr = (np.array([0, 1], np.uint32), np.array([1, 1], np.uint16), np.array([600, 600], np.uint16),
          np.array([0, 0], np.uint8))
    cfg = O.make_config(2, 10, [0], tokens_per_block=64, theta_num=0, theta_den=1, check_invariants=1)
    ev = O.run_trace(cfg, *tr, so_path=so_path).events()
    assert ev[:2].tolist() == [[50_000, 0, 0, 1, 1, O.EV_START], [4020 + 12 * 4030, 0, 0, 1, 1, O.EV_COMMIT]]
    cfg = O.make_config(2, 10, [0], tokens_per_block=64, theta_num=1, theta_den=1000, check_invariants=1)
    ev = O.run_trace(cfg, *tr, so_path=so_path).events()
    assert ev.shape[0] == 0 or ev[0, 0] > 50_000


def test_migration_threshold_equality():
    check_threshold_equality()


# ----------------------------------------------------------- brute force --
def _oracle_tiny(n, m, headroom, trace, policy, so_path=None):
    cfg = O.make_config(n, m, headroom, check_invariants=1, **policy)
    return O.run_trace(cfg, *trace, so_path=so_path)


def _tiny_ref(n, m, headroom, trace, policy, binary=False, binary_h=0):
    p = policy
    sim = tiny_ref.TinySim(
        n, m, headroom, list(zip(*trace)), t_blk=p["tokens_per_block"], bmax=p["max_batch"], base=p["iter_base_us"],
        a=p["iter_us_per_prefill_token"], b=p["iter_us_per_decode_seq"], s_blocks=p["migrate_blocks_per_iter"],
        migration=bool(p["enable_migration"]), interval=p["migrate_interval_us"],
        theta=Fraction(p["theta_num"], p["theta_den"]), binary=binary, binary_h=binary_h)
    return sim.run()


def _same(res, sim):
    assert res.stats["status"] == O.STATUS_DONE, res.stats
    assert list(res.dispatch_instance) == sim.out["dispatch"]
    assert list(res.final_instance) == sim.out["final"]
    assert list(res.first_token_us) == sim.out["first"]
    assert list(res.finish_us) == sim.out["finish"]
    assert list(res.n_migrations) == sim.out["mig"]
    assert list(res.n_preemptions) == sim.out["pre"]
    assert [tuple(int(x) for x in e) for e in res.events()] == [tuple(e) for e in sim.log]
    assert res.stats["steps"] == sim.steps


def check_tiny_agreement(seeds, so_path=None):
    for seed in seeds:
        n, m, headroom, trace, policy = tiny_case(seed)
        res = _oracle_tiny(n, m, headroom, trace, policy, so_path)
        sim = _tiny_ref(n, m, headroom, trace, policy)
        _same(res, sim)


def test_tiny_brute_force_agreement():
    check_tiny_agreement(range(400))


def test_tiny_cases_exercise_every_rule():
    """The tiny cases must reach preemption, queued and running migration,
    commits and aborts, or the brute-force pin would not cover them."""
    kinds, pre = set(), 0
    for seed in range(400):
        n, m, headroom, trace, policy = tiny_case(seed)
        res = _oracle_tiny(n, m, headroom, trace, policy)
        kinds |= set(int(k) for k in res.events()[:, 5])
        pre += int(res.n_preemptions.sum())
    assert kinds == {O.EV_QUEUED, O.EV_START, O.EV_COMMIT, O.EV_ABORT}
    assert pre > 0


def test_k1_headroom_is_one_shift_when_present():
    """K = 1 (Sec. 3.3 Eq. 4 with one tier): U = U(H0 = 0) + H0 when the
    instance holds any request, U(H0 = 0) when it holds none."""
    for h0 in (0, 1, 37, 512):
        cfg, cfg0 = O.make_config(1, 2048, [h0]), O.make_config(1, 2048, [0])
        for running, hol, cnt in (([], 0, 0), ([], 12, 1), ([5, 9], 0, 2), ([5, 9, 30], 7, 5)):
            n, d = O.freeness(cfg, running, hol, [cnt])
            n0, d0 = O.freeness(cfg0, running, hol, [cnt])
            assert d == d0 == max(len(running), 1)
            assert n == n0 - (h0 if cnt > 0 else 0)
            assert n0 == 2048 - sum(running) - hol


def test_k1_h0_zero_closed_form_dispatch():
    """K = 1, H0 = 0 on three empty instances: each arrival goes to the
    freest instance, lowest index on ties (Sec. 3.4); the fourth finds all
    three equally loaded and joins instance 0's running prefill's next batch."""
    P, Ob, T, base, a, b = 160, 50, 16, 4000, 20, 30
    cfg = O.make_config(3, 2048, [0], tokens_per_block=T, enable_migration=0)
    res = O.run_trace(cfg, np.array([0, 1, 2, 3], np.uint32), np.full(4, P, np.uint16), np.full(4, Ob, np.uint16),
                      np.zeros(4, np.uint8))
    assert list(res.dispatch_instance) == [0, 1, 2, 0]
    t0 = base + a * P                       # request 0's prefill iteration ends
    assert int(res.first_token_us[0]) == t0
    assert int(res.first_token_us[1]) - 1 == t0 and int(res.first_token_us[2]) - 2 == t0
    # request 3 waited for that iteration, then shares one with request 0's first decode
    assert int(res.first_token_us[3]) == t0 + base + a * P + b * 1


def test_k1_h0_zero_is_plain_freeness_balanced_vllm():
    """With one tier and no headroom the multi-tier scheduler must give the
    schedule of the original Llumnix rule with no high-priority headroom,
    computed by the independent brute force (Fractions): freeness
    (M - running KV - HoL demand) / B only, FCFS local queues."""
    for seed in range(150):
        n, m, _, trace, policy = tiny_case(3000 + seed)
        trace = (trace[0], trace[1], trace[2], np.zeros_like(trace[3]))
        res = _oracle_tiny(n, m, [0], trace, policy)
        sim = _tiny_ref(n, m, [0, 0], (trace[0], trace[1], trace[2], np.ones_like(trace[3])), policy,
                        binary=True, binary_h=0)
        _same(res, sim)
        # and K = 3 with all headroom zero and every request in tier 0 is the same schedule
        res3 = _oracle_tiny(n, m, [0, 0, 0], trace, policy)
        assert list(res3.dispatch_instance) == list(res.dispatch_instance)
        assert list(res3.finish_us) == list(res.finish_us)
        assert [tuple(e) for e in res3.events().tolist()] == [tuple(e) for e in res.events().tolist()]


def test_k2_reduces_to_binary_llumnix():
    """With K = 2 and table {h, 0}, the multi-tier rule charges h whenever a
    high-priority request is present; the original rule charges h/numHigh to
    each of them (Sec. 3.3).  Both give the same schedule."""
    for seed in range(150):
        n, m, _, trace, policy = tiny_case(1000 + seed)
        tier = (trace[3] % 2).astype(np.uint8)
        trace = (trace[0], trace[1], trace[2], tier)
        h = int(np.random.default_rng(seed).integers(0, m // 2 + 1))
        res = _oracle_tiny(n, m, [h, 0], trace, policy)
        sim = _tiny_ref(n, m, [h, 0], trace, policy, binary=True, binary_h=h)
        _same(res, sim)


# ------------------------------------------------------------ invariants --
def _check_outputs(w, res_by_rep):
    for r, res in res_by_rep.items():
        sl = w.replica_slice(r)
        assert res.stats["status"] == O.STATUS_DONE, (r, res.stats)
        arr = w.arrival_us[sl].astype(np.int64)
        P = w.prompt_len[sl].astype(np.int64)
        Ob = w.output_len[sl].astype(np.int64)
        first = res.first_token_us.astype(np.int64)
        fin = res.finish_us.astype(np.int64)
        assert (fin != O.NONE32).all() and (first != O.NONE32).all()
        assert (first - arr >= w.iter_base_us + w.iter_us_per_prefill_token * P).all()
        assert (fin - first >= (Ob - 1) * (w.iter_base_us + w.iter_us_per_decode_seq)).all()
        assert ((res.dispatch_instance >= 0) & (res.dispatch_instance < w.num_instances)).all()
        assert res.stats["finished"] == len(arr)


def test_invariants_workload0():
    w = W.config(0)
    res = O.run_workload(w, check_invariants=1)
    _check_outputs(w, res)


def test_invariants_workload_samples():
    for cid, reps in ((1, [0, 1]), (2, [0, 700, 2300, 3839])):
        w = W.config(cid, replicas=reps, requests=3000)
        res = O.run_workload(w, check_invariants=1, nthreads=4)
        _check_outputs(w, {i: res[i] for i in range(len(reps))})


def test_invariants_under_memory_pressure():
    """Small KV capacity and long prompts force preemption and aborts."""
    w = W.config(1, replicas=[3], requests=2000)
    w.blocks_per_instance = 300
    w.tables_h = [[64, 32, 16, 8]]
    w.prompt_len = np.minimum(w.prompt_len, 2400).astype(np.uint16)
    res = O.run_workload(w, check_invariants=1)
    _check_outputs(w, {0: res[0]})
    assert res[0].stats["preemptions"] > 0
    assert res[0].stats["migration_aborts"] > 0


def test_migration_switches():
    w = W.config(0, requests=400)
    on = O.run_workload(w)[0]
    assert on.stats["log_events"] > 0
    w.enable_migration = 0
    off = O.run_workload(w)[0]
    assert off.stats["log_events"] == 0 and int(off.n_migrations.sum()) == 0
    w.enable_migration = 1
    w.theta_num, w.theta_den = 10 ** 6, 1
    never = O.run_workload(w)[0]
    assert never.stats["log_events"] == 0


def test_trace_validation():
    cfg = O.make_config(2, 64, [8, 4])
    a = np.array([10, 5], np.uint32)
    p = np.array([4, 4], np.uint16)
    o = np.array([4, 4], np.uint16)
    assert O.run_trace(cfg, a, p, o, np.array([0, 1], np.uint8)).stats["status"] == -2   # unsorted
    a = np.array([5, 10], np.uint32)
    assert O.run_trace(cfg, a, p, o, np.array([0, 2], np.uint8)).stats["status"] == -2   # tier >= K
    assert O.run_trace(cfg, a, np.array([0, 4], np.uint16), o, np.array([0, 1], np.uint8)).stats["status"] == -2
    assert O.run_trace(cfg, a, np.array([1021, 4], np.uint16), o, np.array([0, 1], np.uint8)).stats["status"] == -2  # P+O > M*T
    assert O.run_trace(cfg, a, p, o, np.array([0, 1], np.uint8)).stats["status"] == 0


def test_empty_trace():
    cfg = O.make_config(3, 64, [8])
    z = np.zeros(0, np.uint32)
    res = O.run_trace(cfg, z, z.astype(np.uint16), z.astype(np.uint16), z.astype(np.uint8))
    assert res.stats["status"] == 0 and res.stats["steps"] == 0


def test_step_limit_stops_early():
    w = W.config(0, requests=200)
    full = O.run_workload(w)[0]
    part = O.run_workload(w, max_steps=50)[0]
    assert part.stats["status"] == O.STATUS_INCOMPLETE and part.stats["steps"] == 50
    assert full.stats["status"] == 0 and full.stats["steps"] > 50


# -------------------------------------------------- paper-level behaviour --
def test_tier_ttft_ordering_under_load():
    """Sec. 5.1: with K = 3 tiers under load, tier 0 is served first and tier 2
    last (median TTFT ordered by tier)."""
    T, BMAX, N, M = 16, 64, 4, 1024
    rate = W._load_rate(0.95, N, M, T, BMAX, W.LEN_DEFAULT)
    p = W._params(7, 6000, 3, W.tier_probs("uniform", 3), rate, W.LEN_DEFAULT)
    off, arr, pl, ol, tr = W.generate([p])
    w = W.custom(N, M, [3], [W.headroom_decay_table(256, 3)], [0], [(arr, pl, ol, tr)])
    res = O.run_workload(w)[0]
    ttft = res.first_token_us.astype(np.int64) - arr
    med = [np.median(ttft[tr == k]) for k in range(3)]
    assert med[0] < med[1] < med[2], med


def test_deterministic():
    w = W.config(1, replicas=[5], requests=2000)
    a = O.run_workload(w)[0]
    b = O.run_workload(w)[0]
    assert (a.finish_us == b.finish_us).all() and (a.events() == b.events()).all()
    assert a.stats == b.stats
