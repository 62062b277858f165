"""Seeded tiny traces and cluster shapes for brute-force comparisons."""
import numpy as np


def tiny_case(seed: int, *, max_instances: int = 3, max_requests: int = 14):
    """A random tiny cluster and trace chosen to exercise every rule: few KV
    blocks (preemption), small batches, frequent migration ticks, colliding
    arrival times and several tiers."""
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, max_instances + 1))
    t_blk = int(rng.integers(2, 5))
    m = int(rng.integers(6, 24))
    bmax = int(rng.integers(1, 5))
    k = int(rng.integers(1, 4))
    headroom = [int(x) for x in sorted(rng.integers(0, max(2, m // 3), size=k), reverse=True)]
    q = int(rng.integers(1, max_requests + 1))
    gaps = rng.choice([0, 0, 1, 5, 40, 120, 300], size=q)
    arrival = np.cumsum(gaps).astype(np.uint32)
    cap = m * t_blk
    plen = rng.integers(1, max(2, cap // 2), size=q)
    olen = rng.integers(1, 12, size=q)
    olen = np.minimum(olen, cap - plen)
    olen = np.maximum(olen, 1)
    tier = rng.integers(0, k, size=q).astype(np.uint8)
    policy = dict(tokens_per_block=t_blk, max_batch=bmax, iter_base_us=int(rng.integers(20, 120)),
                  iter_us_per_prefill_token=int(rng.integers(0, 4)), iter_us_per_decode_seq=int(rng.integers(0, 6)),
                  migrate_blocks_per_iter=int(rng.integers(1, 5)), enable_migration=int(rng.integers(0, 4) > 0),
                  migrate_interval_us=int(rng.integers(30, 400)), theta_num=3, theta_den=10)
    trace = (arrival, plen.astype(np.uint16), olen.astype(np.uint16), tier)
    return n, m, headroom, trace, policy


def tiny_case_drain(seed: int):
    """A tiny case (as ``tiny_case``) with a drain schedule and the
    auto-scaling signal on.  Drain starts fall anywhere in the trace's time
    span (or never); in about one case in six every instance drains, so the
    dispatch fallback is reached.  Thresholds are random fractions around the
    small freeness values of tiny clusters so that both signals fire."""
    n, m, headroom, trace, policy = tiny_case(seed, max_instances=4)
    rng = np.random.default_rng(10_000 + seed)
    span = int(trace[0][-1]) + 400
    drain = np.full(n, 0xFFFFFFFF, np.uint32)
    # half of the start times fall exactly on an arrival, where ">=" matters
    times = np.concatenate([trace[0].astype(np.int64), rng.integers(0, span, size=trace[0].shape[0])])
    if rng.integers(0, 6) == 0:
        drain[:] = rng.choice(times, size=n)
    else:
        pick = rng.random(n) < 0.4
        drain[pick] = rng.choice(times, size=int(pick.sum()))
    den = int(rng.integers(1, 5))
    out_num = int(rng.integers(-6 * den, 2 * den))
    in_num = out_num + int(rng.integers(1, 8 * den))
    policy = dict(policy, autoscale=1, scale_out_num=out_num, scale_in_num=in_num, scale_den=den)
    return n, m, headroom, trace, policy, drain
