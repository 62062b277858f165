"""Pins of the per-tier latency statistics (``oracle/latency.py``).

* The bucket function against its defining properties, by brute force:
  every value lies in [floor(b), floor(b + 1)), buckets are contiguous and
  ordered, eight per power of two, at most 1/8 of their floor wide.
* Nearest-rank percentiles against numpy's ``inverted_cdf`` percentile, and
  the statistics' P50 / P90 / P99 equal to it on the values themselves.
* Closed forms for a lone request: TTFT = base + a P, TBT = base + b,
  E2E = TTFT + (O - 1)(base + b) under the iteration-time model.
"""
import numpy as np
import pytest

from oracle import latency as LT
from oracle import oracle as O


def test_bucket_bounds_brute_force():
    rng = np.random.default_rng(0)
    vals = list(range(0, 5000)) + [int(x) for x in rng.integers(0, 1 << 32, size=20000)]
    vals += [(1 << e) + d for e in range(3, 32) for d in (-1, 0, 1)] + [0xFFFFFFFF]
    for v in vals:
        b = LT.bucket(v)
        assert 0 <= b < LT.NUM_BUCKETS
        lo = LT.bucket_floor(b)
        hi = LT.bucket_floor(b + 1) if b + 1 < LT.NUM_BUCKETS else 1 << 32
        assert lo <= v < hi, (v, b, lo, hi)
    assert LT.bucket(0xFFFFFFFF) == LT.NUM_BUCKETS - 1


def test_buckets_contiguous_and_eight_per_octave():
    floors = [LT.bucket_floor(b) for b in range(LT.NUM_BUCKETS)]
    assert floors[:9] == list(range(9))
    assert all(a < b for a, b in zip(floors, floors[1:]))
    for e in range(3, 32):
        inside = [b for b in range(LT.NUM_BUCKETS) if (1 << e) <= floors[b] < (1 << (e + 1))]
        assert len(inside) == 8
        widths = {floors[b + 1] - floors[b] if b + 1 < LT.NUM_BUCKETS else (1 << 32) - floors[b] for b in inside}
        assert widths == {1 << (e - 3)}
        assert max(widths) * 8 <= 1 << e       # at most 1/8 of the bucket's floor
    for b in range(LT.NUM_BUCKETS):
        assert LT.bucket(floors[b]) == b


@pytest.mark.parametrize("n", [1, 2, 3, 99, 100, 101, 1000, 4097])
def test_nearest_rank_matches_numpy(n):
    rng = np.random.default_rng(n)
    v = np.sort(rng.integers(0, 10 ** 7, size=n))
    for p in (1, 50, 90, 99, 100):
        assert LT.nearest_rank(v, p) == int(np.percentile(v, p, method="inverted_cdf"))


@pytest.mark.parametrize("seed,n", [(3, 5000), (4, 1), (5, 2), (6, 7), (7, 101)])
def test_percentiles_are_exact_values(seed, n):
    rng = np.random.default_rng(seed)
    v = rng.lognormal(10, 2, size=n).astype(np.int64)
    st = LT.tier_stats(v)
    assert sum(st["hist"]) == st["count"] == n
    assert st["sum"] == int(v.sum()) and st["max"] == int(v.max())
    for p in LT.PERCENTILES:
        assert st["p%d" % p] == int(np.percentile(v, p, method="inverted_cdf"))
        assert st["p%d" % p] in set(int(x) for x in v)


def test_percentiles_with_ties_and_extremes():
    v = [7] * 50 + [0xFFFFFFFF] * 49 + [0]
    st = LT.tier_stats(v)
    assert (st["p50"], st["p90"], st["p99"]) == (7, 0xFFFFFFFF, 0xFFFFFFFF)
    st = LT.tier_stats([5, 5, 5])
    assert (st["p50"], st["p90"], st["p99"]) == (5, 5, 5)
    assert LT.tier_stats([])["p99"] == 0


def test_lone_request_closed_forms():
    P, Ob, a0 = 553, 221, 1000
    cfg = O.make_config(4, 1024, [256, 128])
    res = O.run_trace(cfg, np.array([a0], np.uint32), np.array([P], np.uint16), np.array([Ob], np.uint16),
                      np.array([1], np.uint8))
    st = LT.replica_stats([a0], [Ob], [1], res.first_token_us, res.finish_us, 2)
    ttft, tbt, e2e = st[1]
    assert ttft["count"] == tbt["count"] == e2e["count"] == 1
    assert ttft["sum"] == 4000 + 20 * P
    assert tbt["sum"] == 4000 + 30
    assert e2e["sum"] == 4000 + 20 * P + (Ob - 1) * (4000 + 30)
    for s in (ttft, tbt, e2e):
        assert s["p50"] == s["p90"] == s["p99"] == s["sum"]
    assert all(s["count"] == 0 for s in st[0])


def test_single_token_requests_have_no_tbt():
    st = LT.replica_stats([0, 0], [1, 3], [0, 0], [100, 200], [100, 400], 1)
    ttft, tbt, e2e = st[0]
    assert ttft["count"] == 2 and e2e["count"] == 2 and tbt["count"] == 1 and tbt["sum"] == 100
    # unfinished requests are not counted
    st = LT.replica_stats([0, 0], [1, 3], [0, 0], [100, O.NONE32], [100, O.NONE32], 1)
    assert st[0][0]["count"] == 1 and st[0][1]["count"] == 0
