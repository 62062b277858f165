"""Per-tier latency statistics of simulated requests (TEST INFRASTRUCTURE ONLY).

Only the test suite, the package smoke check and the benchmark's CPU-baseline
leg use this module.  It states plainly what the GPU reduction computes, for
the latency measures the paper reports per priority tier (Sec. 5.1, Fig. 5-6;
Sec. 5.3 Tables 2-4: TTFT, i.e. prefill latency, time between tokens and
end-to-end latency; their means and P50 / P90 / P99):

* TTFT = first_token - arrival; E2E = finish - arrival (microseconds).
* TBT of a request with O >= 2 output tokens = floor((finish - first_token) /
  (O - 1)), its mean time between tokens; requests with O = 1 have none.
* Only finished requests count.
* Percentile p of n values: the nearest-rank value, i.e. the value of rank
  ceil(p * n / 100) in ascending order (rank 1 when that is 0), exactly (the
  paper's P50 / P90 / P99 are values of the latency distribution).
* Histogram buckets of a value v (32-bit): v itself for v < 8; otherwise,
  with e = floor(log2 v), bucket 8 + 8 (e - 3) + (floor(v / 2^(e-3)) - 8),
  i.e. eight equal buckets per power of two.  240 buckets cover every value.

Percentiles here come from sorting the exact values (no histogram and no
radix selection), so they check the GPU's selection rather than repeat it.
"""
from __future__ import annotations

import numpy as np

NONE32 = 0xFFFFFFFF
NUM_BUCKETS = 240
METRICS = ("ttft", "tbt", "e2e")
PERCENTILES = (50, 90, 99)


def bucket(v: int) -> int:
    """Histogram bucket of a non-negative 32-bit value."""
    if v < 8:
        return v
    e = v.bit_length() - 1
    return 8 + 8 * (e - 3) + ((v >> (e - 3)) - 8)


def bucket_floor(b: int) -> int:
    """Smallest value in bucket b."""
    if b < 8:
        return b
    e = (b - 8) // 8 + 3
    return (8 + (b - 8) % 8) << (e - 3)


def nearest_rank(sorted_values, p: int) -> int:
    n = len(sorted_values)
    rank = max(1, -(-p * n // 100))
    return int(sorted_values[rank - 1])


def request_latencies(arrival, output_len, first_token, finish):
    """(ttft, tbt, e2e, finished mask, has-tbt mask) as int64 arrays."""
    arrival = np.asarray(arrival, np.int64)
    first = np.asarray(first_token, np.int64)
    fin = np.asarray(finish, np.int64)
    out = np.asarray(output_len, np.int64)
    done = fin != NONE32
    ttft = first - arrival
    e2e = fin - arrival
    has_tbt = done & (out >= 2)
    tbt = np.where(has_tbt, (fin - first) // np.maximum(out - 1, 1), 0)
    return ttft, tbt, e2e, done, has_tbt


def tier_stats(values) -> dict:
    """count, sum, max, histogram and nearest-rank percentiles of one group."""
    vals = sorted(int(v) for v in values)
    hist = [0] * NUM_BUCKETS
    for v in vals:
        hist[bucket(v)] += 1
    st = {"count": len(vals), "sum": sum(vals), "max": vals[-1] if vals else 0, "hist": hist}
    for p in PERCENTILES:
        st["p%d" % p] = nearest_rank(vals, p) if vals else 0
    return st


def replica_stats(arrival, output_len, tier, first_token, finish, num_tiers: int) -> list[dict]:
    """[tier][metric] statistics of one replica's requests."""
    ttft, tbt, e2e, done, has_tbt = request_latencies(arrival, output_len, first_token, finish)
    tier = np.asarray(tier, np.int64)
    out = []
    for k in range(num_tiers):
        sel = tier == k
        out.append([tier_stats(ttft[sel & done]), tier_stats(tbt[sel & has_tbt]), tier_stats(e2e[sel & done])])
    return out
