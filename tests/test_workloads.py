"""The seeded input generator: determinism, sortedness, shapes of the
length, tier and arrival distributions, and the five workload definitions."""
import math

import numpy as np

from paper_2608_16336_gb300 import workloads as W


def test_deterministic_and_sorted():
    a = W.config(1, replicas=range(4), requests=3000)
    b = W.config(1, replicas=range(4), requests=3000, nthreads=1)
    for f in ("arrival_us", "prompt_len", "output_len", "tier"):
        assert (getattr(a, f) == getattr(b, f)).all()
    for r in range(4):
        arr = a.arrival_us[a.replica_slice(r)]
        assert (np.diff(arr.astype(np.int64)) >= 0).all()
    c = W.config(1, replicas=range(4), requests=3000, seed_block=1)
    assert (c.arrival_us != a.arrival_us).any()


def test_subset_keeps_the_replicas_traces():
    full = W.config(2, replicas=[5, 6, 7], requests=500)
    sub = full.subset([2, 0])
    assert (sub.arrival_us[sub.replica_slice(0)] == full.arrival_us[full.replica_slice(2)]).all()
    assert (sub.tier[sub.replica_slice(1)] == full.tier[full.replica_slice(0)]).all()
    alone = W.config(2, replicas=[7], requests=500)
    assert (alone.prompt_len == full.prompt_len[full.replica_slice(2)]).all()


def test_length_distributions():
    w = W.config(1, replicas=range(8))
    p = w.prompt_len.astype(np.float64)
    o = w.output_len.astype(np.float64)
    assert p.min() >= 16 and p.max() <= 4096 and o.min() >= 8 and o.max() <= 2048
    # median of round(exp(N(mu, sigma))) is about exp(mu)
    assert abs(np.median(p) - math.exp(6.0)) < 0.05 * math.exp(6.0)
    assert abs(np.median(o) - math.exp(5.0)) < 0.05 * math.exp(5.0)
    assert abs(np.log(p).std() - 0.8) < 0.05


def test_tier_distributions():
    w = W.config(1, replicas=range(8))
    freq = np.bincount(w.tier, minlength=4) / len(w.tier)
    assert np.allclose(freq, [0.05, 0.15, 0.30, 0.50], atol=0.01)
    for k in range(1, 11):
        for d in ("uniform", "gaussian", "geometric", "paper_gaussian", "paper_enterprise"):
            p = W.tier_probs(d, k)
            assert len(p) == k and abs(sum(p) - 1.0) < 1e-9 and min(p) >= 0
    g = W.tier_probs("gaussian", 5)
    assert g[2] == max(g) and abs(g[1] - g[3]) < 1e-12     # centred on (K-1)/2
    geo = W.tier_probs("geometric", 4)
    assert all(b == 2 * a for a, b in zip(geo, geo[1:]))    # mass doubles toward the low tiers


def test_arrival_processes():
    w = W.config(1, replicas=range(4))
    rate = W._load_rate(0.85, 16, 2048, 16, 64, W.LEN_DEFAULT)
    gaps = np.concatenate([np.diff(w.arrival_us[w.replica_slice(r)].astype(np.float64)) for r in range(4)])
    assert abs(gaps.mean() - 1e6 / rate) < 0.02 * 1e6 / rate
    assert abs(gaps.std() / gaps.mean() - 1.0) < 0.05          # exponential gaps: CV 1
    b = W.config(3, replicas=[0], requests=100000)
    gb = np.diff(b.arrival_us.astype(np.float64))
    assert 2.4 < gb.std() / gb.mean() < 3.6                     # Gamma gaps: CV 3


def test_workload_shapes():
    shapes = {0: (1, 4, 1024, 2, 64), 1: (1024, 16, 2048, 4, 64), 3: (256, 128, 4096, 10, 32),
              4: (16384, 64, 2048, 4, 64)}
    for cid, (r, n, m, k, s) in shapes.items():
        w = W.config(cid, replicas=[0], requests=10)
        assert (w.num_instances, w.blocks_per_instance, max(w.tables_k), w.migrate_blocks_per_iter) == (n, m, k, s)
    w2 = W.config(2, requests=5)
    assert w2.num_replicas == 3840 and w2.num_instances == 32
    assert sorted(set(w2.tables_k)) == list(range(1, 11))
    # replica order ((K-1)*3 + dist)*2 + load)*64 + seed
    assert w2.labels[0] == "K1-uniform-0.6" and w2.labels[64] == "K1-uniform-0.9"
    assert w2.labels[128] == "K1-gaussian-0.6" and w2.labels[3839] == "K10-geometric-0.9"
    w0 = W.config(0)
    assert w0.tables_h == [[256, 128]] and w0.total_requests == 2000
