"""The adaptive-headroom rule (paper_2608_16336_gb300/adaptive.py), host
logic on CPU: raise by a quarter (at least one block, capped) when a tier's
mean TTFT over the epoch is above its target, lower by a quarter when it is
at most half the target, leave it otherwise; tiers without finished requests
and tiers a replica does not have are left alone."""
import numpy as np

from paper_2608_16336_gb300 import adaptive
from paper_2608_16336_gb300 import workloads as W


def test_rule_directions_and_bounds():
    h = np.array([[8, 0, 100, 40], [3, 3, 3, 3]])
    k_of = [4, 2]
    slo = [100, 100, 100, 100]
    n = np.array([[2, 2, 4, 0], [1, 1, 1, 1]])
    s = np.array([[201, 250, 200, 0], [100, 50, 999, 1]])  # means 100.5, 125, 50, -; 100, 50, (tier >= K)
    out = adaptive.next_tables(h, k_of, n, s, slo, h_max=105)
    # replica 0: tier 0 above target -> 8 + 2; tier 1 above -> 0 + 1 (at least one block);
    # tier 2 at half the target -> 100 - 25; tier 3 no finished requests -> unchanged
    assert out[0].tolist() == [10, 1, 75, 40]
    # replica 1: tier 0 exactly at target -> unchanged; tier 1 at half -> 3 - 0; tiers 2, 3 absent
    assert out[1].tolist() == [3, 3, 3, 3]
    # the cap
    assert adaptive.next_tables([[104]], [1], [[1]], [[500]], [100], h_max=105).tolist() == [[105]]
    assert adaptive.next_tables([[105]], [1], [[1]], [[500]], [100], h_max=105).tolist() == [[105]]
    # lowering never goes below zero
    assert adaptive.next_tables([[1]], [1], [[1]], [[0]], [100], h_max=105).tolist() == [[1]]
    assert adaptive.next_tables([[0]], [1], [[1]], [[0]], [100], h_max=105).tolist() == [[0]]


def test_per_replica_tables_keep_the_traces():
    w = W.config(2, replicas=[0, 70, 3000], requests=50)
    v = adaptive.per_replica_tables(w)
    assert v.num_replicas == 3 and list(v.replica_table) == [0, 1, 2]
    for r in range(3):
        assert v.replica_k(r) == w.replica_k(r) and v.replica_h(r) == w.replica_h(r)
    assert v.arrival_us is w.arrival_us and w.replica_table.tolist() != [0, 1, 2]
