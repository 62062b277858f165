"""Seeded synthetic workloads: cluster shape, tier headroom tables, policy
constants and request traces for the five benchmark workloads.

This module produces inputs only.  It imports neither the CUDA binding nor
the oracle, and it holds none of the scheduling arithmetic; the trace arrays
come from ``csrc/tracegen.c`` (one xoshiro256** stream per replica).

Shapes follow the paper's evaluation setup: K priority tiers with tier 0 the
highest priority (Sec. 4.2), per-tier headroom budgets decaying exponentially
with the tier index (Sec. 3.3, Eq. 3), Poisson arrivals (Sec. 4.4), and a
50 ms migration interval with imbalance threshold 0.3 (Sec. 3.5).  Request
lengths are clipped lognormals; bursty arrivals use Gamma gaps with a given
coefficient of variation.
"""
from __future__ import annotations

import ctypes
import math
import os
from dataclasses import dataclass, field
from functools import lru_cache

import numpy as np

from . import _build

MAX_TIERS = 16
ARRIVAL_POISSON = 0
ARRIVAL_GAMMA = 1


class TgParams(ctypes.Structure):
    """Mirror of ``tg_params_t`` in csrc/tracegen.c."""

    _fields_ = [
        ("seed", ctypes.c_uint64),
        ("num_requests", ctypes.c_int64),
        ("num_tiers", ctypes.c_int32),
        ("arrival_kind", ctypes.c_int32),
        ("rate_per_s", ctypes.c_double),
        ("gamma_cv", ctypes.c_double),
        ("prompt_mu", ctypes.c_double),
        ("prompt_sigma", ctypes.c_double),
        ("prompt_min", ctypes.c_int32),
        ("prompt_max", ctypes.c_int32),
        ("output_mu", ctypes.c_double),
        ("output_sigma", ctypes.c_double),
        ("output_min", ctypes.c_int32),
        ("output_max", ctypes.c_int32),
        ("tier_probs", ctypes.c_double * MAX_TIERS),
    ]


_TG = None


def _tg():
    global _TG
    if _TG is None:
        so = _build.build_tracegen()
        lib = ctypes.CDLL(so)
        lib.tg_generate_many.restype = ctypes.c_int
        lib.tg_generate_many.argtypes = [
            ctypes.c_int, ctypes.POINTER(TgParams), ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
        ]
        lib.tg_mean_clipped_lognormal.restype = ctypes.c_double
        lib.tg_mean_clipped_lognormal.argtypes = [
            ctypes.c_double, ctypes.c_double, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64,
        ]
        lib.tg_mix_seed.restype = ctypes.c_uint64
        lib.tg_mix_seed.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        _TG = lib
    return _TG


def mix_seed(a: int, b: int) -> int:
    return int(_tg().tg_mix_seed(a, b))


@lru_cache(maxsize=64)
def mean_clipped_lognormal(mu: float, sigma: float, lo: int, hi: int, n: int = 1 << 20) -> float:
    return float(_tg().tg_mean_clipped_lognormal(mu, sigma, lo, hi, n, 12345))


# ------------------------------------------------------------------ tiers --
def tier_probs(dist: str, k: int) -> list[float]:
    """Categorical distribution over tiers 0..k-1 (tier 0 = highest priority).

    * ``uniform``: 1/K each (Sec. 4.2).
    * ``gaussian``: a normal over the tier index with mean (K-1)/2 and sd K/4,
      rounded to the nearest tier and clipped to [0, K-1].
    * ``paper_gaussian``: the paper's centre floor(K/2), sd K/4 (Sec. 4.2).
    * ``enterprise``: 0.05/0.15/0.30/0.50 for K = 4, highest tier first.
    * ``geometric``: weight 0.5^(K-1-k), i.e. mass grows toward the low tiers.
    * ``paper_enterprise``: about 10 % tier 0, 15 % tier K-1 and the rest spread
      over the middle tiers (Sec. 4.2 gives ~10 %, ~70 %, 5-20 %).
    """
    if k < 1 or k > MAX_TIERS:
        raise ValueError("tier count must be in [1, %d]" % MAX_TIERS)
    if dist == "uniform":
        return [1.0 / k] * k
    if dist in ("gaussian", "paper_gaussian"):
        mu = (k - 1) / 2.0 if dist == "gaussian" else float(k // 2)
        sd = k / 4.0
        cdf = lambda x: 0.5 * (1.0 + math.erf((x - mu) / (sd * math.sqrt(2.0))))
        p = []
        for t in range(k):
            lo = 0.0 if t == 0 else cdf(t - 0.5)
            hi = 1.0 if t == k - 1 else cdf(t + 0.5)
            p.append(max(hi - lo, 0.0))
        return p
    if dist == "enterprise":
        if k != 4:
            raise ValueError("the 4-tier enterprise mix needs K = 4; use 'geometric' or 'paper_enterprise'")
        return [0.05, 0.15, 0.30, 0.50]
    if dist == "geometric":
        w = [0.5 ** (k - 1 - t) for t in range(k)]
        s = sum(w)
        return [x / s for x in w]
    if dist == "paper_enterprise":
        if k == 1:
            return [1.0]
        if k == 2:
            return [0.10, 0.90]
        mid = 0.75 / (k - 2)
        return [0.10] + [mid] * (k - 2) + [0.15]
    raise ValueError("unknown tier distribution %r" % dist)


# --------------------------------------------------------------- headroom --
def headroom_decay_table(h0: int, k: int) -> list[int]:
    """Integer exponential decay H_k = floor(H0 * 0.5^k) (Sec. 3.3, Eq. 3 with
    e^-lambda replaced by 1/2 so the table is exact in integers)."""
    return [int(h0) >> t for t in range(k)]


def headroom_exp_table(m: int, k: int, h_max: float = 0.20, lam: float = 1.0) -> list[int]:
    """The paper's schedule H_p = M * h_max * exp(-lambda * p) (Sec. 3.3, Eq. 3),
    floored to whole blocks."""
    return [int(math.floor(m * h_max * math.exp(-lam * p))) for p in range(k)]


# ---------------------------------------------------------------- configs --
@dataclass
class Workload:
    """Everything the simulator needs: cluster, tier tables, policy, trace."""

    name: str
    num_instances: int
    blocks_per_instance: int
    tokens_per_block: int
    max_batch: int
    # tier tables: one per distinct (K, H) and a replica -> table map
    tables_k: list[int]
    tables_h: list[list[int]]
    replica_table: np.ndarray          # int32 [R]
    # policy
    iter_base_us: int = 4000
    iter_us_per_prefill_token: int = 20
    iter_us_per_decode_seq: int = 30
    migrate_blocks_per_iter: int = 64
    migrate_interval_us: int = 50_000
    theta_num: int = 3
    theta_den: int = 10
    enable_migration: int = 1
    # auto-scaling signal (Sec. 3.6): thresholds on the mean F_normal, scale_out_num/scale_den
    # and scale_in_num/scale_den (the paper's -1/2 and 3/2)
    autoscale: int = 0
    scale_out_num: int = -1
    scale_in_num: int = 3
    scale_den: int = 2
    # drain schedule (Sec. 3.5): uint32 [R, N] start times, 0xFFFFFFFF = never; None = no draining
    drain_start_us: np.ndarray = field(default=None)
    # trace (concatenated SoA, replica r owns [offsets[r], offsets[r+1]))
    offsets: np.ndarray = field(default=None)   # int64 [R+1]
    arrival_us: np.ndarray = field(default=None)
    prompt_len: np.ndarray = field(default=None)
    output_len: np.ndarray = field(default=None)
    tier: np.ndarray = field(default=None)
    labels: list[str] = field(default_factory=list)

    @property
    def num_replicas(self) -> int:
        return int(self.replica_table.shape[0])

    @property
    def total_requests(self) -> int:
        return int(self.offsets[-1])

    def replica_slice(self, r: int) -> slice:
        return slice(int(self.offsets[r]), int(self.offsets[r + 1]))

    def replica_k(self, r: int) -> int:
        return self.tables_k[int(self.replica_table[r])]

    def replica_h(self, r: int) -> list[int]:
        return self.tables_h[int(self.replica_table[r])]

    def subset(self, replicas) -> "Workload":
        """A workload made of the given replicas (their traces unchanged)."""
        idx = np.asarray(list(replicas), dtype=np.int64)
        lens = self.offsets[idx + 1] - self.offsets[idx]
        off = np.zeros(idx.shape[0] + 1, dtype=np.int64)
        np.cumsum(lens, out=off[1:])
        parts = [np.arange(self.offsets[r], self.offsets[r + 1], dtype=np.int64) for r in idx]
        sel = np.concatenate(parts) if parts else np.zeros(0, dtype=np.int64)
        w = Workload(
            name=self.name + "[subset]", num_instances=self.num_instances,
            blocks_per_instance=self.blocks_per_instance, tokens_per_block=self.tokens_per_block,
            max_batch=self.max_batch, tables_k=list(self.tables_k), tables_h=[list(h) for h in self.tables_h],
            replica_table=self.replica_table[idx].copy(),
            iter_base_us=self.iter_base_us, iter_us_per_prefill_token=self.iter_us_per_prefill_token,
            iter_us_per_decode_seq=self.iter_us_per_decode_seq,
            migrate_blocks_per_iter=self.migrate_blocks_per_iter, migrate_interval_us=self.migrate_interval_us,
            theta_num=self.theta_num, theta_den=self.theta_den, enable_migration=self.enable_migration,
            autoscale=self.autoscale, scale_out_num=self.scale_out_num, scale_in_num=self.scale_in_num,
            scale_den=self.scale_den,
            drain_start_us=None if self.drain_start_us is None else self.drain_start_us[idx].copy(),
            offsets=off, arrival_us=self.arrival_us[sel], prompt_len=self.prompt_len[sel],
            output_len=self.output_len[sel], tier=self.tier[sel],
            labels=[self.labels[r] for r in idx] if self.labels else [],
        )
        return w


def instance_capacity(m: int, t: int, bmax: int, ep: float, eo: float,
                      base: float = 4000.0, a: float = 20.0, b: float = 30.0) -> float:
    """Requests/s one instance sustains under the iteration-time model
    base + a*prefill_tokens + b*decode_seqs: prefill costs a*E[P]; each of the
    E[O] decode iterations costs b plus the base shared by B_eff requests,
    where B_eff is the batch that fits in M*T tokens at mean occupancy."""
    b_eff = min(float(bmax), m * t / (ep + eo / 2.0))
    return 1e6 / (a * ep + eo * (b + base / b_eff))


LEN_DEFAULT = dict(prompt_mu=6.0, prompt_sigma=0.8, prompt_min=16, prompt_max=4096,
                   output_mu=5.0, output_sigma=0.9, output_min=8, output_max=2048)
LEN_LONG_PROMPT = dict(LEN_DEFAULT, prompt_mu=7.0, prompt_sigma=1.0, prompt_max=8192)


def _load_rate(load: float, n: int, m: int, t: int, bmax: int, lens: dict) -> float:
    ep = mean_clipped_lognormal(lens["prompt_mu"], lens["prompt_sigma"], lens["prompt_min"], lens["prompt_max"])
    eo = mean_clipped_lognormal(lens["output_mu"], lens["output_sigma"], lens["output_min"], lens["output_max"])
    return load * n * instance_capacity(m, t, bmax, ep, eo)


def _params(seed: int, q: int, k: int, probs: list[float], rate: float, lens: dict,
            arrival_kind: int = ARRIVAL_POISSON, cv: float = 1.0) -> TgParams:
    p = TgParams()
    p.seed = seed
    p.num_requests = q
    p.num_tiers = k
    p.arrival_kind = arrival_kind
    p.rate_per_s = rate
    p.gamma_cv = cv
    for key, v in lens.items():
        setattr(p, key, v)
    for i in range(MAX_TIERS):
        p.tier_probs[i] = probs[i] if i < len(probs) else 0.0
    return p


def generate(params: list[TgParams], nthreads: int | None = None):
    """Runs the trace generator for every replica; returns the SoA arrays."""
    r = len(params)
    off = np.zeros(r + 1, dtype=np.int64)
    np.cumsum([p.num_requests for p in params], out=off[1:])
    n = int(off[-1])
    arrival = np.empty(n, dtype=np.uint32)
    plen = np.empty(n, dtype=np.uint16)
    olen = np.empty(n, dtype=np.uint16)
    tier = np.empty(n, dtype=np.uint8)
    arr = (TgParams * max(r, 1))(*params)
    nth = nthreads or min(os.cpu_count() or 1, 64)
    rc = _tg().tg_generate_many(r, arr, off.ctypes.data, arrival.ctypes.data, plen.ctypes.data,
                                olen.ctypes.data, tier.ctypes.data, nth)
    if rc != 0:
        raise RuntimeError("trace generation failed (code %d)" % rc)
    return off, arrival, plen, olen, tier


CONFIG_NAMES = {
    0: "1 replica, 4 x 1024 blocks, K=2 uniform, 2,000 requests, Poisson 8 req/s",
    1: "1,024 replicas, 16 x 2048 blocks, K=4 enterprise, 20,000 requests/replica, Poisson 0.85 load",
    2: "3,840-replica sweep, 32 x 2048 blocks, K=1..10 x {uniform, gaussian, geometric} x {0.6, 0.9} load x 64 seeds, 10,000 requests/replica",
    3: "256 replicas, 128 x 4096 blocks, K=10 gaussian, 200,000 requests/replica, Gamma CV=3 at 0.95 load, 32 migration blocks/iteration",
    4: "16,384 replicas, 64 x 2048 blocks, K=4 enterprise, 50,000 requests/replica, Poisson 0.9 load",
}


def _specs(cid: int):
    """Shape of workload ``cid``: (N, M, Q, S, per-replica specs, arrival kind, CV).
    Each spec holds K, the tier distribution, the arrival rate, the load it
    corresponds to, the length model, H0 and a label."""
    T, BMAX = 16, 64
    if cid == 0:
        n, m, q, s = 4, 1024, 2000, 64
        cap = n * instance_capacity(m, T, BMAX, *_mean_lens(LEN_DEFAULT))
        specs = [dict(k=2, dist="uniform", rate=8.0, load=8.0 / cap, lens=LEN_DEFAULT, h0=256, label="K2-uniform")]
        return n, m, q, s, specs, ARRIVAL_POISSON, 1.0
    if cid == 1:
        n, m, q, s = 16, 2048, 20000, 64
        rate = _load_rate(0.85, n, m, T, BMAX, LEN_DEFAULT)
        spec = dict(k=4, dist="enterprise", rate=rate, load=0.85, lens=LEN_DEFAULT, h0=512, label="K4-enterprise")
        return n, m, q, s, [spec] * 1024, ARRIVAL_POISSON, 1.0
    if cid == 2:
        n, m, q, s = 32, 2048, 10000, 64
        specs = []
        for k in range(1, 11):
            for dist in ("uniform", "gaussian", "geometric"):
                for load in (0.6, 0.9):
                    rate = _load_rate(load, n, m, T, BMAX, LEN_DEFAULT)
                    for _seed in range(64):
                        specs.append(dict(k=k, dist=dist, rate=rate, load=load, lens=LEN_DEFAULT, h0=512,
                                          label="K%d-%s-%.1f" % (k, dist, load)))
        return n, m, q, s, specs, ARRIVAL_POISSON, 1.0
    if cid == 3:
        n, m, q, s = 128, 4096, 200000, 32
        rate = _load_rate(0.95, n, m, T, BMAX, LEN_LONG_PROMPT)
        spec = dict(k=10, dist="gaussian", rate=rate, load=0.95, lens=LEN_LONG_PROMPT, h0=1024, label="K10-gaussian")
        return n, m, q, s, [spec] * 256, ARRIVAL_GAMMA, 3.0
    if cid == 4:
        n, m, q, s = 64, 2048, 50000, 64
        rate = _load_rate(0.9, n, m, T, BMAX, LEN_DEFAULT)
        spec = dict(k=4, dist="enterprise", rate=rate, load=0.9, lens=LEN_DEFAULT, h0=512, label="K4-enterprise")
        return n, m, q, s, [spec] * 16384, ARRIVAL_POISSON, 1.0
    raise ValueError("workload id must be 0..4")


def _mean_lens(lens: dict) -> tuple[float, float]:
    ep = mean_clipped_lognormal(lens["prompt_mu"], lens["prompt_sigma"], lens["prompt_min"], lens["prompt_max"])
    eo = mean_clipped_lognormal(lens["output_mu"], lens["output_sigma"], lens["output_min"], lens["output_max"])
    return ep, eo


def num_replicas(cid: int) -> int:
    """Replica count of workload ``cid`` (no trace is generated)."""
    return len(_specs(cid)[4])


def predicted_work(cid: int, requests: int | None = None) -> np.ndarray:
    """Predicted simulation work of each replica of workload ``cid``,
    requests x instances x load (float64 [R]); no trace is generated."""
    n, _m, q, _s, specs, _kind, _cv = _specs(cid)
    qq = q if requests is None else int(requests)
    return np.array([float(qq) * n * sp["load"] for sp in specs], dtype=np.float64)


def partition(weights, parts: int) -> list[tuple[int, int]]:
    """Splits replicas 0..R-1 into ``parts`` contiguous ranges [lo, hi) whose
    summed weights are as even as cutting the prefix sums at multiples of
    total/parts makes them; every replica lands in exactly one range and every
    range is non-empty (R >= parts is required)."""
    w = np.asarray(weights, dtype=np.float64)
    r = int(w.shape[0])
    if parts < 1 or r < parts:
        raise ValueError("need 1 <= parts <= replicas (%d parts, %d replicas)" % (parts, r))
    if (w < 0).any():
        raise ValueError("weights must be non-negative")
    pre = np.concatenate([[0.0], np.cumsum(w)])
    total = pre[-1]
    cuts = [0]
    for k in range(1, parts):
        c = int(np.searchsorted(pre, total * k / parts, side="left"))
        # a cut may not leave a range empty, before or after it
        c = max(c, cuts[-1] + 1)
        c = min(c, r - (parts - k))
        cuts.append(c)
    cuts.append(r)
    return [(cuts[k], cuts[k + 1]) for k in range(parts)]


def config(cid: int, replicas=None, requests: int | None = None, nthreads: int | None = None,
           seed_block: int = 0) -> Workload:
    """Builds workload ``cid`` (0..4).  ``replicas`` selects a subset of replica
    indices (their seeds are those of the full workload, so a subset is a true
    sample of it); ``requests`` overrides the per-replica request count;
    ``seed_block`` > 0 draws an independent copy of the workload (same shapes,
    other seeds)."""
    T, BMAX = 16, 64
    n, m, q, s, specs, kind, cv = _specs(cid)
    idx = list(range(len(specs))) if replicas is None else [int(i) for i in replicas]
    if any(i < 0 or i >= len(specs) for i in idx):
        raise ValueError("replica index out of range for workload %d" % cid)
    qq = q if requests is None else int(requests)
    tables: dict[tuple, int] = {}
    tables_k, tables_h, rt, params, labels = [], [], [], [], []
    for i in idx:
        sp = specs[i]
        h = headroom_decay_table(sp["h0"], sp["k"])
        key = (sp["k"], tuple(h))
        if key not in tables:
            tables[key] = len(tables_k)
            tables_k.append(sp["k"])
            tables_h.append(h)
        rt.append(tables[key])
        seed = (0 if cid == 0 else mix_seed(cid, i)) if seed_block == 0 else mix_seed(cid, (seed_block << 24) + i)
        params.append(_params(seed, qq, sp["k"], tier_probs(sp["dist"], sp["k"]), sp["rate"], sp["lens"], kind, cv))
        labels.append(sp["label"])
    off, arrival, plen, olen, tier = generate(params, nthreads)
    return Workload(
        name="workload-%d" % cid, num_instances=n, blocks_per_instance=m, tokens_per_block=T, max_batch=BMAX,
        tables_k=tables_k, tables_h=tables_h, replica_table=np.asarray(rt, dtype=np.int32),
        migrate_blocks_per_iter=s, offsets=off, arrival_us=arrival, prompt_len=plen, output_len=olen,
        tier=tier, labels=labels,
    )


def custom(num_instances: int, blocks_per_instance: int, tables_k, tables_h, replica_table,
           traces, tokens_per_block: int = 16, max_batch: int = 64, **policy) -> Workload:
    """A workload from explicit per-replica traces: ``traces`` is a list of
    (arrival_us, prompt_len, output_len, tier) array tuples."""
    lens = [len(tr[0]) for tr in traces]
    off = np.zeros(len(traces) + 1, dtype=np.int64)
    np.cumsum(lens, out=off[1:])
    cat = lambda j, dt: (np.concatenate([np.asarray(tr[j], dtype=dt) for tr in traces])
                         if traces else np.zeros(0, dtype=dt))
    w = Workload(
        name="custom", num_instances=num_instances, blocks_per_instance=blocks_per_instance,
        tokens_per_block=tokens_per_block, max_batch=max_batch, tables_k=list(tables_k),
        tables_h=[list(h) for h in tables_h], replica_table=np.asarray(replica_table, dtype=np.int32),
        offsets=off, arrival_us=cat(0, np.uint32), prompt_len=cat(1, np.uint16),
        output_len=cat(2, np.uint16), tier=cat(3, np.uint8),
    )
    for k, v in policy.items():
        if not hasattr(w, k):
            raise TypeError("unknown policy field %r" % k)
        setattr(w, k, v)
    return w
