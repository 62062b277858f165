"""Brute-force checker for tiny clusters (TEST INFRASTRUCTURE ONLY).

A second, deliberately naive statement of the same simulation as
``sim_oracle.cpp``, used to pin the oracle on tiny inputs: pure Python, exact
``fractions.Fraction`` freeness, virtual usage summed request by request
(Sec. 3.2, Eq. 2) with headroom charged once per present tier (Sec. 3.3,
Eq. 4), explicit batch-membership sets, and selections made with ``min``/
``max`` over explicit keys.  Only for a handful of instances and a few dozen
requests.

Draining (Sec. 3.5, the last case of Eq. 2) is the literal sentinel: the
freeness of a draining instance is minus infinity, so comparisons do the
rest; only the dispatch fallback when every instance drains (Sec. 3.4) looks
at ordinary freeness.  The auto-scaling signal (Sec. 3.6) averages the
normal-priority freeness, a ``Fraction`` without the headroom term, over the
instances that are not draining.

``binary=True`` replaces the per-tier table by the original two-class
Llumnix rule quoted in Sec. 3.3: every high-priority request (tier 0) present
on an instance carries headroom h / numHighPriorityRequests and every other
request none.
"""
from __future__ import annotations

from fractions import Fraction

NONE32 = 0xFFFFFFFF
QUEUED, START, COMMIT, ABORT, SCALE_OUT, SCALE_IN = 0, 1, 2, 3, 4, 5
MINUS_INF = float("-inf")


def _ceil_div(a: int, b: int) -> int:
    return -(-a // b)


class TinySim:
    def __init__(self, n, m, headroom, trace, *, t_blk=16, bmax=64, base=4000, a=20, b=30, s_blocks=64,
                 migration=True, interval=50_000, theta=Fraction(3, 10), binary=False, binary_h=0,
                 drain=None, autoscale=False, scale_out=Fraction(-1, 2), scale_in=Fraction(3, 2),
                 headroom_schedule=None):
        self.N, self.M, self.T, self.Bmax = n, m, t_blk, bmax
        self.H = list(headroom)
        self.K = len(self.H)
        # adaptive headroom: [(step, table)], table in force from the step of that index on
        self.schedule = sorted(headroom_schedule or [], key=lambda e: e[0])
        self.base, self.a, self.b, self.S = base, a, b, s_blocks
        self.migration, self.interval, self.theta = migration, interval, theta
        self.binary, self.binary_h = binary, binary_h
        self.drain = list(drain) if drain is not None else [NONE32] * n
        self.autoscale, self.scale_out, self.scale_in = autoscale, scale_out, scale_in
        self.signals = {"out": 0, "in": 0}
        self.trace = [tuple(int(x) for x in rec) for rec in trace]   # (arrival, P, O, tier)
        q = len(self.trace)
        self.g = [0] * q
        self.blocks = [0] * q
        self.loc = [None] * q            # ("wait", i) / ("run", i) / None
        self.out = {"dispatch": [-1] * q, "final": [-1] * q, "first": [NONE32] * q, "finish": [NONE32] * q,
                    "mig": [0] * q, "pre": [0] * q}
        self.queues = [[[] for _ in range(self.K)] for _ in range(n)]
        self.running = [[] for _ in range(n)]
        self.batch = [set() for _ in range(n)]
        self.busy_until = [None] * n
        self.free = [m] * n
        self.reserved = [0] * n
        self.mig = {}                    # source -> dict(req, dst, copied)
        self.log = []
        self.steps = 0
        self.now = 0

    # ---------------------------------------------------------- freeness --
    def demand(self, r):
        P = self.trace[r][1]
        return _ceil_div(P + self.g[r], self.T)

    def hol(self, i):
        for k in range(self.K):
            if self.queues[i][k]:
                return self.queues[i][k][0]
        return None

    def present(self, i):
        reqs = list(self.running[i]) + [r for k in range(self.K) for r in self.queues[i][k]]
        return reqs

    def virtual_usage(self, i):
        h = self.hol(i)
        total = Fraction(0)
        reqs = self.present(i)
        for r in reqs:
            if r in self.running[i]:
                total += self.blocks[r]
            elif r == h:
                total += self.demand(r)
        if self.binary:
            high = [r for r in reqs if self.trace[r][3] == 0]
            for _r in high:
                total += Fraction(self.binary_h, len(high))
        else:
            for k in sorted({self.trace[r][3] for r in reqs}):
                total += self.H[k]
        total += self.reserved[i]
        return total

    def draining(self, i):
        return self.now >= self.drain[i]

    def F_plain(self, i):
        return (self.M - self.virtual_usage(i)) / max(len(self.running[i]), 1)

    def F(self, i):
        """F_full with the drain sentinel: infinite usage, minus infinite freeness."""
        return MINUS_INF if self.draining(i) else self.F_plain(i)

    def F_normal(self, i):
        h = self.hol(i)
        used = sum(self.blocks[r] for r in self.running[i]) + (self.demand(h) if h is not None else 0)
        used += self.reserved[i]
        return Fraction(self.M - used, max(len(self.running[i]), 1))

    def dst_of(self, i):
        for s, mg in self.mig.items():
            if mg["dst"] == i:
                return s
        return None

    # ------------------------------------------------------------ events --
    def _abort(self, s):
        mg = self.mig.pop(s)
        d = mg["dst"]
        self.free[d] += mg["copied"]
        self.reserved[d] -= mg["copied"]
        self.log.append((self.now, mg["req"], s, d, mg["copied"], ABORT))

    def _leave_running(self, i, r):
        self.running[i].remove(r)
        self.batch[i].discard(r)
        if i in self.mig and self.mig[i]["req"] == r:
            self._abort(i)

    def _complete(self, i):
        self.busy_until[i] = None
        members = [r for r in self.running[i] if r in self.batch[i]]
        self.batch[i] = set()
        for r in members:
            self.g[r] += 1
            if self.out["first"][r] == NONE32:
                self.out["first"][r] = self.now
            if self.g[r] == self.trace[r][2]:
                self.out["finish"][r] = self.now
                self.out["final"][r] = i
                self.free[i] += self.blocks[r]
                self.blocks[r] = 0
                self.loc[r] = None
                self._leave_running(i, r)
        if i in self.mig:
            mg = self.mig[i]
            r, d = mg["req"], mg["dst"]
            c = min(self.S, self.blocks[r] - mg["copied"])
            if self.free[d] < c:
                self._abort(i)
                return
            self.free[d] -= c
            self.reserved[d] += c
            mg["copied"] += c
            if mg["copied"] == self.blocks[r] and len(self.running[d]) < self.Bmax:
                del self.mig[i]
                self.free[i] += self.blocks[r]
                self.running[i].remove(r)
                self.reserved[d] -= mg["copied"]
                self.running[d].append(r)
                self.loc[r] = ("run", d)
                self.out["mig"][r] += 1
                self.log.append((self.now, r, i, d, self.blocks[r], COMMIT))

    def _dispatch(self, arrivals):
        for r in sorted(arrivals, key=lambda x: (self.trace[x][3], x)):
            best = max(range(self.N), key=lambda i: (self.F(i), -i))
            if self.F(best) == MINUS_INF:   # all draining: the least loaded of them
                best = max(range(self.N), key=lambda i: (self.F_plain(i), -i))
            self.queues[best][self.trace[r][3]].append(r)
            self.loc[r] = ("wait", best)
            self.out["dispatch"][r] = best

    def _tick(self):
        busy = set(self.mig) | {mg["dst"] for mg in self.mig.values()}
        pool = [i for i in range(self.N) if i not in busy]
        while len(pool) >= 2:
            fs = {i: self.F(i) for i in pool}
            s = min(pool, key=lambda i: (fs[i], i))
            d = max((i for i in pool if i != s), key=lambda i: (fs[i], -i))
            if fs[d] == MINUS_INF or fs[d] - fs[s] < self.theta:
                break
            moved = False
            tiers = [k for k in range(self.K) if self.queues[s][k]]
            if tiers:
                k = max(tiers)
                r = self.queues[s][k].pop()
                self.queues[d][k].append(r)
                self.loc[r] = ("wait", d)
                self.out["mig"][r] += 1
                self.log.append((self.now, r, s, d, 0, QUEUED))
                moved = True
            elif self.running[s]:
                r = max(self.running[s], key=lambda x: (self.trace[x][3], -self.blocks[x], x))
                if self.free[d] >= self.blocks[r]:
                    self.mig[s] = {"req": r, "dst": d, "copied": 0}
                    self.log.append((self.now, r, s, d, self.blocks[r], START))
                    moved = True
            pool.remove(s)
            if moved:
                pool.remove(d)

    def _autoscale(self):
        live = [i for i in range(self.N) if not self.draining(i)]
        if not live:
            return
        mean = sum(self.F_normal(i) for i in live) / len(live)
        if mean < self.scale_out:
            self.signals["out"] += 1
            self.log.append((self.now, NONE32, 255, 255, 0, SCALE_OUT))
        elif mean > self.scale_in:
            self.signals["in"] += 1
            self.log.append((self.now, NONE32, 255, 255, 0, SCALE_IN))

    def _form(self, i):
        if self.busy_until[i] is not None:
            return
        if not self.running[i] and self.hol(i) is None:
            return
        j = 0
        while j < len(self.running[i]):
            r = self.running[i][j]
            gone = False
            while self.demand(r) > self.blocks[r]:
                if self.free[i] > 0:
                    self.free[i] -= 1
                    self.blocks[r] += 1
                    continue
                v = max(self.running[i], key=lambda x: (self.trace[x][3], x))
                vj = self.running[i].index(v)
                self.free[i] += self.blocks[v]
                self.blocks[v] = 0
                self._leave_running(i, v)
                self.queues[i][self.trace[v][3]].insert(0, v)
                self.loc[v] = ("wait", i)
                self.out["pre"][v] += 1
                if v == r:
                    gone = True
                    break
                if vj < j:
                    j -= 1
            if not gone:
                j += 1
        decode = len(self.running[i])
        prefill = 0
        while len(self.running[i]) < self.Bmax:
            h = self.hol(i)
            if h is None or self.demand(h) > self.free[i]:
                break
            self.queues[i][self.trace[h][3]].pop(0)
            self.blocks[h] = self.demand(h)
            self.free[i] -= self.blocks[h]
            self.running[i].append(h)
            self.loc[h] = ("run", i)
            prefill += self.trace[h][1] + self.g[h]
        if self.running[i]:
            self.busy_until[i] = self.now + self.base + self.a * prefill + self.b * decode
            self.batch[i] = set(self.running[i])

    def run(self, max_steps=10 ** 9):
        q = len(self.trace)
        nxt = 0
        tick = self.interval
        while sum(1 for x in self.out["finish"] if x != NONE32) < q and self.steps < max_steps:
            for step, table in self.schedule:
                if step == self.steps:
                    self.H = list(table)
            cands = [bu for bu in self.busy_until if bu is not None]
            if nxt < q:
                cands.append(self.trace[nxt][0])
            if not cands:
                raise RuntimeError("deadlock")
            t = min(cands)
            do_tick = (self.migration or self.autoscale) and tick <= t
            if do_tick:
                t = tick
            self.now = t
            self.steps += 1
            for i in range(self.N):
                if self.busy_until[i] == t:
                    self._complete(i)
            arrivals = []
            while nxt < q and self.trace[nxt][0] == t:
                arrivals.append(nxt)
                nxt += 1
            self._dispatch(arrivals)
            if do_tick:
                tick += self.interval
                if self.autoscale:
                    self._autoscale()
                if self.migration:
                    self._tick()
            for i in range(self.N):
                self._form(i)
        return self
