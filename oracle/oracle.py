"""Python access to the reference CPU simulator in ``sim_oracle.cpp``.

TEST INFRASTRUCTURE ONLY: the test suite, the package smoke check and the
benchmark's CPU-baseline leg are the only callers.  The product path never
imports this module.

``run_workload`` takes any object with the attributes of
``paper_2608_16336_gb300.workloads.Workload`` (duck-typed; nothing from the
package is imported here) and returns per-request results, per-replica
statistics and migration logs as numpy arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_DIR = os.path.join(HERE, "_lib")
SRC = os.path.join(HERE, "sim_oracle.cpp")
SO = os.path.join(LIB_DIR, "liboracle.so")

MAXK = 16
NONE32 = 0xFFFFFFFF
STATUS_DONE, STATUS_INCOMPLETE = 0, 1
EV_QUEUED, EV_START, EV_COMMIT, EV_ABORT, EV_SCALE_OUT, EV_SCALE_IN = 0, 1, 2, 3, 4, 5


class OracleConfig(ctypes.Structure):
    _fields_ = [
        ("num_instances", ctypes.c_int32),
        ("blocks_per_instance", ctypes.c_int32),
        ("tokens_per_block", ctypes.c_int32),
        ("max_batch", ctypes.c_int32),
        ("num_tiers", ctypes.c_int32),
        ("headroom", ctypes.c_int32 * MAXK),
        ("iter_base_us", ctypes.c_int64),
        ("iter_us_per_prefill_token", ctypes.c_int64),
        ("iter_us_per_decode_seq", ctypes.c_int64),
        ("migrate_blocks_per_iter", ctypes.c_int32),
        ("enable_migration", ctypes.c_int32),
        ("migrate_interval_us", ctypes.c_int64),
        ("theta_num", ctypes.c_int32),
        ("theta_den", ctypes.c_int32),
        ("check_invariants", ctypes.c_int32),
        ("autoscale", ctypes.c_int32),
        ("scale_out_num", ctypes.c_int32),
        ("scale_in_num", ctypes.c_int32),
        ("scale_den", ctypes.c_int32),
        ("pad_", ctypes.c_int32),
        ("drain_start_us", ctypes.c_void_p),
        ("n_headroom_changes", ctypes.c_int32),
        ("pad2_", ctypes.c_int32),
        ("headroom_change_step", ctypes.c_void_p),
        ("headroom_change_table", ctypes.c_void_p),
    ]


class OracleStats(ctypes.Structure):
    _fields_ = [
        ("steps", ctypes.c_int64),
        ("iterations", ctypes.c_int64),
        ("member_iterations", ctypes.c_int64),
        ("events", ctypes.c_int64),
        ("migrations", ctypes.c_int64),
        ("preemptions", ctypes.c_int64),
        ("migration_starts", ctypes.c_int64),
        ("migration_aborts", ctypes.c_int64),
        ("log_events", ctypes.c_int64),
        ("finished", ctypes.c_int64),
        ("last_time", ctypes.c_uint32),
        ("status", ctypes.c_int32),
        ("scale_out_signals", ctypes.c_int64),
        ("scale_in_signals", ctypes.c_int64),
    ]


class OracleIO(ctypes.Structure):
    _fields_ = [
        ("nreq", ctypes.c_int64),
        ("arrival_us", ctypes.c_void_p),
        ("prompt_len", ctypes.c_void_p),
        ("output_len", ctypes.c_void_p),
        ("tier", ctypes.c_void_p),
        ("dispatch_instance", ctypes.c_void_p),
        ("final_instance", ctypes.c_void_p),
        ("first_token_us", ctypes.c_void_p),
        ("finish_us", ctypes.c_void_p),
        ("n_migrations", ctypes.c_void_p),
        ("n_preemptions", ctypes.c_void_p),
        ("log_capacity", ctypes.c_int64),
        ("ev_time", ctypes.c_void_p),
        ("ev_req", ctypes.c_void_p),
        ("ev_src", ctypes.c_void_p),
        ("ev_dst", ctypes.c_void_p),
        ("ev_blocks", ctypes.c_void_p),
        ("ev_kind", ctypes.c_void_p),
    ]


def build(force: bool = False, so_path: str = SO, defines: list[str] | None = None, src: str = SRC,
          opt: str = "-O3") -> str:
    """Compiles the oracle with g++ (no architecture-specific flags)."""
    if force or defines or not os.path.exists(so_path) or os.path.getmtime(so_path) < os.path.getmtime(src):
        os.makedirs(os.path.dirname(so_path), exist_ok=True)
        tmp = so_path + ".tmp%d" % os.getpid()
        cmd = ["g++", opt, "-std=c++17", "-fPIC", "-shared", "-pthread", src, "-o", tmp]
        cmd += ["-D" + d for d in (defines or [])]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError("oracle build failed:\n" + res.stderr)
        os.replace(tmp, so_path)
    return so_path


_LIBS: dict[str, ctypes.CDLL] = {}


def lib(so_path: str | None = None) -> ctypes.CDLL:
    path = so_path or build()
    if path not in _LIBS:
        L = ctypes.CDLL(path)
        L.oracle_run_replica.restype = ctypes.c_int
        L.oracle_run_replica.argtypes = [ctypes.POINTER(OracleConfig), ctypes.POINTER(OracleIO), ctypes.c_int64,
                                         ctypes.POINTER(OracleStats)]
        L.oracle_run_many.restype = ctypes.c_int
        L.oracle_run_many.argtypes = [ctypes.c_int32, ctypes.POINTER(OracleConfig), ctypes.POINTER(OracleIO),
                                      ctypes.c_int64, ctypes.POINTER(OracleStats), ctypes.c_int32]
        L.oracle_freeness.restype = ctypes.c_int
        L.oracle_freeness.argtypes = [ctypes.POINTER(OracleConfig), ctypes.c_int32, ctypes.c_void_p, ctypes.c_int32,
                                      ctypes.c_void_p, ctypes.c_int32, ctypes.POINTER(ctypes.c_int64),
                                      ctypes.POINTER(ctypes.c_int64)]
        _LIBS[path] = L
    return _LIBS[path]


def make_config(num_instances, blocks_per_instance, headroom, *, tokens_per_block=16, max_batch=64,
                iter_base_us=4000, iter_us_per_prefill_token=20, iter_us_per_decode_seq=30,
                migrate_blocks_per_iter=64, enable_migration=1, migrate_interval_us=50_000,
                theta_num=3, theta_den=10, check_invariants=0, autoscale=0, scale_out_num=-1, scale_in_num=3,
                scale_den=2, drain_start_us=None, headroom_schedule=None) -> OracleConfig:
    """A replica's configuration; ``drain_start_us`` ([num_instances] times,
    NONE32 = never) is kept alive on the returned object as ``_drain``.
    ``headroom_schedule``: [(step, table)] — before the step of that index
    (0-based) is processed, the headroom table becomes ``table``; its arrays
    are kept alive as ``_sched``."""
    c = OracleConfig()
    c.num_instances = num_instances
    c.blocks_per_instance = blocks_per_instance
    c.tokens_per_block = tokens_per_block
    c.max_batch = max_batch
    c.num_tiers = len(headroom)
    for k, h in enumerate(headroom):
        c.headroom[k] = int(h)
    c.iter_base_us = iter_base_us
    c.iter_us_per_prefill_token = iter_us_per_prefill_token
    c.iter_us_per_decode_seq = iter_us_per_decode_seq
    c.migrate_blocks_per_iter = migrate_blocks_per_iter
    c.enable_migration = enable_migration
    c.migrate_interval_us = migrate_interval_us
    c.theta_num = theta_num
    c.theta_den = theta_den
    c.check_invariants = check_invariants
    c.autoscale = autoscale
    c.scale_out_num = scale_out_num
    c.scale_in_num = scale_in_num
    c.scale_den = scale_den
    c._drain = None
    if drain_start_us is not None:
        c._drain = np.ascontiguousarray(drain_start_us, np.uint32)
        if c._drain.shape != (num_instances,):
            raise ValueError("drain_start_us needs one time per instance")
        c.drain_start_us = c._drain.ctypes.data
    c._sched = None
    if headroom_schedule:
        steps = np.ascontiguousarray([int(st) for st, _ in headroom_schedule], np.int64)
        tables = np.zeros((len(headroom_schedule), MAXK), np.int32)
        for j, (_, tab) in enumerate(headroom_schedule):
            if len(tab) != len(headroom):
                raise ValueError("every scheduled table needs one entry per tier")
            tables[j, : len(tab)] = tab
        c._sched = (steps, tables)
        c.n_headroom_changes = len(headroom_schedule)
        c.headroom_change_step = steps.ctypes.data
        c.headroom_change_table = tables.ctypes.data
    return c


def config_for(w, r: int, check_invariants: int = 0, headroom_schedule=None) -> OracleConfig:
    return make_config(
        w.num_instances, w.blocks_per_instance, w.tables_h[int(w.replica_table[r])],
        tokens_per_block=w.tokens_per_block, max_batch=w.max_batch, iter_base_us=w.iter_base_us,
        iter_us_per_prefill_token=w.iter_us_per_prefill_token, iter_us_per_decode_seq=w.iter_us_per_decode_seq,
        migrate_blocks_per_iter=w.migrate_blocks_per_iter, enable_migration=w.enable_migration,
        migrate_interval_us=w.migrate_interval_us, theta_num=w.theta_num, theta_den=w.theta_den,
        check_invariants=check_invariants, autoscale=getattr(w, "autoscale", 0),
        scale_out_num=getattr(w, "scale_out_num", -1), scale_in_num=getattr(w, "scale_in_num", 3),
        scale_den=getattr(w, "scale_den", 2),
        drain_start_us=None if getattr(w, "drain_start_us", None) is None else w.drain_start_us[r],
        headroom_schedule=headroom_schedule)


class ReplicaResult:
    """Outputs of one simulated replica."""

    def __init__(self, n: int, cap: int):
        self.dispatch_instance = np.empty(n, np.int32)
        self.final_instance = np.empty(n, np.int32)
        self.first_token_us = np.empty(n, np.uint32)
        self.finish_us = np.empty(n, np.uint32)
        self.n_migrations = np.empty(n, np.int32)
        self.n_preemptions = np.empty(n, np.int32)
        self.ev_time = np.empty(cap, np.uint32)
        self.ev_req = np.empty(cap, np.uint32)
        self.ev_src = np.empty(cap, np.int32)
        self.ev_dst = np.empty(cap, np.int32)
        self.ev_blocks = np.empty(cap, np.int32)
        self.ev_kind = np.empty(cap, np.int32)
        self.stats: dict = {}

    def events(self) -> np.ndarray:
        """Migration log as an (n, 6) int64 array: time, request, src, dst, blocks, kind."""
        n = min(int(self.stats["log_events"]), self.ev_time.shape[0])
        return np.stack([self.ev_time[:n], self.ev_req[:n], self.ev_src[:n], self.ev_dst[:n],
                         self.ev_blocks[:n], self.ev_kind[:n]], axis=1).astype(np.int64)


def _io_for(arrival, plen, olen, tier, res: ReplicaResult) -> tuple[OracleIO, list]:
    keep = [np.ascontiguousarray(arrival, np.uint32), np.ascontiguousarray(plen, np.uint16),
            np.ascontiguousarray(olen, np.uint16), np.ascontiguousarray(tier, np.uint8)]
    io = OracleIO()
    io.nreq = keep[0].shape[0]
    io.arrival_us, io.prompt_len, io.output_len, io.tier = [k.ctypes.data for k in keep]
    for f in ("dispatch_instance", "final_instance", "first_token_us", "finish_us", "n_migrations", "n_preemptions",
              "ev_time", "ev_req", "ev_src", "ev_dst", "ev_blocks", "ev_kind"):
        setattr(io, f, getattr(res, f).ctypes.data)
    io.log_capacity = res.ev_time.shape[0]
    return io, keep


def _stats_dict(s: OracleStats) -> dict:
    return {name: getattr(s, name) for name, _ in OracleStats._fields_}


def run_trace(cfg: OracleConfig, arrival, plen, olen, tier, *, max_steps: int = 1 << 62,
              log_capacity: int = 1 << 16, so_path: str | None = None) -> ReplicaResult:
    res = ReplicaResult(len(arrival), log_capacity)
    io, keep = _io_for(arrival, plen, olen, tier, res)
    st = OracleStats()
    lib(so_path).oracle_run_replica(ctypes.byref(cfg), ctypes.byref(io), max_steps, ctypes.byref(st))
    res.stats = _stats_dict(st)
    return res


def run_workload(w, replicas=None, *, nthreads: int = 1, max_steps: int = 1 << 62, log_capacity: int = 1 << 16,
                 check_invariants: int = 0, so_path: str | None = None,
                 headroom_schedules: dict | None = None) -> dict[int, ReplicaResult]:
    """Simulates the chosen replicas of workload ``w``; returns {replica: result}.
    ``headroom_schedules``: {replica: [(step, table)]} (see make_config)."""
    reps = list(range(w.num_replicas)) if replicas is None else [int(r) for r in replicas]
    n = len(reps)
    cfgs = (OracleConfig * max(n, 1))()
    ios = (OracleIO * max(n, 1))()
    stats = (OracleStats * max(n, 1))()
    results, keep = {}, []
    for j, r in enumerate(reps):
        sl = slice(int(w.offsets[r]), int(w.offsets[r + 1]))
        res = ReplicaResult(sl.stop - sl.start, log_capacity)
        io, k = _io_for(w.arrival_us[sl], w.prompt_len[sl], w.output_len[sl], w.tier[sl], res)
        keep.append(k)
        cfg = config_for(w, r, check_invariants, (headroom_schedules or {}).get(r))
        keep.append(cfg._drain)
        keep.append(cfg._sched)
        cfgs[j] = cfg
        ios[j] = io
        results[r] = res
    lib(so_path).oracle_run_many(n, cfgs, ios, max_steps, stats, nthreads)
    for j, r in enumerate(reps):
        results[r].stats = _stats_dict(stats[j])
    return results


def freeness(cfg: OracleConfig, running_blocks, hol_demand: int, cnt, reserved_in: int = 0) -> tuple[int, int]:
    rb = np.ascontiguousarray(running_blocks, np.int32)
    cn = np.zeros(MAXK, np.int32)
    cn[: len(cnt)] = cnt
    num, den = ctypes.c_int64(), ctypes.c_int64()
    rc = lib().oracle_freeness(ctypes.byref(cfg), rb.shape[0], rb.ctypes.data, hol_demand, cn.ctypes.data,
                               reserved_in, ctypes.byref(num), ctypes.byref(den))
    if rc != 0:
        raise ValueError("oracle_freeness rejected its arguments")
    return num.value, den.value


def timed_sample(w, replicas, nthreads: int) -> dict:
    """Times the oracle over ``replicas`` of ``w`` on ``nthreads`` host threads."""
    t0 = time.perf_counter()
    res = run_workload(w, replicas, nthreads=nthreads, log_capacity=0)
    dt = time.perf_counter() - t0
    steps = sum(int(r.stats["steps"]) for r in res.values())
    events = sum(int(r.stats["events"]) for r in res.values())
    ok = all(r.stats["status"] == STATUS_DONE for r in res.values())
    return {"seconds": dt, "steps": steps, "events": events, "replicas": len(res), "all_done": ok}
