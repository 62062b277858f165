"""ctypes binding of libmtsim (include/mtsim.h).

The module-level functions carry the C names and only marshal arguments;
every step of the simulation runs in the library's CUDA kernels.  There is no
CPU fallback: if ``_lib/libmtsim.so`` is missing, ``lib()`` raises.

``Simulator`` is a convenience wrapper that feeds a
``workloads.Workload`` through the C ABI, using PyTorch for device memory
(trace tensors and, optionally, the caching allocator) and for the stream.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import _build

SIM_OK = 0
SIM_ERR_ARG, SIM_ERR_TRACE, SIM_ERR_STATE, SIM_ERR_OOM = -1, -2, -3, -4
SIM_ERR_OVERFLOW, SIM_ERR_CUDA, SIM_ERR_INTERNAL, SIM_ERR_DEADLOCK, SIM_ERR_UNFINISHED = -5, -7, -8, -10, -11
SIM_REPLICA_DONE, SIM_REPLICA_RUNNING = 0, 1
SIM_EV_QUEUED, SIM_EV_START, SIM_EV_COMMIT, SIM_EV_ABORT, SIM_EV_SCALE_OUT, SIM_EV_SCALE_IN = 0, 1, 2, 3, 4, 5
SIM_NONE32, SIM_NONE16 = 0xFFFFFFFF, 0xFFFF
SIM_MAX_TIERS = 16

RESULT_DTYPE = np.dtype([("dispatch_instance", "<u2"), ("final_instance", "<u2"), ("first_token_us", "<u4"),
                         ("finish_us", "<u4"), ("n_preemptions", "<u2"), ("n_migrations", "<u2")])
STATS_DTYPE = np.dtype([("steps", "<u8"), ("iterations", "<u8"), ("member_iterations", "<u8"), ("events", "<u8"),
                        ("migrations", "<u4"), ("preemptions", "<u4"), ("migration_starts", "<u4"),
                        ("migration_aborts", "<u4"), ("log_events", "<u4"), ("finished", "<u4"),
                        ("last_time_us", "<u4"), ("status", "<i4"), ("scale_out_signals", "<u4"),
                        ("scale_in_signals", "<u4")])
EVENT_DTYPE = np.dtype([("time_us", "<u4"), ("request", "<u4"), ("blocks", "<u2"), ("src", "u1"), ("dst", "u1"),
                        ("kind", "u1"), ("pad", "u1", (3,))])
SIM_HIST_BUCKETS = 240
SIM_LAT_TTFT, SIM_LAT_TBT, SIM_LAT_E2E = 0, 1, 2
LATENCY_DTYPE = np.dtype([("count", "<u4"), ("max_us", "<u4"), ("sum_us", "<u8"), ("p50_us", "<u4"),
                          ("p90_us", "<u4"), ("p99_us", "<u4"), ("pad", "<u4"), ("hist", "<u4", (SIM_HIST_BUCKETS,))])
assert RESULT_DTYPE.itemsize == 16 and STATS_DTYPE.itemsize == 72 and EVENT_DTYPE.itemsize == 16
assert LATENCY_DTYPE.itemsize == 992


class sim_cluster_t(ctypes.Structure):
    _fields_ = [("num_replicas", ctypes.c_int32), ("num_instances", ctypes.c_int32),
                ("blocks_per_instance", ctypes.c_int32), ("tokens_per_block", ctypes.c_int32),
                ("max_batch", ctypes.c_int32)]


class sim_tier_table_t(ctypes.Structure):
    _fields_ = [("num_tables", ctypes.c_int32), ("max_tiers", ctypes.c_int32),
                ("num_tiers", ctypes.c_void_p), ("headroom_blocks", ctypes.c_void_p),
                ("replica_table", ctypes.c_void_p)]


class sim_policy_t(ctypes.Structure):
    _fields_ = [("policy", ctypes.c_int32), ("enable_migration", ctypes.c_int32),
                ("iter_base_us", ctypes.c_int64), ("iter_us_per_prefill_token", ctypes.c_int64),
                ("iter_us_per_decode_seq", ctypes.c_int64), ("migrate_blocks_per_iter", ctypes.c_int32),
                ("theta_num", ctypes.c_int32), ("theta_den", ctypes.c_int32),
                ("event_log_capacity", ctypes.c_int32), ("migrate_interval_us", ctypes.c_int64),
                ("autoscale", ctypes.c_int32), ("scale_out_num", ctypes.c_int32), ("scale_in_num", ctypes.c_int32),
                ("scale_den", ctypes.c_int32)]


class sim_launch_info_t(ctypes.Structure):
    _fields_ = [("grid_blocks", ctypes.c_int32), ("block_threads", ctypes.c_int32),
                ("blocks_per_sm", ctypes.c_int32), ("instances_per_lane", ctypes.c_int32),
                ("slots_in_shared", ctypes.c_int32), ("extended", ctypes.c_int32),
                ("shared_bytes", ctypes.c_int64)]


ALLOC_FN = ctypes.CFUNCTYPE(ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p)
FREE_FN = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p)


class sim_allocator_t(ctypes.Structure):
    _fields_ = [("ctx", ctypes.c_void_p), ("alloc", ALLOC_FN), ("free", FREE_FN)]


EXPORTS = ["sim_create", "sim_load_trace", "sim_reset", "sim_run", "sim_metrics", "sim_destroy",
           "sim_last_error", "sim_strerror", "sim_device_bytes", "sim_run_static", "sim_set_drain",
           "sim_latency_stats", "sim_launch_info", "sim_set_order", "sim_set_headroom"]
SIM_STATIC_SCRATCH_BYTES = 32 << 20

_LIB = None


def lib() -> ctypes.CDLL:
    """Loads libmtsim.so; raises if it has not been built."""
    global _LIB
    if _LIB is None:
        path = _build.MTSIM_SO
        if not os.path.exists(path):
            raise RuntimeError("libmtsim.so is missing (%s); build it with __graft_entry__.build() "
                               "or paper_2608_16336_gb300._build.build_mtsim()" % path)
        L = ctypes.CDLL(path)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        L.sim_create.argtypes = [ctypes.POINTER(sim_cluster_t), ctypes.POINTER(sim_tier_table_t),
                                 ctypes.POINTER(sim_policy_t), vp, ctypes.POINTER(sim_allocator_t),
                                 ctypes.POINTER(vp)]
        L.sim_create.restype = ctypes.c_int
        L.sim_load_trace.argtypes = [vp, vp, vp, vp, vp, vp, ctypes.c_int]
        L.sim_load_trace.restype = ctypes.c_int
        L.sim_reset.argtypes = [vp]
        L.sim_reset.restype = ctypes.c_int
        L.sim_set_drain.argtypes = [vp, vp, ctypes.c_int]
        L.sim_set_drain.restype = ctypes.c_int
        L.sim_latency_stats.argtypes = [vp, vp, ctypes.c_int]
        L.sim_latency_stats.restype = ctypes.c_int
        L.sim_run.argtypes = [vp, i64, ctypes.POINTER(i64)]
        L.sim_run.restype = ctypes.c_int
        L.sim_metrics.argtypes = [vp, vp, vp, vp, ctypes.c_int]
        L.sim_metrics.restype = ctypes.c_int
        L.sim_destroy.argtypes = [vp]
        L.sim_destroy.restype = None
        L.sim_last_error.argtypes = [vp]
        L.sim_last_error.restype = ctypes.c_char_p
        L.sim_strerror.argtypes = [ctypes.c_int]
        L.sim_strerror.restype = ctypes.c_char_p
        L.sim_device_bytes.argtypes = [vp]
        L.sim_device_bytes.restype = ctypes.c_size_t
        L.sim_set_headroom.argtypes = [vp, vp]
        L.sim_set_headroom.restype = ctypes.c_int
        L.sim_set_order.argtypes = [vp, vp]
        L.sim_set_order.restype = ctypes.c_int
        L.sim_launch_info.argtypes = [vp, ctypes.POINTER(sim_launch_info_t)]
        L.sim_launch_info.restype = ctypes.c_int
        L.sim_run_static.argtypes = [ctypes.POINTER(sim_cluster_t), ctypes.POINTER(sim_tier_table_t),
                                     ctypes.POINTER(sim_policy_t), vp, vp, vp, vp, vp, vp, vp, vp, vp]
        L.sim_run_static.restype = ctypes.c_int
        _LIB = L
    return _LIB


class SimError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__("%s (%d): %s" % (sim_strerror(code), code, msg))
        self.code = code


# ------------------------------------------------- C-named thin wrappers --
def sim_strerror(code: int) -> str:
    return lib().sim_strerror(code).decode()


def sim_last_error(handle) -> str:
    return (lib().sim_last_error(handle) or b"").decode()


def _check(code: int, handle) -> int:
    if code != SIM_OK:
        raise SimError(code, sim_last_error(handle))
    return code


def sim_create(cluster: sim_cluster_t, tiers: sim_tier_table_t, policy: sim_policy_t, cuda_stream: int = 0,
               allocator: sim_allocator_t | None = None):
    out = ctypes.c_void_p()
    rc = lib().sim_create(ctypes.byref(cluster), ctypes.byref(tiers), ctypes.byref(policy),
                          ctypes.c_void_p(cuda_stream or None), ctypes.byref(allocator) if allocator else None,
                          ctypes.byref(out))
    _check(rc, None)
    return out


def sim_load_trace(handle, replica_offsets_ptr: int, arrival_ptr: int, prompt_ptr: int, output_ptr: int,
                   tier_ptr: int, on_device: int) -> int:
    return _check(lib().sim_load_trace(handle, replica_offsets_ptr, arrival_ptr, prompt_ptr, output_ptr, tier_ptr,
                                       on_device), handle)


def sim_reset(handle) -> int:
    return _check(lib().sim_reset(handle), handle)


def sim_set_drain(handle, drain_ptr, on_device: int) -> int:
    return _check(lib().sim_set_drain(handle, drain_ptr, on_device), handle)


def sim_latency_stats(handle, out_ptr, on_device: int) -> int:
    return _check(lib().sim_latency_stats(handle, out_ptr, on_device), handle)


def sim_run(handle, max_steps_per_replica: int, want_unfinished: bool = True):
    n = ctypes.c_int64(-1)
    _check(lib().sim_run(handle, max_steps_per_replica, ctypes.byref(n) if want_unfinished else None), handle)
    return int(n.value) if want_unfinished else None


def sim_metrics(handle, per_request_ptr, per_replica_ptr, events_ptr, on_device: int) -> int:
    return _check(lib().sim_metrics(handle, per_request_ptr, per_replica_ptr, events_ptr, on_device), handle)


def sim_destroy(handle) -> None:
    lib().sim_destroy(handle)


def sim_device_bytes(handle) -> int:
    return int(lib().sim_device_bytes(handle))


def sim_set_headroom(handle, headroom_ptr) -> int:
    return _check(lib().sim_set_headroom(handle, headroom_ptr), handle)


def sim_set_order(handle, order_ptr) -> int:
    return _check(lib().sim_set_order(handle, order_ptr), handle)


def sim_launch_info(handle) -> dict:
    """The launch configuration sim_run would use now, as a dict."""
    out = sim_launch_info_t()
    _check(lib().sim_launch_info(handle, ctypes.byref(out)), handle)
    return {name: int(getattr(out, name)) for name, _ in sim_launch_info_t._fields_}


def sim_run_static(cluster: sim_cluster_t, tiers: sim_tier_table_t, policy: sim_policy_t, replica_offsets_ptr: int,
                   arrival_ptr: int, prompt_ptr: int, output_ptr: int, tier_ptr: int, per_request_ptr: int,
                   per_replica_ptr: int, events_ptr, cuda_stream: int = 0) -> int:
    """Whole simulation without any device allocation (state in the library's
    fixed 32 MiB device array); trace and outputs are device pointers."""
    rc = lib().sim_run_static(ctypes.byref(cluster), ctypes.byref(tiers), ctypes.byref(policy), replica_offsets_ptr,
                              arrival_ptr, prompt_ptr, output_ptr, tier_ptr, per_request_ptr, per_replica_ptr,
                              events_ptr or None, ctypes.c_void_p(cuda_stream or None))
    return _check(rc, None)


# ------------------------------------------------------- torch allocator --
class TorchAllocator:
    """Routes the library's device allocations through PyTorch's caching allocator."""

    def __init__(self, device: int):
        import torch

        self._torch = torch
        self.device = device

        def _alloc(_ctx, nbytes, stream):
            try:
                return int(torch.cuda.caching_allocator_alloc(int(nbytes), self.device, int(stream or 0)))
            except Exception:
                return None

        def _free(_ctx, ptr, _nbytes, _stream):
            torch.cuda.caching_allocator_delete(int(ptr))

        self._alloc = ALLOC_FN(_alloc)
        self._free = FREE_FN(_free)
        self.struct = sim_allocator_t(None, self._alloc, self._free)


# ------------------------------------------------------------ Simulator --
class Simulator:
    """One simulation object for a ``workloads.Workload`` on the current CUDA device."""

    def __init__(self, w, *, event_log_capacity: int = 4096, stream=None, torch_allocator: bool = True):
        import torch

        self._torch = torch
        if not torch.cuda.is_available():
            raise RuntimeError("Simulator needs a CUDA device")
        self.w = w
        self.device = torch.cuda.current_device()
        self.stream = stream or torch.cuda.current_stream()
        self.event_log_capacity = int(event_log_capacity)
        R = w.num_replicas
        self._cl = sim_cluster_t(R, w.num_instances, w.blocks_per_instance, w.tokens_per_block, w.max_batch)
        kmax = max(w.tables_k)
        self._tk = np.asarray(w.tables_k, np.int32)
        self._th = np.zeros((len(w.tables_k), kmax), np.int32)
        for t, h in enumerate(w.tables_h):
            self._th[t, : len(h)] = h
        self._rt = np.ascontiguousarray(w.replica_table, np.int32)
        self._tt = sim_tier_table_t(len(w.tables_k), kmax, self._tk.ctypes.data, self._th.ctypes.data,
                                    self._rt.ctypes.data)
        self._pol = sim_policy_t(0, w.enable_migration, w.iter_base_us, w.iter_us_per_prefill_token,
                                 w.iter_us_per_decode_seq, w.migrate_blocks_per_iter, w.theta_num, w.theta_den,
                                 self.event_log_capacity, w.migrate_interval_us, getattr(w, "autoscale", 0),
                                 getattr(w, "scale_out_num", -1), getattr(w, "scale_in_num", 3),
                                 getattr(w, "scale_den", 2))
        self._alloc = TorchAllocator(self.device) if torch_allocator else None
        self.handle = sim_create(self._cl, self._tt, self._pol, self.stream.cuda_stream,
                                 self._alloc.struct if self._alloc else None)
        self._trace = None

    # -- inputs
    def device_trace(self):
        t = self._torch
        w = self.w
        dev = t.device("cuda", self.device)
        self._trace = [t.from_numpy(np.ascontiguousarray(a)).to(dev) for a in
                       (w.arrival_us.view(np.int32), w.prompt_len.view(np.int16), w.output_len.view(np.int16),
                        w.tier)]
        return self._trace

    def load(self, on_device: bool = True) -> None:
        w = self.w
        self._off = np.ascontiguousarray(w.offsets, np.int64)
        drain = getattr(w, "drain_start_us", None)
        if drain is not None:
            d = np.ascontiguousarray(drain, np.uint32)
            if d.shape != (w.num_replicas, w.num_instances):
                raise ValueError("drain_start_us must be [num_replicas, num_instances]")
            sim_set_drain(self.handle, d.ctypes.data, 0)
        if on_device:
            tr = self._trace or self.device_trace()
            ptrs = [x.data_ptr() for x in tr]
            with self._torch.cuda.stream(self.stream):
                sim_load_trace(self.handle, self._off.ctypes.data, *ptrs, 1)
        else:
            self._host = [np.ascontiguousarray(a) for a in (w.arrival_us, w.prompt_len, w.output_len, w.tier)]
            sim_load_trace(self.handle, self._off.ctypes.data, *[a.ctypes.data for a in self._host], 0)

    def reset(self) -> None:
        sim_reset(self.handle)

    def run(self, max_steps: int = 1 << 62, sync: bool = True):
        return sim_run(self.handle, max_steps, sync)

    def metrics(self):
        """(per-request results, per-replica stats, migration events [R, capacity]) as numpy arrays."""
        w = self.w
        res = np.empty(w.total_requests, RESULT_DTYPE)
        st = np.empty(w.num_replicas, STATS_DTYPE)
        ev = np.empty(w.num_replicas * max(self.event_log_capacity, 1), EVENT_DTYPE)
        sim_metrics(self.handle, res.ctypes.data if len(res) else None, st.ctypes.data,
                    ev.ctypes.data if self.event_log_capacity else None, 0)
        return res, st, ev.reshape(w.num_replicas, -1)[:, : self.event_log_capacity]

    def stats(self) -> np.ndarray:
        """Per-replica stats only (STATS_DTYPE [R]); nothing else is copied."""
        st = np.empty(self.w.num_replicas, STATS_DTYPE)
        sim_metrics(self.handle, None, st.ctypes.data, None, 0)
        return st

    def set_headroom(self, tables) -> None:
        """New headroom tables, [num_tables][max_tiers] (entries past a table's K ignored)."""
        t = np.ascontiguousarray(tables, np.int32)
        if t.shape != self._th.shape:
            raise ValueError("tables must be [num_tables, max_tiers] = %s" % (self._th.shape,))
        sim_set_headroom(self.handle, t.ctypes.data)
        self._th = t

    def set_order(self, order) -> None:
        """Replica start order (a permutation of 0..R-1), or None for trace order."""
        if order is None:
            sim_set_order(self.handle, None)
            return
        self._order = np.ascontiguousarray(order, np.int32)
        if self._order.shape != (self.w.num_replicas,):
            raise ValueError("order must have one entry per replica")
        sim_set_order(self.handle, self._order.ctypes.data)

    def launch_info(self) -> dict:
        return sim_launch_info(self.handle)

    def latency_stats(self) -> np.ndarray:
        """Per-tier TTFT / TBT / E2E statistics, LATENCY_DTYPE [R, max tiers, 3]."""
        kmax = max(self.w.tables_k)
        out = np.empty(self.w.num_replicas * kmax * 3, LATENCY_DTYPE)
        sim_latency_stats(self.handle, out.ctypes.data, 0)
        return out.reshape(self.w.num_replicas, kmax, 3)

    def events_of(self, ev, st, r: int) -> np.ndarray:
        """Replica r's migration log as an (n, 6) int64 array: time, request, src, dst, blocks, kind."""
        n = min(int(st["log_events"][r]), self.event_log_capacity)
        e = ev[r, :n]
        return np.stack([e["time_us"], e["request"], e["src"], e["dst"], e["blocks"], e["kind"]],
                        axis=1).astype(np.int64)

    def device_bytes(self) -> int:
        return sim_device_bytes(self.handle)

    def close(self) -> None:
        if getattr(self, "handle", None):
            sim_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
