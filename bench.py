"""Throughput of the batched multi-tier scheduler simulation on GB300.

A step is one complete simulation of a workload -- by default the largest
one, 16,384 independent replicas, each a 64-instance x 2,048-block cluster
with K = 4 enterprise-mix tiers and 50,000 requests (Poisson at 0.9 of
capacity) -- from t = 0 until every request has finished: state reset plus one
persistent simulation kernel, inputs resident in HBM, every migration-log
record written (the log is sized by a first run so that no replica
overflows it).  `value` is simulated replica-steps per second (a replica-step
= one distinct event time processed in one replica), summed over GPUs.  `e2e`
repeats the measurement through the C ABI with the trace in pinned host
memory: the host-to-device copy, validation, simulation and the
device-to-host copy of every per-request result, the per-replica stats and
the migration log are inside the timed region.  The smaller workloads 0-3 are
timed after the headline and reported under `other_workloads`.

Multi-GPU (torchrun, one process per GPU): the workload's replicas are split
into contiguous ranges balanced by predicted work (requests x instances x
load), one range per rank; there is no collective on the data path, only a
barrier and a max/sum of the timings (total work fixed: strong scaling).

--impl reference times the CPU oracle (the plain single-threaded reference
simulator, one replica per host thread) on a bounded sample of the same
workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

HERE = os.path.dirname(os.path.abspath(__file__))
if HERE not in sys.path:
    sys.path.insert(0, HERE)

import numpy as np  # noqa: E402

HEADLINE_WORKLOAD = 4
WORKLOAD_NAMES = {
    0: "1 replica x 4 instances x 1,024 KV blocks (16 tokens/block, batch 64), K=2 uniform tiers, 2,000 requests, "
       "Poisson 8 req/s, H_k = 256 >> k, 64 migration blocks/iteration, 50 ms / theta 0.3 rebalancing",
    1: "1,024 replicas x 16 instances x 2,048 KV blocks (16 tokens/block, batch 64), K=4 enterprise tiers "
       "(.05/.15/.30/.50), 20,000 requests/replica, Poisson at 0.85 load, H_k = 512 >> k, "
       "64 migration blocks/iteration, 50 ms / theta 0.3 rebalancing",
    2: "3,840-replica sweep (K=1..10 x uniform/gaussian/geometric tiers x load 0.6/0.9 x 64 seeds) x 32 instances "
       "x 2,048 KV blocks, 10,000 requests/replica, Poisson, H_k = 512 >> k, 64 migration blocks/iteration",
    3: "256 replicas x 128 instances x 4,096 KV blocks, K=10 gaussian tiers, 200,000 requests/replica, bursty "
       "Gamma arrivals (CV 3) at 0.95 load, prompts LN(7.0, 1.0) in [16, 8192], H_k = 1024 >> k, "
       "32 migration blocks/iteration",
    4: "16,384 replicas x 64 instances x 2,048 KV blocks (16 tokens/block, batch 64), K=4 enterprise tiers "
       "(.05/.15/.30/.50), 50,000 requests/replica, Poisson at 0.9 load, H_k = 512 >> k, "
       "64 migration blocks/iteration, 50 ms / theta 0.3 rebalancing",
}
METRIC = "simulated replica-steps/sec (1 GB300) and achieved HBM GB/s fraction of peak"
UNIT = "replica-steps/s"
# Algorithmic bytes of the method (the least it must move through HBM):
BYTES_PER_REQUEST = 9 + 14       # read the trace record (u32, u16, u16, u8), write the result fields
BYTES_PER_MEMBER_ITERATION = 8   # read + write a running request's 2-byte token and 2-byte block counters
BYTES_PER_TOUCHED_INSTANCE = 64  # ~32 B of instance state read + written per instance touched in a step
BYTES_PER_LOG_RECORD = 16        # one migration-log record
KERNELS_PER_STEP = 3             # k_init_state, k_init_requests, k_run


def algorithmic_bytes(q: int, st) -> dict:
    """Algorithmic bytes of one complete simulation from its exact counters.
    Touched instance-steps are counted as: each iteration (its end and the
    next formation touch the instance once), each dispatched request (its
    destination), and each migration-log record (its source and destination)."""
    member = float(st["member_iterations"].sum())
    iters = float(st["iterations"].sum())
    logs = float(st["log_events"].sum())
    touched = iters + float(q) + 2.0 * logs
    total = (q * BYTES_PER_REQUEST + member * BYTES_PER_MEMBER_ITERATION + touched * BYTES_PER_TOUCHED_INSTANCE
             + logs * BYTES_PER_LOG_RECORD)
    return {"total": total, "requests": float(q), "member_iterations": member, "iterations": iters,
            "touched_instance_steps": touched, "log_records": logs}


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return ws, rank, local


def aggregate(local_seconds: float, local_units: float, local_events: float):
    """Max of the timings and sum of the work over ranks (identity at N = 1)."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return local_seconds, local_units, local_events
    dev = torch.device("cuda") if dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([local_seconds], dtype=torch.float64, device=dev)
    u = torch.tensor([local_units, local_events], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u[0].item()), float(u[1].item())


def barrier():
    import torch.distributed as dist

    if dist.is_available() and dist.is_initialized():
        dist.barrier()


def measured_peak_hbm():
    path = os.path.join(HERE, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def kernel_source_hash() -> str:
    src = os.path.join(HERE, "paper_2608_16336_gb300", "csrc", "mtsim.cu")
    return hashlib.sha256(open(src, "rb").read()).hexdigest()


def profile_record(cid: int):
    """The committed ncu figures for k_run on (a reduced case of) workload
    ``cid``: DRAM bytes per request and warp-instructions per replica-step, or
    None when the kernel source has changed since they were taken."""
    path = os.path.join(HERE, "profiles", "k_run_workload%d_traffic.json" % cid)
    try:
        with open(path) as f:
            rec = json.load(f)
        if kernel_source_hash() != rec["mtsim_cu_sha256"]:
            return None
        return rec
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, out_dir: str):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join(out_dir, "clocks_bench_%d.csv" % gpu_index)

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.QUERY,
                                          "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def sized_simulator(mtsim, w, cap: int, stream, order=None):
    """A simulator whose migration log holds every record of every replica:
    one complete run with capacity ``cap``; if some replica produced more
    records, the simulator is rebuilt with exactly enough room.  ``order``:
    the replicas' start order (sim_set_order), or None.  Returns the
    simulator (after that run), its capacity and the run's stats."""
    while True:
        sim = mtsim.Simulator(w, event_log_capacity=cap, stream=stream)
        if order is not None:
            sim.set_order(order)
        sim.load(on_device=True)
        mtsim.sim_run(sim.handle, 1 << 62, False)
        st = sim.stats()
        need = int(st["log_events"].max()) if len(st) else 0
        if need <= cap:
            return sim, cap, st
        sim.close()
        sim._trace = None
        cap = (need + 15) // 16 * 16


def initial_log_capacity(w) -> int:
    q = int(np.diff(w.offsets).max()) if w.num_replicas else 0
    return max(1024, (q * 3 // 2 + 15) // 16 * 16)


def time_device_steps(torch, mtsim, sim, stream, steps: int, warmup: int, clocks=None):
    """W untimed and K timed complete simulations (reset + run) on the device:
    (seconds per step over the whole region, mean k_run launch seconds, clocks)."""
    def step():
        mtsim.sim_reset(sim.handle)
        mtsim.sim_run(sim.handle, 1 << 62, False)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    k_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    if clocks:
        clocks.start()
    barrier()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for i in range(steps):
        mtsim.sim_reset(sim.handle)
        k_ev[i][0].record(stream)
        mtsim.sim_run(sim.handle, 1 << 62, False)
        k_ev[i][1].record(stream)
    t1.record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop() if clocks else None
    dev_s = t0.elapsed_time(t1) / 1e3
    k_s = sum(a.elapsed_time(b) for a, b in k_ev) / 1e3 / steps
    return dev_s, k_s, clk


def bench_gpu(args):
    import torch

    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    from paper_2608_16336_gb300 import mtsim, workloads

    cid = args.workload
    r_all = args.replicas or workloads.num_replicas(cid)
    work = workloads.predicted_work(cid, args.requests)[:r_all]
    lo, hi = workloads.partition(work, ws)[rank]
    w = workloads.config(cid, replicas=range(lo, hi), requests=args.requests)
    stream = torch.cuda.current_stream()
    # replicas with the most predicted work start first (ties: trace order)
    order = None if args.trace_order else np.argsort(-work[lo:hi], kind="stable").astype(np.int32)
    sim, cap, st0 = sized_simulator(mtsim, w, args.log_capacity or initial_log_capacity(w), stream, order)
    R, Q = w.num_replicas, w.total_requests

    clocks = ClockSampler(local, args.clocks_dir)
    dev_s, k_s, clk = time_device_steps(torch, mtsim, sim, stream, args.steps, args.warmup, clocks)

    st = sim.stats()
    assert (st["status"] == mtsim.SIM_REPLICA_DONE).all(), "a replica did not finish"
    assert int(st["log_events"].max()) <= cap, "a replica overflowed its migration log"
    assert (st["steps"] == st0["steps"]).all() and (st["log_events"] == st0["log_events"]).all()
    launch = sim.launch_info()
    lat_info = time_latency_stats(torch, mtsim, sim, w, stream)
    steps_per_run = float(st["steps"].sum())
    events_per_run = float(st["events"].sum())
    alg = algorithmic_bytes(Q, st)

    # end to end through the C ABI with pinned host buffers: trace in, every
    # result, the per-replica stats and the whole migration log out
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
    h_arr, h_p, h_o, h_t = (pin(w.arrival_us.view(np.int32)), pin(w.prompt_len.view(np.int16)),
                            pin(w.output_len.view(np.int16)), pin(w.tier))
    h_res = torch.empty(Q * mtsim.RESULT_DTYPE.itemsize, dtype=torch.uint8).pin_memory()
    h_st = torch.empty(R * mtsim.STATS_DTYPE.itemsize, dtype=torch.uint8).pin_memory()
    h_ev = torch.empty(R * cap * mtsim.EVENT_DTYPE.itemsize, dtype=torch.uint8).pin_memory()
    off = np.ascontiguousarray(w.offsets, np.int64)

    def e2e_step():
        mtsim.sim_load_trace(sim.handle, off.ctypes.data, h_arr.data_ptr(), h_p.data_ptr(), h_o.data_ptr(),
                             h_t.data_ptr(), 0)
        mtsim.sim_run(sim.handle, 1 << 62, False)
        mtsim.sim_metrics(sim.handle, h_res.data_ptr(), h_st.data_ptr(), h_ev.data_ptr(), 0)

    e2e_step()
    barrier()
    torch.cuda.synchronize()
    e0 = time.perf_counter()
    for _ in range(args.e2e_steps):
        e2e_step()
    torch.cuda.synchronize()
    barrier()
    e2e_s = (time.perf_counter() - e0) / args.e2e_steps
    st_e2e = h_st.numpy().view(mtsim.STATS_DTYPE)
    assert (st_e2e["steps"] == st["steps"]).all() and (st_e2e["status"] == 0).all()
    h2d = int(off.nbytes + Q * 9)
    d2h = int(h_res.numel() + h_st.numel() + h_ev.numel())
    sim.close()
    del sim, h_arr, h_p, h_o, h_t, h_res, h_st, h_ev

    tot_s, tot_units, tot_events = aggregate(dev_s, steps_per_run * args.steps, events_per_run * args.steps)
    e2e_max, e2e_units, _ = aggregate(e2e_s, steps_per_run, events_per_run)
    peak, peak_kind = measured_peak_hbm()
    achieved = alg["total"] / k_s / 1e9
    prof = profile_record(cid)
    sm_mhz = (clk or {}).get("sm_mhz") or 0.0
    resident = min(R, launch["grid_blocks"] * launch["block_threads"] // 32)
    latency = {
        "bound": "dependent instruction chain per replica (one warp per replica)",
        "sm_mhz": sm_mhz or None,
        "resident_warps": resident,
        "replicas": R,
        "cycles_per_replica_step_per_warp": (k_s * sm_mhz * 1e6 * resident / steps_per_run) if sm_mhz else None,
        "longest_replica_steps": int(st["steps"].max()),
        "mean_replica_steps": float(st["steps"].mean()),
        "cycles_per_step_of_longest_replica": (k_s * sm_mhz * 1e6 / float(st["steps"].max())) if sm_mhz else None,
        "warp_instructions_per_replica_step": prof.get("warp_instructions_per_replica_step") if prof else None,
        "launch": launch,
    }
    line = {
        "metric": METRIC,
        "value": tot_units / tot_s,
        "unit": UNIT,
        "n_gpus": ws,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": tot_s / args.steps * 1e3,
        "higher_is_better": True,
        "scaling": "strong",
        "vs_baseline": None,
        "dtype": "int32",
        "data": "synthetic (seeded traces shaped like the paper's workloads; no dataset)",
        "config": {
            "workload": WORKLOAD_NAMES[cid] if not (args.replicas or args.requests) else
            "REDUCED profiling case of: " + WORKLOAD_NAMES[cid],
            "workload_id": cid,
            "replicas": r_all,
            "replicas_this_gpu": [lo, hi],
            "requests_this_gpu": Q,
            "replica_steps_per_gpu_step": int(steps_per_run),
            "migration_log_capacity": cap,
            "migration_log_records": int(st["log_events"].sum()),
            "max_log_records_per_replica": int(st["log_events"].max()),
            "parallelism": "replicas partitioned across GPUs by predicted work, no collective on the data path",
            "replica_order": "trace order" if args.trace_order else "descending predicted work (requests x instances x load), ties in trace order",
            "l2": "inputs larger than L2: trace %.0f MB + per-request state %.0f MB resident" % (
                Q * 9 / 1e6, Q * 32 / 1e6),
        },
        "request_events_per_s": tot_events / tot_s,
        "e2e": {"value": e2e_units / e2e_max, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": KERNELS_PER_STEP * args.steps,
        "roofline": {
            "bound": "hbm",
            "achieved": achieved,
            "peak": peak,
            "peak_kind": peak_kind,
            "unit": "GB/s",
            "frac": achieved / peak,
            "traffic": float(prof["dram_bytes_per_request"]) * Q if prof else None,
            "kernel": "k_run",
            "kernel_ms": k_s * 1e3,
            "algorithmic_bytes_per_launch": alg["total"],
            "algorithmic_terms": alg,
        },
        "latency": latency,
        "clocks": clk,
        "aux_kernels": [lat_info],
    }
    if ws == 1 and not args.no_others:
        line["other_workloads"] = [bench_other(torch, mtsim, workloads, c, stream, args)
                                   for c in sorted(WORKLOAD_NAMES) if c != cid]
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, cid, args.cpu_replicas)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


def bench_other(torch, mtsim, workloads, cid: int, stream, args) -> dict:
    """One smaller workload at full size, timed the same way (3 warm-up and
    3 timed complete simulations, every log record kept, the same replica
    order rule)."""
    w = workloads.config(cid)
    order = None if args.trace_order else np.argsort(-workloads.predicted_work(cid), kind="stable").astype(np.int32)
    sim, cap, _ = sized_simulator(mtsim, w, initial_log_capacity(w), stream, order)
    dev_s, k_s, _ = time_device_steps(torch, mtsim, sim, stream, 3, 3)
    st = sim.stats()
    launch = sim.launch_info()
    sim.close()
    assert (st["status"] == mtsim.SIM_REPLICA_DONE).all() and int(st["log_events"].max()) <= cap
    alg = algorithmic_bytes(w.total_requests, st)
    peak, _ = measured_peak_hbm()
    steps = float(st["steps"].sum())
    return {"workload_id": cid, "workload": WORKLOAD_NAMES[cid], "value": steps / (dev_s / 3), "unit": UNIT,
            "ms_per_step": dev_s / 3 * 1e3, "kernel_ms": k_s * 1e3, "replica_steps": int(steps),
            "longest_replica_steps": int(st["steps"].max()), "migration_log_capacity": cap,
            "hbm_frac": alg["total"] / k_s / 1e9 / peak, "launch": launch}


def time_latency_stats(torch, mtsim, sim, w, stream, reps: int = 10) -> dict:
    """CUDA-event time of the per-tier latency reduction (sim_latency_stats) over the
    finished simulation, device output, outside the timed step: the histogram
    pass, the percentile buckets and the exact selection passes.  Its inputs
    (16 + 4 + 2 + 1 bytes per request) are larger than L2 at this size."""
    R, Q = w.num_replicas, w.total_requests
    kmax = max(w.tables_k)
    out = torch.empty(R * kmax * 3 * mtsim.LATENCY_DTYPE.itemsize, dtype=torch.uint8, device=stream.device)
    for _ in range(3):
        mtsim.sim_latency_stats(sim.handle, out.data_ptr(), 1)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    torch.cuda.synchronize()
    for a, b in ev:
        a.record(stream)
        mtsim.sim_latency_stats(sim.handle, out.data_ptr(), 1)
        b.record(stream)
    torch.cuda.synchronize()
    ms = sum(a.elapsed_time(b) for a, b in ev) / reps
    nbytes = Q * (16 + 4 + 2 + 1) + out.numel()
    peak, kind = measured_peak_hbm()
    gbs = nbytes / (ms / 1e3) / 1e9
    return {"kernel": "sim_latency_stats: k_latency_hist, k_latency_pct and up to four k_latency_refine + "
                      "k_latency_step selection passes (output clear included)",
            "work": "per-tier TTFT/TBT/E2E histograms and exact nearest-rank P50/P90/P99 of every request; "
                    "algorithmic bytes = one read of the inputs, which each selection pass still open reads again",
            "bound": "hbm", "ms": ms, "algorithmic_bytes_per_launch": nbytes, "achieved": gbs, "peak": peak,
            "peak_kind": kind, "unit": "GB/s", "frac": gbs / peak}


def cpu_baseline(w, cid: int, nrep: int) -> dict:
    """The oracle, as it stands, on the first `nrep` replicas of the same
    workload, one replica per host thread on all host cores."""
    from oracle import oracle

    cores = os.cpu_count() or 1
    reps = list(range(min(nrep, w.num_replicas)))
    q = int(np.diff(w.offsets).max())
    r = oracle.timed_sample(w, reps, cores)
    one = oracle.timed_sample(w, reps[:4], 1)  # the same oracle on one core, one replica at a time
    return {"value": r["steps"] / r["seconds"], "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "first %d of %d replicas of workload %d, full %d requests each (%d replica-steps, %.1f s wall)"
                      % (len(reps), w.num_replicas, cid, q, r["steps"], r["seconds"]),
            "request_events_per_s": r["events"] / r["seconds"],
            "single_core": {"value": one["steps"] / one["seconds"], "unit": UNIT,
                            "sample": "first %d replicas, one after another on one thread (%.2f s)" % (
                                one["replicas"], one["seconds"])}}


def bench_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    from oracle import oracle
    from paper_2608_16336_gb300 import workloads

    cid = args.workload
    cores = os.cpu_count() or 1
    n = min(args.cpu_replicas_per_step, workloads.num_replicas(cid))
    w = workloads.config(cid, replicas=range(n))
    reps = list(range(n))
    for _ in range(args.warmup):
        oracle.timed_sample(w, reps[: max(1, min(cores, n))], cores)
    tot_s, tot_steps, tot_events = 0.0, 0, 0
    for i in range(args.steps):
        r = oracle.timed_sample(w, reps, cores)
        tot_s += r["seconds"]
        tot_steps += r["steps"]
        tot_events += r["events"]
    value = tot_steps / tot_s
    sample = "first %d of %d replicas of workload %d per step, full requests" % (
        n, workloads.num_replicas(cid), cid)
    line = {
        "impl": "reference",
        "metric": METRIC,
        "value": value,
        "unit": UNIT,
        "n_gpus": ws,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": tot_s / args.steps * 1e3,
        "higher_is_better": True,
        "scaling": "strong",
        "vs_baseline": None,
        "dtype": "int64",
        "data": "synthetic (seeded traces shaped like the paper's workloads; no dataset)",
        "config": {"workload": WORKLOAD_NAMES[cid], "workload_id": cid, "sample_per_step": sample},
        "request_events_per_s": tot_events / tot_s,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", type=int, default=HEADLINE_WORKLOAD, choices=sorted(WORKLOAD_NAMES))
    ap.add_argument("--e2e-steps", type=int, default=2)
    ap.add_argument("--log-capacity", type=int, default=0,
                    help="initial migration-log capacity per replica (0: 1.5 x requests); grown to fit every record")
    ap.add_argument("--cpu-replicas", type=int, default=192)
    ap.add_argument("--cpu-replicas-per-step", type=int, default=64)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-others", action="store_true", help="skip the smaller workloads' lines")
    ap.add_argument("--trace-order", action="store_true",
                    help="start replicas in trace order instead of by descending predicted work")
    ap.add_argument("--clocks-dir", default=os.path.join(tempfile.gettempdir(), "mtsim_bench"),
                    help="where the raw nvidia-smi clock samples of the timed region are written")
    ap.add_argument("--replicas", type=int, default=0, help="profiling only: first N replicas of the workload")
    ap.add_argument("--requests", type=int, default=None, help="profiling only: requests per replica")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("at least 3 warm-up steps are required")
    if args.impl == "reference":
        bench_reference(args)
    else:
        bench_gpu(args)


if __name__ == "__main__":
    main()
