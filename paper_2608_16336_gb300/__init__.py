"""Batched multi-tier LLM-serving scheduler simulation on GB300 (sm_103a).

Submodules:
  workloads -- seeded synthetic inputs (cluster, tier tables, traces)
  mtsim     -- ctypes binding of the C-ABI library libmtsim.so
Importing the package loads no native code.

Example (a CUDA device and a built library: ``python -c "import
__graft_entry__ as g; g.build()"`` at the repository root)::

    import torch
    from paper_2608_16336_gb300 import mtsim, workloads

    w = workloads.config(1, replicas=range(64))   # 64 clusters of 16 instances
    w.autoscale = 1                               # report the Sec. 3.6 signal
    sim = mtsim.Simulator(w, event_log_capacity=4096)
    sim.load()                                    # trace to the GPU, validated
    assert sim.run() == 0                         # every replica finished
    res, stats, log = sim.metrics()               # per request / replica / log
    lat = sim.latency_stats()                     # [replica, tier, TTFT|TBT|E2E]
    print(lat[0, 0, mtsim.SIM_LAT_TTFT]["p99_us"], stats["steps"].sum())
    sim.close()

Draining (Sec. 3.5) is an input: set ``w.drain_start_us`` to a uint32
[replicas, instances] array of start times (0xFFFFFFFF = never) before
``load``.  ``workloads.custom`` builds a workload from explicit traces.
"""
__all__ = ["workloads", "mtsim"]
