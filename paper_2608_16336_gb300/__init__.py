"""Batched multi-tier LLM-serving scheduler simulation on GB300 (sm_103a).

Submodules:
  workloads -- seeded synthetic inputs (cluster, tier tables, traces)
  mtsim     -- ctypes binding of the C-ABI library libmtsim.so
Importing the package loads no native code.
"""
__all__ = ["workloads", "mtsim"]
