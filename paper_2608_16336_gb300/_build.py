"""Build helpers for the in-tree native libraries.

``libtracegen.so`` (plain C, host only) and ``libmtsim.so`` (CUDA for sm_103a
plus the C-ABI host layer) are compiled into ``paper_2608_16336_gb300/_lib``.
Both are rebuilt when a source is newer than the library.
"""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
REPO_DIR = os.path.dirname(PKG_DIR)
LIB_DIR = os.path.join(PKG_DIR, "_lib")
CSRC = os.path.join(PKG_DIR, "csrc")
INCLUDE = os.path.join(REPO_DIR, "include")

TRACEGEN_SO = os.path.join(LIB_DIR, "libtracegen.so")
MTSIM_SO = os.path.join(LIB_DIR, "libmtsim.so")

ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def _stale(target: str, sources: list[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(s) > t for s in sources)


def _run(cmd: list[str]) -> None:
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError("build failed: %s\n%s\n%s" % (" ".join(cmd), res.stdout, res.stderr))


def _nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found; the CUDA toolkit is required to build libmtsim")
    return cand


def build_tracegen(force: bool = False) -> str:
    src = os.path.join(CSRC, "tracegen.c")
    if force or _stale(TRACEGEN_SO, [src]):
        os.makedirs(LIB_DIR, exist_ok=True)
        tmp = TRACEGEN_SO + ".tmp%d" % os.getpid()
        _run(["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-pthread", src, "-o", tmp, "-lm"])
        os.replace(tmp, TRACEGEN_SO)
    return TRACEGEN_SO


def mtsim_sources() -> list[str]:
    return [os.path.join(CSRC, f) for f in sorted(os.listdir(CSRC)) if f.endswith((".cu", ".cuh"))] + [
        os.path.join(INCLUDE, "mtsim.h")
    ]


def build_mtsim(force: bool = False, extra_flags: list[str] | None = None) -> str:
    """Compiles every csrc/*.cu to an object in parallel, then links libmtsim.so."""
    srcs = mtsim_sources()
    if force or extra_flags or _stale(MTSIM_SO, srcs):
        obj_dir = os.path.join(LIB_DIR, "obj")
        os.makedirs(obj_dir, exist_ok=True)
        cus = [s for s in srcs if s.endswith(".cu")]
        tag = "%d" % os.getpid()
        objs = [os.path.join(obj_dir, os.path.basename(c)[:-3] + ".%s.o" % tag) for c in cus]
        flags = [ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE] + list(extra_flags or [])
        with ThreadPoolExecutor(len(cus)) as ex:
            for f in [ex.submit(_run, [_nvcc(), "-c", c, "-o", o] + flags) for c, o in zip(cus, objs)]:
                f.result()
        tmp = MTSIM_SO + ".tmp%d" % os.getpid()
        _run([_nvcc(), ARCH, "-shared", "-Xcompiler", "-fPIC", *objs, "-o", tmp])
        os.replace(tmp, MTSIM_SO)
        for o in objs:
            os.remove(o)
    return MTSIM_SO


def build_all(force: bool = False) -> None:
    with ThreadPoolExecutor(2) as ex:
        futs = [ex.submit(build_tracegen, force), ex.submit(build_mtsim, force)]
        for f in futs:
            f.result()
