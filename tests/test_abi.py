"""The C-ABI library loads, exports every entry point include/mtsim.h
declares, and rejects bad arguments on the host before touching the GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2608_16336_gb300 import _build, mtsim

HEADER = os.path.join(_build.INCLUDE, "mtsim.h")


@pytest.fixture(scope="module")
def L():
    _build.build_mtsim()
    return mtsim.lib()


def declared_entry_points():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sim_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_entry_points()
    for n in ("sim_create", "sim_load_trace", "sim_run", "sim_metrics", "sim_destroy", "sim_last_error"):
        assert n in names


def test_library_exports_every_declared_symbol(L):
    for name in declared_entry_points():
        assert hasattr(L, name), name
    assert sorted(mtsim.EXPORTS) == sorted(declared_entry_points())


def test_struct_sizes_match_header():
    assert ctypes.sizeof(mtsim.sim_cluster_t) == 20
    assert ctypes.sizeof(mtsim.sim_policy_t) == 72
    assert mtsim.RESULT_DTYPE.itemsize == 16
    assert mtsim.STATS_DTYPE.itemsize == 72
    assert mtsim.EVENT_DTYPE.itemsize == 16
    assert mtsim.LATENCY_DTYPE.itemsize == 992


def _valid():
    cl = mtsim.sim_cluster_t(2, 4, 1024, 16, 64)
    tk = np.array([2], np.int32)
    th = np.array([256, 128], np.int32)
    rt = np.array([0, 0], np.int32)
    tt = mtsim.sim_tier_table_t(1, 2, tk.ctypes.data, th.ctypes.data, rt.ctypes.data)
    pol = mtsim.sim_policy_t(0, 1, 4000, 20, 30, 64, 3, 10, 1024, 50000)
    return cl, tt, pol, (tk, th, rt)


@pytest.mark.parametrize("field,value", [
    ("num_replicas", 0), ("num_instances", 0), ("num_instances", 257), ("blocks_per_instance", 0),
    ("blocks_per_instance", 65536), ("tokens_per_block", 0), ("tokens_per_block", 65), ("max_batch", 0),
    ("max_batch", 65)])
def test_create_rejects_bad_cluster(L, field, value):
    cl, tt, pol, keep = _valid()
    setattr(cl, field, value)
    out = ctypes.c_void_p()
    rc = L.sim_create(ctypes.byref(cl), ctypes.byref(tt), ctypes.byref(pol), None, None, ctypes.byref(out))
    assert rc == mtsim.SIM_ERR_ARG and not out.value
    assert L.sim_last_error(None)


@pytest.mark.parametrize("field,value", [
    ("policy", 3), ("enable_migration", 2), ("iter_base_us", -1), ("iter_base_us", 0), ("iter_us_per_decode_seq", 1 << 25),
    ("migrate_blocks_per_iter", 0), ("theta_den", 0), ("theta_num", -1), ("event_log_capacity", -5),
    ("migrate_interval_us", 0), ("migrate_interval_us", 1 << 32)])
def test_create_rejects_bad_policy(L, field, value):
    cl, tt, pol, keep = _valid()
    setattr(pol, field, value)
    out = ctypes.c_void_p()
    rc = L.sim_create(ctypes.byref(cl), ctypes.byref(tt), ctypes.byref(pol), None, None, ctypes.byref(out))
    assert rc == mtsim.SIM_ERR_ARG


@pytest.mark.parametrize("fields", [
    dict(autoscale=2), dict(autoscale=1, scale_out_num=-1, scale_in_num=3, scale_den=0),
    dict(autoscale=1, scale_out_num=-1, scale_in_num=3, scale_den=65),
    dict(autoscale=1, scale_out_num=3, scale_in_num=3, scale_den=2),
    dict(autoscale=1, scale_out_num=-5000, scale_in_num=3, scale_den=2),
    dict(autoscale=1, scale_out_num=-1, scale_in_num=4097, scale_den=2)])
def test_create_rejects_bad_autoscale(L, fields):
    cl, tt, pol, keep = _valid()
    for k, v in fields.items():
        setattr(pol, k, v)
    out = ctypes.c_void_p()
    rc = L.sim_create(ctypes.byref(cl), ctypes.byref(tt), ctypes.byref(pol), None, None, ctypes.byref(out))
    assert rc == mtsim.SIM_ERR_ARG and not out.value
    assert b"auto" in L.sim_last_error(None)


def test_create_rejects_bad_tier_tables(L):
    cl, tt, pol, (tk, th, rt) = _valid()
    out = ctypes.c_void_p()
    for mutate in (lambda: tk.__setitem__(0, 3), lambda: th.__setitem__(1, -1), lambda: rt.__setitem__(1, 1),
                   lambda: th.__setitem__(0, 600000)):
        cl, tt, pol, (tk, th, rt) = _valid()
        mutate()
        tt = mtsim.sim_tier_table_t(1, 2, tk.ctypes.data, th.ctypes.data, rt.ctypes.data)
        rc = L.sim_create(ctypes.byref(cl), ctypes.byref(tt), ctypes.byref(pol), None, None, ctypes.byref(out))
        assert rc == mtsim.SIM_ERR_ARG, L.sim_last_error(None)
    rc = L.sim_create(ctypes.byref(cl), None, ctypes.byref(pol), None, None, ctypes.byref(out))
    assert rc == mtsim.SIM_ERR_ARG
    assert L.sim_create(ctypes.byref(cl), ctypes.byref(tt), ctypes.byref(pol), None, None, None) == mtsim.SIM_ERR_ARG


def test_allocation_failure_is_reported(L):
    """An allocator that always fails makes sim_create return SIM_ERR_OOM."""
    calls = []

    def alloc(_ctx, n, _stream):
        calls.append(n)
        return None

    def free(_ctx, _p, _n, _stream):
        raise AssertionError("nothing was allocated")

    a = mtsim.sim_allocator_t(None, mtsim.ALLOC_FN(alloc), mtsim.FREE_FN(free))
    cl, tt, pol, keep = _valid()
    out = ctypes.c_void_p()
    rc = L.sim_create(ctypes.byref(cl), ctypes.byref(tt), ctypes.byref(pol), None, ctypes.byref(a), ctypes.byref(out))
    assert rc == mtsim.SIM_ERR_OOM and calls and not out.value
    assert b"allocation" in L.sim_last_error(None)


def test_null_object_calls(L):
    assert L.sim_run(None, 10, None) == mtsim.SIM_ERR_ARG
    assert L.sim_reset(None) == mtsim.SIM_ERR_ARG
    assert L.sim_set_drain(None, None, 0) == mtsim.SIM_ERR_ARG
    assert L.sim_latency_stats(None, None, 0) == mtsim.SIM_ERR_ARG
    assert L.sim_metrics(None, None, None, None, 0) == mtsim.SIM_ERR_ARG
    assert L.sim_load_trace(None, None, None, None, None, None, 0) == mtsim.SIM_ERR_ARG
    assert L.sim_device_bytes(None) == 0
    L.sim_destroy(None)
    for code in (0, -1, -2, -3, -4, -5, -7, -8, -10):
        assert L.sim_strerror(code)


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(mtsim, "_LIB", None)
    monkeypatch.setattr(_build, "MTSIM_SO", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="missing"):
        mtsim.lib()
