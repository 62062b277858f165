"""The allocation-free entry point sim_run_static, for callers that cannot
call cudaMalloc (their device memory belongs to another allocator or budget,
or they run where an allocation is not allowed).  It must give exactly the
oracle's results and those of the allocating path (sim_create ...
sim_metrics), call after call, although every call reuses the same fixed
device array, and a call must not change the device's free memory."""
import ctypes

import numpy as np
import pytest

from paper_2608_16336_gb300 import mtsim
from paper_2608_16336_gb300 import workloads as W
from tests import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    t = pytest.importorskip("torch")
    if not t.cuda.is_available():
        pytest.skip("no CUDA device")
    t.cuda.set_device(0)
    return t


def _static_args(torch, w, cap):
    """sim_run_static's arguments for w: host descriptors, caller-owned device
    trace and output buffers, the current stream."""
    R = w.num_replicas
    kmax = max(w.tables_k)
    tk = np.asarray(w.tables_k, np.int32)
    th = np.zeros((len(w.tables_k), kmax), np.int32)
    for t, h in enumerate(w.tables_h):
        th[t, : len(h)] = h
    rt = np.ascontiguousarray(w.replica_table, np.int32)
    cl = mtsim.sim_cluster_t(R, w.num_instances, w.blocks_per_instance, w.tokens_per_block, w.max_batch)
    tt = mtsim.sim_tier_table_t(len(w.tables_k), kmax, tk.ctypes.data, th.ctypes.data, rt.ctypes.data)
    pol = mtsim.sim_policy_t(0, w.enable_migration, w.iter_base_us, w.iter_us_per_prefill_token,
                             w.iter_us_per_decode_seq, w.migrate_blocks_per_iter, w.theta_num, w.theta_den, cap,
                             w.migrate_interval_us)
    off = np.ascontiguousarray(w.offsets, np.int64)
    dev = torch.device("cuda", 0)
    tr = [torch.from_numpy(np.ascontiguousarray(a)).to(dev) for a in
          (w.arrival_us.view(np.int32), w.prompt_len.view(np.int16), w.output_len.view(np.int16), w.tier)]
    res = torch.empty(w.total_requests * mtsim.RESULT_DTYPE.itemsize, dtype=torch.uint8, device=dev)
    st = torch.empty(R * mtsim.STATS_DTYPE.itemsize, dtype=torch.uint8, device=dev)
    ev = torch.empty(R * cap * mtsim.EVENT_DTYPE.itemsize, dtype=torch.uint8, device=dev)
    keep = (tk, th, rt, off, tr, res, st, ev)  # the buffers must outlive the call
    return _StaticArgs(cl, tt, pol, off, tr, res, st, ev, keep)


class _StaticArgs(tuple):
    """(cluster, tiers, policy, offsets ptr, 4 trace ptrs, res ptr, stats ptr,
    events ptr, stream) plus the tensors behind them."""

    def __new__(cls, cl, tt, pol, off, tr, res, st, ev, keep):
        import torch as _t

        self = super().__new__(cls, (cl, tt, pol, off.ctypes.data, *[x.data_ptr() for x in tr], res.data_ptr(),
                                     st.data_ptr(), ev.data_ptr(), _t.cuda.current_stream().cuda_stream))
        self.keep = keep
        self.res, self.st, self.ev = res, st, ev
        return self


def _static_run(torch, w, cap):
    """Runs w through sim_run_static with caller-owned device inputs and outputs."""
    R = w.num_replicas
    args = _static_args(torch, w, cap)
    res, st, ev = args.res, args.st, args.ev
    torch.cuda.synchronize()
    mtsim.sim_run_static(*args)
    res_h = res.cpu().numpy().view(mtsim.RESULT_DTYPE)
    st_h = st.cpu().numpy().view(mtsim.STATS_DTYPE)
    ev_h = ev.cpu().numpy().view(mtsim.EVENT_DTYPE).reshape(R, cap)
    events = []
    for r in range(R):
        n = min(int(st_h["log_events"][r]), cap)
        e = ev_h[r, :n]
        events.append(np.stack([e["time_us"], e["request"], e["src"], e["dst"], e["blocks"], e["kind"]],
                               axis=1).astype(np.int64))
    return res_h, st_h, events


def test_static_entry_point_matches_allocating_path(torch):
    cap = 2048
    w = W.config(1, replicas=range(11), requests=2500)
    want = parity.run_gpu(w, event_log_capacity=cap)
    ref = parity.run_oracle(w, range(w.num_replicas), event_log_capacity=cap)
    for _ in range(2):  # the second call reuses the scratch the first one left behind
        got = _static_run(torch, w, cap)
        for r in range(w.num_replicas):  # against the oracle itself ...
            parity.compare_replica(w, r, got[0], got[1], got[2], ref[r])
        assert (got[0] == want[0]).all()  # ... and the allocating path
        assert (got[1] == want[1]).all()
        for a, b in zip(got[2], want[2]):
            assert (a == b).all()
    # a different shape right after, on the same scratch
    w0 = W.config(0, requests=500)
    want0 = parity.run_gpu(w0, event_log_capacity=cap)
    got0 = _static_run(torch, w0, cap)
    assert (got0[0] == want0[0]).all() and (got0[1] == want0[1]).all()


def test_static_entry_point_allocates_nothing(torch):
    """With the module loaded and the outputs allocated, a call leaves the
    device's free memory exactly as it found it."""
    cap = 256
    w = W.config(0, requests=300)
    _static_run(torch, w, cap)  # loads the kernels and settles local-memory reservations
    args = _static_args(torch, w, cap)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    mtsim.sim_run_static(*args)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


def test_static_entry_point_reports_unfinished(torch):
    """A replica that cannot finish (its iteration end overflows 32-bit time)
    makes the call return SIM_ERR_UNFINISHED, with the replica's status in
    per_replica."""
    base = 1 << 24
    tr = (np.array([0xFFFF0000], np.uint32), np.array([1], np.uint16), np.array([2], np.uint16),
          np.array([0], np.uint8))
    ok = (np.array([0], np.uint32), np.array([1], np.uint16), np.array([2], np.uint16), np.array([0], np.uint8))
    w = W.custom(2, 16, [1], [[0]], [0, 0], [ok, tr], iter_base_us=base)
    args = _static_args(torch, w, 16)
    with pytest.raises(mtsim.SimError) as e:
        mtsim.sim_run_static(*args)
    assert e.value.code == mtsim.SIM_ERR_UNFINISHED
    st_h = args.st.cpu().numpy().view(mtsim.STATS_DTYPE)
    assert int(st_h["status"][0]) == mtsim.SIM_REPLICA_DONE
    assert int(st_h["status"][1]) == mtsim.SIM_ERR_OVERFLOW


def test_static_entry_point_rejects_oversize(torch):
    w = W.config(1, replicas=range(2), requests=10)
    w.offsets = np.array([0, 10, 10 + 4_000_000], np.int64)  # 4M records need > 32 MiB of state
    R = 2
    tk = np.array([4], np.int32)
    th = np.array([512, 256, 128, 64], np.int32)
    rt = np.zeros(R, np.int32)
    cl = mtsim.sim_cluster_t(R, 16, 2048, 16, 64)
    tt = mtsim.sim_tier_table_t(1, 4, tk.ctypes.data, th.ctypes.data, rt.ctypes.data)
    pol = mtsim.sim_policy_t(0, 1, 4000, 20, 30, 64, 3, 10, 0, 50000)
    # real (small) device buffers: the size check must reject the call before any of them is used
    small = [torch.zeros(64, dtype=torch.uint8, device="cuda") for _ in range(6)]
    with pytest.raises(mtsim.SimError) as e:
        mtsim.sim_run_static(cl, tt, pol, w.offsets.ctypes.data, *[x.data_ptr() for x in small], None,
                             torch.cuda.current_stream().cuda_stream)
    assert e.value.code == mtsim.SIM_ERR_ARG
    assert "scratch" in str(e.value)
