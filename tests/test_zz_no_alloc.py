"""GPU test of kvev_evict_prefill_noalloc, the prefill eviction for callers that
cannot allocate device memory (their allocator or framework owns all of it, or
cudaMalloc is off limits where they run).  It must give the same kept
positions, counts, gathered K/V rows and H2O state as kvev_evict_prefill with a
caller workspace, on two calls in a row (the library's scratch keeps the last
call's contents between them), and refuse requests larger than its scratch.

The file name makes pytest collect it last.
"""
import ctypes as C

import numpy as np
import pytest

from paper_2606_15157_gb300 import inputs as gen

pytestmark = pytest.mark.gpu

REL = 2e-3  # score tolerance used by the parity tests


@pytest.fixture(scope="module")
def env():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_15157_gb300 import kvev
    kvev.load()
    return torch, kvev


def _run_both(torch, kvev, wl, dev):
    plan = kvev.Plan.from_workload(wl)
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    K = [dev[l][0] for l in range(wl.L)]
    V = [dev[l][1] for l in range(wl.L)]
    Q = [dev[l][2] for l in range(wl.L)]
    ref = plan.buffers(wl.B, wl.S_cap)
    plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, ref)
    torch.cuda.synchronize()
    assert plan.status() == kvev.OK
    ptr = lambda t: None if t is None else t.data_ptr()
    outs = []
    for _ in range(2):  # two calls in a row share the library's scratch
        b = plan.buffers(wl.B, wl.S_cap)
        for k in ("out_K", "out_V", "out_idx", "h2o_state"):
            b[k].fill_(7)  # make stale values visible
        status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        rc = kvev.kvev_evict_prefill_noalloc(
            plan.handle, [ptr(k) for k in K], [ptr(v) for v in V], [ptr(q) for q in Q],
            lens.data_ptr(), wl.B, wl.S_cap, b["out_K"].data_ptr(), b["out_V"].data_ptr(),
            b["out_idx"].data_ptr(), b["out_count"].data_ptr(), b["h2o_state"].data_ptr(),
            status.data_ptr(), torch.cuda.current_stream().cuda_stream)
        assert rc == kvev.OK
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        outs.append(b)
    rows = ref["rows"]
    for b in outs:
        assert torch.equal(b["out_count"], ref["out_count"])
        assert torch.equal(b["out_idx"][:rows], ref["out_idx"][:rows])
        assert torch.equal(b["out_K"][:rows].view(torch.int16), ref["out_K"][:rows].view(torch.int16))
        assert torch.equal(b["out_V"][:rows].view(torch.int16), ref["out_V"][:rows].view(torch.int16))
        h2o_rows = np.zeros(rows, bool)
        for l in range(wl.L):
            if wl.route[l] == gen.H2O:
                off = plan.layer_offset(wl.B, l)
                h2o_rows[off: off + wl.B * wl.H_kv * int(wl.budget[l])] = True
        idx = ref["out_idx"][:rows].cpu().numpy()
        sel = h2o_rows & (idx >= 0)
        a = b["h2o_state"][:rows].cpu().numpy()[sel].astype(np.float64)
        r = ref["h2o_state"][:rows].cpu().numpy()[sel].astype(np.float64)
        assert np.all(np.abs(a - r) <= REL * np.maximum(np.abs(r), 1e-4 * max(r.max(initial=0), 1e-30)))
    return plan


def test_noalloc_matches_workspace_entry_tiny(env):
    torch, kvev = env
    wl = gen.config_tiny(seed=2)
    host = gen.host_tensors(wl)
    f = lambda a: torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)
    dev = {l: (f(K), f(V), f(Q)) for l, (K, V, Q) in host.items()}
    _run_both(torch, kvev, wl, dev)


def test_noalloc_matches_workspace_entry_8k(env):
    # 32 SnapKV layers at 8K: several chunks per unit, so the cross-CTA
    # normaliser hand-off runs through the library's scratch as well.
    torch, kvev = env
    wl = gen.config_homog8k(seed=0)
    plan = kvev.Plan.from_workload(wl)
    assert plan.query(wl.B, wl.S_cap)[3] <= kvev.NOALLOC_SCRATCH_BYTES
    dev = {l: gen.device_layer(wl, l) for l in range(wl.L)}
    _run_both(torch, kvev, wl, dev)


def test_noalloc_rejects_requests_beyond_its_scratch(env):
    torch, kvev = env
    wl = gen.config_long(kvev.alloc_from_scores, seed=0)
    plan = kvev.Plan.from_workload(wl)
    assert plan.query(wl.B, wl.S_cap)[3] > kvev.NOALLOC_SCRATCH_BYTES
    fake = 1 << 20  # never dereferenced: the size check comes before any device work
    ptrs = [fake] * wl.L
    rc = kvev.kvev_evict_prefill_noalloc(plan.handle, ptrs, ptrs, ptrs, fake, wl.B, wl.S_cap, fake,
                                         fake, fake, fake, fake, fake, None)
    assert rc == kvev.ENOMEM


def _tiny_call(torch, kvev, plan, wl, dev, status):
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    b = plan.buffers(wl.B, wl.S_cap)
    ptr = lambda t: t.data_ptr()
    rc = kvev.kvev_evict_prefill_noalloc(
        plan.handle, [ptr(dev[l][0]) for l in range(wl.L)], [ptr(dev[l][1]) for l in range(wl.L)],
        [ptr(dev[l][2]) for l in range(wl.L)], lens.data_ptr(), wl.B, wl.S_cap,
        b["out_K"].data_ptr(), b["out_V"].data_ptr(), b["out_idx"].data_ptr(),
        b["out_count"].data_ptr(), b["h2o_state"].data_ptr(),
        None if status is None else status.data_ptr(), torch.cuda.current_stream().cuda_stream)
    return rc, b


def _tiny_env(torch):
    wl = gen.config_tiny(seed=1)
    host = gen.host_tensors(wl)
    f = lambda a: torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)
    return wl, {l: (f(K), f(V), f(Q)) for l, (K, V, Q) in host.items()}


def test_noalloc_requires_a_status_word(env):
    # The status word is where this call's device-side errors go; without one
    # they could not be seen, so the call refuses to run.
    torch, kvev = env
    wl, dev = _tiny_env(torch)
    plan = kvev.Plan.from_workload(wl)
    rc, _ = _tiny_call(torch, kvev, plan, wl, dev, None)
    assert rc == kvev.EINVAL


def test_noalloc_reports_a_wait_that_ran_out(env):
    # A unit whose normaliser is never published (test hook): the kernels give
    # up after the plan's short wait limit and record the timeout bit in the
    # caller's status word, not in the plan's; a clean call then reports 0.
    torch, kvev = env
    wl, dev = _tiny_env(torch)
    plan = kvev.Plan.from_workload(wl)
    kvev.kvev_plan_set_wait_limit(plan.handle, 20_000_000)  # 20 ms
    kvev.kvev_plan_debug_stall_unit(plan.handle, 0)
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    rc, _ = _tiny_call(torch, kvev, plan, wl, dev, status)
    assert rc == kvev.OK
    torch.cuda.synchronize()
    assert int(status.item()) & 1  # the timeout bit
    assert plan.status() == kvev.OK  # never reported through the plan
    kvev.kvev_plan_debug_stall_unit(plan.handle, -1)
    rc, _ = _tiny_call(torch, kvev, plan, wl, dev, status)
    assert rc == kvev.OK
    torch.cuda.synchronize()
    assert int(status.item()) == 0


def test_noalloc_call_allocates_no_device_memory(env):
    # After a first call (which looks up the scratch address on this device),
    # a call leaves the device's free memory exactly as it was.
    torch, kvev = env
    wl, dev = _tiny_env(torch)
    plan = kvev.Plan.from_workload(wl)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    b = plan.buffers(wl.B, wl.S_cap)
    args = ([dev[l][0].data_ptr() for l in range(wl.L)], [dev[l][1].data_ptr() for l in range(wl.L)],
            [dev[l][2].data_ptr() for l in range(wl.L)], lens.data_ptr(), wl.B, wl.S_cap,
            b["out_K"].data_ptr(), b["out_V"].data_ptr(), b["out_idx"].data_ptr(),
            b["out_count"].data_ptr(), b["h2o_state"].data_ptr(), status.data_ptr(),
            torch.cuda.current_stream().cuda_stream)
    assert kvev.kvev_evict_prefill_noalloc(plan.handle, *args) == kvev.OK
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(3):
        assert kvev.kvev_evict_prefill_noalloc(plan.handle, *args) == kvev.OK
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert int(status.item()) == 0
