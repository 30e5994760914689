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
                                         fake, fake, fake, fake, None, None)
    assert rc == kvev.ENOMEM
