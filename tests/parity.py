"""Parity helpers: run the CUDA path and the oracle on the same seeded inputs and
compare them under the match criteria.

Criteria (fp32 accumulation from bf16 against the fp64 oracle):
  * window scores: |gpu - ref| <= 2e-3 * max(|ref|, 1e-4 * max_k ref);
  * kept positions: identical sets, except positions whose oracle key (pooled
    score for SnapKV, raw score for H2O) lies within 2e-3 (relative) of the
    oracle's k-th largest key; counts exact, ascending order, -1 padding;
  * gathered K/V rows: byte-identical to the source rows of the kept positions,
    zero rows in unused slots;
  * H2O state: the kept positions' scores, within the score tolerance.
"""
from __future__ import annotations

import numpy as np

from paper_2606_15157_gb300 import inputs as gen

REL = 2e-3
FLOOR = 1e-4


def oracle_method(m: int) -> int:
    # The oracle numbers its operators the same way; map explicitly anyway.
    import oracle
    return {gen.FULL: oracle.FULL, gen.SNAPKV: oracle.SNAPKV, gen.H2O: oracle.H2O,
            gen.STREAMING: oracle.STREAMING}[int(m)]


def score_tol(ref: np.ndarray) -> np.ndarray:
    mx = float(ref.max()) if ref.size else 0.0
    return REL * np.maximum(np.abs(ref), FLOOR * mx)


class GpuRun:
    """Outputs of one kvev_evict_prefill call, copied to the host."""

    def __init__(self, plan, wl, bufs, lens_np):
        import torch
        torch.cuda.synchronize()
        self.plan, self.wl = plan, wl
        self.idx = bufs["out_idx"].cpu().numpy()
        self.count = bufs["out_count"].cpu().numpy()
        self.state = bufs["h2o_state"].cpu().numpy()
        self.bufs = bufs
        self.lens = lens_np
        self._outK = bufs["out_K"]
        self._outV = bufs["out_V"]
        self.scores = {}
        for l in range(wl.L):
            if wl.route[l] in (gen.SNAPKV, gen.H2O):
                self.scores[l] = plan.scores(bufs, wl.B, wl.S_cap, l).cpu().numpy()

    def unit_rows(self, l, s, h):
        b = int(self.wl.budget[l])
        base = self.plan.layer_offset(self.wl.B, l) + (s * self.wl.H_kv + h) * b
        return base, b

    def out_rows(self, base, b):
        import torch
        kk = self._outK[base: base + b].view(torch.int16).cpu().numpy().view(np.uint16)
        vv = self._outV[base: base + b].view(torch.int16).cpu().numpy().view(np.uint16)
        return kk, vv


def oracle_spec(wl, l, s, h, K_rows, Q_group):
    return dict(method=oracle_method(wl.route[l]), n=int(wl.lens[s]) if np.ndim(wl.lens) else int(wl.lens),
                b=int(wl.budget[l]), W=wl.W, pool_kernel=wl.pool_kernel, pool_type=wl.pool_type,
                sink=wl.sink, recent=wl.recent, h2o_recent=wl.h2o_recent, K=K_rows, Q=Q_group)


def check_unit(wl, l, s, h, n, res, gpu: GpuRun, K_rows, V_rows, stats=None):
    """Compare one unit.  K_rows/V_rows: uint16 [>=n][d] source rows (host)."""
    route = int(wl.route[l])
    if route == gen.FULL:
        assert gpu.count[l, s, h] == n
        return
    b = int(wl.budget[l])
    where = f"layer {l} seq {s} head {h} (n={n}, b={b}, route={route})"
    base, _ = gpu.unit_rows(l, s, h)
    idx_g = gpu.idx[base: base + b]
    cnt_g = int(gpu.count[l, s, h])
    if n == 0:
        assert cnt_g == 0 and np.all(idx_g == -1), f"{where}: empty sequence"
        Kg, Vg = gpu.out_rows(base, b)
        assert not Kg.any() and not Vg.any(), f"{where}: unused slots not zero"
        return
    assert cnt_g == res.count, f"{where}: count {cnt_g} != {res.count}"
    assert np.all(idx_g[cnt_g:] == -1), f"{where}: padding not -1"
    kept = idx_g[:cnt_g]
    assert np.all(np.diff(kept) > 0), f"{where}: indices not ascending"
    assert kept.size == 0 or (kept[0] >= 0 and kept[-1] < n), f"{where}: index out of range"

    # ---- scores ----
    identity = n <= b if route != gen.STREAMING else False
    scored = route == gen.H2O or (route == gen.SNAPKV and not identity)
    if scored:
        raw_g = gpu.scores[l][s, h, :n].astype(np.float64)
        raw_o = res.raw
        err = np.abs(raw_g - raw_o)
        tol = score_tol(raw_o)
        bad = np.nonzero(err > tol)[0]
        assert bad.size == 0, (f"{where}: {bad.size} scores off, first k={bad[0]} gpu={raw_g[bad[0]]} "
                               f"ref={raw_o[bad[0]]}")
        if stats is not None:
            stats.setdefault("max_rel_err", 0.0)
            rel = err / np.maximum(np.abs(raw_o), FLOOR * raw_o.max())
            stats["max_rel_err"] = max(stats["max_rel_err"], float(rel.max()))

    # ---- kept set ----
    set_o = set(res.idx[: res.count].tolist())
    set_g = set(kept.tolist())
    if set_g != set_o:
        assert scored, f"{where}: closed-form rule differs"
        if route == gen.SNAPKV:
            E, k = n - wl.W, b - wl.W
            keys = res.pooled[:E]
        else:
            r = wl.h2o_recent if wl.h2o_recent >= 0 else b // 2
            E, k = n - r, b - r
            keys = res.raw[:E]
        thr = np.sort(keys)[::-1][k - 1]
        for p in set_g ^ set_o:
            assert p < E, f"{where}: protected position {p} differs"
            assert abs(keys[p] - thr) <= REL * abs(thr), (
                f"{where}: position {p} key {keys[p]} not a near-tie of threshold {thr}")
        assert len([p for p in set_g if p < E]) == k
        if stats is not None:
            stats["near_tie_swaps"] = stats.get("near_tie_swaps", 0) + len(set_g - set_o)

    # ---- gathered rows ----
    Kg, Vg = gpu.out_rows(base, b)
    assert np.array_equal(Kg[:cnt_g], K_rows[kept]), f"{where}: gathered K rows differ"
    assert np.array_equal(Vg[:cnt_g], V_rows[kept]), f"{where}: gathered V rows differ"
    assert not Kg[cnt_g:].any() and not Vg[cnt_g:].any(), f"{where}: unused slots not zero"

    # ---- H2O state ----
    if route == gen.H2O:
        st = gpu.state[base: base + cnt_g].astype(np.float64)
        ref = res.raw[kept]
        tol = REL * np.maximum(np.abs(ref), FLOOR * res.raw.max())
        assert np.all(np.abs(st - ref) <= tol), f"{where}: H2O state off"


def run_gpu(wl, layers_dev, lens_np, plan=None, lse=None):
    """Run kvev_evict_prefill on device tensors {l: (K, V, Q)} (kvev_evict_prefill_lse
    with the per-layer window-row log-sum-exp `lse`); returns (plan, bufs)."""
    import torch
    from paper_2606_15157_gb300 import kvev
    if plan is None:
        plan = kvev.Plan.from_workload(wl)
    bufs = plan.buffers(wl.B, wl.S_cap)
    lens = torch.from_numpy(np.asarray(lens_np, np.int32)).cuda()
    K = [layers_dev[l][0] if l in layers_dev else None for l in range(wl.L)]
    V = [layers_dev[l][1] if l in layers_dev else None for l in range(wl.L)]
    Q = [layers_dev[l][2] if l in layers_dev else None for l in range(wl.L)]
    plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs, lse=lse)
    torch.cuda.synchronize()
    assert plan.status() == 0, "device status word set"
    return plan, bufs


def to_host_u16(t):
    import torch
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def check_workload(wl, layers_dev, lens_np, units=None, nthreads=0, stats=None, lse=None):
    """Run the GPU path on the whole workload and compare `units` (default: all)."""
    import oracle
    plan, bufs = run_gpu(wl, layers_dev, lens_np, lse=lse)
    gpu = GpuRun(plan, wl, bufs, lens_np)
    if units is None:
        units = [(l, s, h) for l in range(wl.L) for s in range(wl.B) for h in range(wl.H_kv)]
    # One oracle call per layer: the host copies of a layer's inputs are freed
    # before the next layer's (a full-size workload is tens of GB).
    by_layer = {}
    for u in units:
        by_layer.setdefault(u[0], []).append(u)
    for l in sorted(by_layer):
        specs, meta = [], []
        cache = {}
        for (_, s, h) in by_layer[l]:
            n = int(lens_np[s])
            if s not in cache:
                K, V, Q = layers_dev[l]
                cache[s] = (to_host_u16(K[s]), to_host_u16(V[s]),
                            None if Q is None else to_host_u16(Q[s]))
            Kh, Vh, Qh = cache[s]
            Qg = None if Qh is None else Qh[h * wl.G:(h + 1) * wl.G]
            spec = oracle_spec(wl, l, s, h, Kh[h][:max(n, 1)], Qg)
            spec["n"] = n
            if wl.route[l] == gen.FULL:
                spec["b"] = max(n, 1)
            specs.append(spec)
            meta.append((l, s, h, n, Kh[h], Vh[h]))
        results = oracle.evict_units(specs, d=wl.d, G=wl.G, nthreads=nthreads)
        for (_, s, h, n, Kr, Vr), res in zip(meta, results):
            check_unit(wl, l, s, h, n, res, gpu, Kr, Vr, stats)
        if stats is not None:
            stats["units_checked"] = stats.get("units_checked", 0) + len(meta)
    return plan, bufs, gpu
