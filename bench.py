#!/usr/bin/env python
"""Benchmark of the prefill eviction hot path on GB300.

One step = one kvev_evict_prefill() over the whole synthetic workload: window
scores of every SnapKV/H2O layer, selection, gather-compaction of every
layer of the heterogeneous route.  The default workload is the batch-8,
ragged 16K-32K-token, window-64 route of 32 LLaMA-3.1-8B-shaped layers
(18 SnapKV / 7 H2O / 7 StreamingLLM, Dirichlet capacity allocation summing to
1024 tokens per layer on average), whose inputs (about 34 GB of K/V) are far
larger than L2.

Usage:  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Under torchrun each rank runs its own batch (different seed): weak scaling,
no collective on the data path; rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2606_15157_gb300 import inputs as gen  # noqa: E402

METRIC = "KV-eviction GB/s and % of HBM peak (Llama-3.1-8B shape, 32K ctx)"
NOMINAL_HBM_GBS = 8000.0


# ---------------------------------------------------------------------------
# Workload accounting (algorithmic bytes, evicted tokens)
# ---------------------------------------------------------------------------

def unit_bytes(wl, l: int, n: int) -> tuple[int, int]:
    """(algorithmic bytes, score-kernel bytes) of one (sequence, layer, KV head).

    Scoring layer: all K read (n rows) + the group's window queries + kept K
    and V written; the score kernel's share is K read + window queries + the
    fp32 scores it writes.  StreamingLLM: kept K and V read and written.
    """
    row = wl.d * 2
    m = int(wl.route[l])
    b = int(wl.budget[l])
    if m in (gen.SNAPKV, gen.H2O):
        if m == gen.SNAPKV and n <= b:      # identity, no scoring
            return 4 * n * row, 0
        q = wl.G * wl.W * row
        return n * row + q + 2 * min(n, b) * row, n * row + q + 4 * n
    if m == gen.STREAMING:
        cap = wl.sink + (wl.recent if wl.recent >= 0 else b - wl.sink)
        return 4 * min(n, cap) * row, 0
    return 0, 0


def score_flops(wl) -> int:
    """Tensor-core work of the window-score kernel: Q_win K^T (2 R n d flops
    for R = G W rows and n keys) once per sweep, two sweeps per unit (the row
    normaliser needs every key before any score is final)."""
    tot = 0
    for l in range(wl.L):
        m, b = int(wl.route[l]), int(wl.budget[l])
        for s in range(wl.B):
            n = int(wl.lens[s])
            if m == gen.H2O or (m == gen.SNAPKV and n > b):
                tot += 2 * (2 * wl.G * wl.W * n * wl.d) * wl.H_kv
    return tot


def score_exp2(wl) -> int:
    """exp2 evaluations of the window-score kernel: one per (window row, key)
    in each sweep (sweep 1 for the row's running sum, sweep 2 for the key's
    normalised weight), i.e. two per multiply-add column of score_flops."""
    return score_flops(wl) // (2 * wl.d)


# MUFU exp2 rate of one SM: one warp instruction (32 lanes) per clock
MUFU_EX2_PER_CLK_SM = 32


def h2o_full_flops(wl) -> tuple[int, int]:
    """(algorithmic, performed) tensor-core flops of the scoring launches when
    H2O layers score every prompt row.  Algorithmic: each causal q.k product
    once (2 G d n(n+1)/2 per H2O unit, 2 G W n d per SnapKV unit).  Performed:
    the row pass (each block of Pb = 256 // G positions against the 256-key
    super-tiles up to its end) and the key pass (each 256-key super-tile
    against the blocks from the one holding its first key), 256 rows x 256
    keys x d per pair."""
    alg = perf = 0
    pb = max(1, 256 // wl.G)
    for l in range(wl.L):
        m, b = int(wl.route[l]), int(wl.budget[l])
        for s in range(wl.B):
            n = int(wl.lens[s])
            if m == gen.H2O and n > 0:
                alg += wl.G * wl.d * n * (n + 1) * wl.H_kv
                nb = (n + pb - 1) // pb
                pairs = sum((min(n, (q + 1) * pb) + 255) // 256 for q in range(nb))
                pairs += sum(nb - (256 * t) // pb for t in range((n + 255) // 256))
                perf += pairs * 2 * 256 * 256 * wl.d * wl.H_kv
            elif m == gen.SNAPKV and n > b:
                alg += 2 * wl.G * wl.W * n * wl.d * wl.H_kv
                perf += 2 * (2 * wl.G * wl.W * n * wl.d) * wl.H_kv
    return alg, perf


def workload_bytes(wl):
    """(algorithmic bytes, score-kernel bytes, evicted rows) of one step over
    the whole batch; evicted rows count every (sequence, layer, KV head)."""
    tot = sc = ev = 0
    for l in range(wl.L):
        for s in range(wl.B):
            n = int(wl.lens[s])
            a, c = unit_bytes(wl, l, n)
            tot += a * wl.H_kv
            sc += c * wl.H_kv
            if wl.route[l] != gen.FULL:
                ev += (n - min(n, int(wl.budget[l]))) * wl.H_kv
    return tot, sc, ev


def make_workload(name: str, seed: int, alloc, batch: int | None = None):
    if name == "long":
        wl = gen.config_long(alloc, seed=seed)
        if batch:  # first `batch` sequences of the same draw (small profiling case)
            wl.B, wl.lens = batch, wl.lens[:batch].copy()
            wl.name += f"_first{batch}"
        return wl
    if name == "long32k":
        return gen.config_long(alloc, seed=seed, fixed_len=32768)
    if name == "homog8k":
        return gen.config_homog8k(seed=seed)
    if name == "hetero8k":
        return gen.config_hetero8k(alloc, seed=seed, bbar=512)
    raise ValueError(name)


def workload_config(wl, extra=None):
    cfg = {
        "workload": wl.name,
        "layers": wl.L, "heads_q": wl.H_q, "heads_kv": wl.H_kv, "head_dim": wl.d,
        "batch": wl.B, "seq_lens": [int(x) for x in wl.lens], "window": wl.W,
        "pool": f"{'avg' if wl.pool_type == gen.POOL_AVG else 'max'}{wl.pool_kernel}",
        "route": {"snapkv": int((wl.route == gen.SNAPKV).sum()), "h2o": int((wl.route == gen.H2O).sum()),
                  "streaming": int((wl.route == gen.STREAMING).sum())},
        "budget_mean": float(np.mean(wl.budget)), "budget_total": int(np.sum(wl.budget)),
        "l2": "inputs larger than L2 (no flush needed)",
    }
    if extra:
        cfg.update(extra)
    return cfg


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (FileNotFoundError, OSError):
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        mhz, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                mhz.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        os.unlink(self.path)
        if not mhz:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(mhz)}


# ---------------------------------------------------------------------------
# CPU oracle on a bounded sample (CPU baseline and the reference arm)
# ---------------------------------------------------------------------------

def sample_units(wl, count: int, seed: int = 0):
    """A sample of (layer, seq, head) units with the route's operator mix."""
    rng = np.random.default_rng(seed)
    active = [l for l in range(wl.L) if wl.route[l] != gen.FULL]
    out = []
    for i in range(count):
        l = active[i % len(active)] if i < len(active) else int(rng.choice(active))
        out.append((l, int(rng.integers(wl.B)), int(rng.integers(wl.H_kv))))
    return out


def oracle_sample(wl, units, nthreads=0):
    """Time the oracle on `units` (inputs generated on the host); returns (seconds, bytes)."""
    import oracle
    oracle.build()
    specs, nbytes = [], 0
    for (l, s, h) in units:
        n = int(wl.lens[s])
        pos = np.arange(n, dtype=np.int64)
        K = gen.k_rows(wl, l, s, h, pos)
        Q = gen.q_group(wl, l, s, h) if wl.route[l] in (gen.SNAPKV, gen.H2O) else None
        specs.append(dict(method=int(wl.route[l]), n=n, b=int(wl.budget[l]), W=wl.W,
                          pool_kernel=wl.pool_kernel, pool_type=wl.pool_type, sink=wl.sink,
                          recent=wl.recent, h2o_recent=wl.h2o_recent, K=K, Q=Q))
        nbytes += unit_bytes(wl, l, n)[0]
    t0 = time.perf_counter()
    oracle.evict_units(specs, d=wl.d, G=wl.G, nthreads=nthreads)
    return time.perf_counter() - t0, nbytes


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# ---------------------------------------------------------------------------
# The two arms
# ---------------------------------------------------------------------------

def run_reference(args, rank, world):
    if rank != 0:
        return
    import oracle
    wl = make_workload(args.workload, 0, oracle.alloc_from_scores, args.batch)
    cores = cpu_cores()
    units = sample_units(wl, args.ref_units)
    for _ in range(args.warmup):
        oracle_sample(wl, units[: max(1, len(units) // 4)], cores)
    tot_s, tot_b = 0.0, 0
    for k in range(args.steps):
        s, b = oracle_sample(wl, sample_units(wl, args.ref_units, seed=k), cores)
        tot_s += s
        tot_b += b
    value = tot_b / tot_s / 1e9
    sample = f"{args.ref_units} (sequence, layer, KV-head) units of the workload per step, route mix kept"
    out = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_s / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; shapes of LLaMA-3.1-8B long-context workloads)",
        "config": workload_config(wl, {"sample": sample}),
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": min(cores, args.ref_units),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out), flush=True)


def _code_only(src: str) -> str:
    """C/C++ source without comments and whitespace (string literals kept)."""
    out, i, n = [], 0, len(src)
    while i < n:
        if src.startswith("//", i):
            i = src.find("\n", i)
            i = n if i < 0 else i
        elif src.startswith("/*", i):
            i = src.find("*/", i + 2)
            i = n if i < 0 else i + 2
        elif src[i] == '"':
            j = i + 1
            while j < n and src[j] != '"':
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        else:
            if not src[i].isspace():
                out.append(src[i])
            i += 1
    return "".join(out)


def kernel_hash() -> str:
    """Identity of the window-score kernel's code (comments and layout ignored):
    a stored DRAM-traffic measurement is used only while it matches."""
    h = hashlib.sha256()
    for f in ("score.cu", "score_common.cuh", "kvev_internal.cuh"):
        h.update(_code_only(open(os.path.join(ROOT, "paper_2606_15157_gb300", "csrc", f)).read()).encode())
    return h.hexdigest()[:16]


def rank_reducers(dist: bool, device: str):
    """(max over ranks, sum over ranks) of a host float: an all-reduce of one
    fp64 value on `device` (NCCL between GPU ranks, gloo on CPU); the identity
    for a single process."""
    if not dist:
        return (lambda x: x), (lambda x: x)
    import torch
    import torch.distributed as td

    def red(x: float, op) -> float:
        t = torch.tensor([float(x)], dtype=torch.float64, device=device)
        td.all_reduce(t, op=op)
        return float(t.item())

    return (lambda x: red(x, td.ReduceOp.MAX)), (lambda x: red(x, td.ReduceOp.SUM))


def time_prefill(plan, wl, K, V, Q, lens, bufs, stream, steps, barrier, kvev, lse=None):
    """Device time of `steps` back-to-back prefill evictions (inputs resident in
    HBM): (ms per step, per-kernel ms, clock summary, kernels launched).

    The steps are issued back to back: no host synchronisation falls inside the
    timed region.  The library records a CUDA event pair around each of its
    kernels on the launching stream in every step; the per-kernel times are
    those of the last timed step, read back after the region."""
    import torch
    kvev.kvev_plan_enable_timing(plan.handle, True)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device()) as clk:
        barrier()
        ev0.record(stream)
        for _ in range(steps):
            plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs, stream, lse=lse)
        ev1.record(stream)
        barrier()
    last = kvev.kvev_plan_last_timings(plan.handle)
    per_kernel = {k: (v if v >= 0 else None) for k, v in last.items()}
    # the supplied normalisers' fill kernel runs inside the prologue's event pair
    launched = (sum(1 for v in last.values() if v >= 0) + (1 if lse is not None else 0)) * steps
    return ev0.elapsed_time(ev1) / steps, per_kernel, clk.summary(), launched


def window_lse_device(wl, K, Q):
    """The normalisers a caller's own prefill attention returns: per SnapKV / H2O
    layer, fp32 [B][H_q][W] log-sum-exp of each window row over the keys it sees
    (plain fp32 torch on the device, outside any timed region)."""
    import torch
    tf32 = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    out = []
    scale = 1.0 / math.sqrt(wl.d)
    for l in range(wl.L):
        if wl.route[l] not in (gen.SNAPKV, gen.H2O) or Q[l] is None:
            out.append(None)
            continue
        lse = torch.zeros((wl.B, wl.H_q, wl.W), dtype=torch.float32, device="cuda")
        for s in range(wl.B):
            n = int(wl.lens[s])
            t = n - wl.W + torch.arange(wl.W, device="cuda")
            mask = torch.arange(n, device="cuda")[None, :] > t[:, None]  # [W][n]
            for h in range(wl.H_kv):
                q = Q[l][s, h * wl.G:(h + 1) * wl.G].float()              # [G][W][d]
                S = torch.matmul(q, K[l][s, h, :n].float().T) * scale     # [G][W][n]
                S.masked_fill_(mask[None], float("-inf"))
                lse[s, h * wl.G:(h + 1) * wl.G] = torch.logsumexp(S, dim=-1)
        out.append(lse)
    torch.backends.cuda.matmul.allow_tf32 = tf32
    torch.cuda.synchronize()
    return out


def prompt_lse_device(wl, K, Q, rows=1024):
    """Every prompt row's log-sum-exp for the H2O layers scored over the whole
    prompt (Q[l] is then [B][H_q][S_cap][d]): fp32 [B][H_q][S_cap], the layout
    a flash-attention prefill returns; plain fp32 torch, row blocks of `rows`."""
    import torch
    tf32 = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    scale = 1.0 / math.sqrt(wl.d)
    out = {}
    for l in range(wl.L):
        if wl.route[l] != gen.H2O:
            continue
        lse = torch.zeros((wl.B, wl.H_q, wl.S_cap), dtype=torch.float32, device="cuda")
        for s in range(wl.B):
            n = int(wl.lens[s])
            for h in range(wl.H_kv):
                k = K[l][s, h, :n].float()
                for t0 in range(0, n, rows):
                    t1 = min(n, t0 + rows)
                    q = Q[l][s, h * wl.G:(h + 1) * wl.G, t0:t1].float()        # [G][r][d]
                    S = torch.matmul(q, k[:t1].T) * scale                      # [G][r][t1]
                    t = torch.arange(t0, t1, device="cuda")
                    S.masked_fill_(torch.arange(t1, device="cuda")[None, :] > t[:, None], float("-inf"))
                    lse[s, h * wl.G:(h + 1) * wl.G, t0:t1] = torch.logsumexp(S, dim=-1)
        out[l] = lse
    torch.backends.cuda.matmul.allow_tf32 = tf32
    torch.cuda.synchronize()
    return out


def cudart():
    """The CUDA runtime that torch loaded (the same library instance, so torch's
    stream handles are valid in calls made through it)."""
    paths = []
    try:
        paths = [ln.split()[-1] for ln in open("/proc/self/maps") if "libcudart.so" in ln]
    except OSError:
        pass
    lib = ctypes.CDLL(paths[0] if paths else "libcudart.so")
    vp, sz = ctypes.c_void_p, ctypes.c_size_t
    lib.cudaMemcpy2DAsync.argtypes = [vp, sz, vp, sz, sz, sz, ctypes.c_int, vp]
    lib.cudaMemcpy2DAsync.restype = ctypes.c_int
    return lib


def host_link_peak(nbytes: int = 2 << 30, reps: int = 5) -> dict:
    """Host -> device copy rate of one large pinned buffer (cudaMemcpyAsync)."""
    import torch
    h = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    d = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    d.copy_(h, non_blocking=True)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        d.copy_(h, non_blocking=True)
    e1.record()
    torch.cuda.synchronize()
    gbs = reps * nbytes / (e0.elapsed_time(e1) / 1e3) / 1e9
    del h, d
    return {"h2d_gbs": gbs, "how": f"one pinned {nbytes >> 30} GiB host buffer copied to the device, "
                                   f"{reps} times, CUDA events"}


def run_ours(args, rank, world, local_rank):
    import torch
    from paper_2606_15157_gb300 import kvev

    torch.cuda.set_device(local_rank)
    dist = world > 1
    if dist:
        import torch.distributed as td

    wl = make_workload(args.workload, rank, kvev.alloc_from_scores, args.batch)
    tot_bytes, score_bytes, evicted = workload_bytes(wl)
    need_q = lambda l: wl.route[l] in (gen.SNAPKV, gen.H2O)
    dev = {l: gen.device_layer(wl, l, need_q=need_q(l)) for l in range(wl.L)}
    plan = kvev.Plan.from_workload(wl)
    if args.h2o_full_prompt:
        plan.set_h2o_full_prompt(True)  # before sizing the workspace: it holds every row's lse
    bufs = plan.buffers(wl.B, wl.S_cap)
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    K = [dev[l][0] for l in range(wl.L)]
    V = [dev[l][1] for l in range(wl.L)]
    Q = [dev[l][2] for l in range(wl.L)]
    if args.h2o_full_prompt:
        # H2O layers score every prompt row: their queries are the whole
        # prompt's, seeded normal bf16 [B][H_q][S_cap][d]
        g = torch.Generator(device="cuda")
        g.manual_seed(4242 + rank)
        for l in range(wl.L):
            if wl.route[l] == gen.H2O:
                Q[l] = torch.randn((wl.B, wl.H_q, wl.S_cap, wl.d), generator=g, device="cuda",
                                   dtype=torch.float32).to(torch.bfloat16)
        args.no_e2e = args.no_cpu_baseline = True
    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()

    def barrier():
        if dist:
            td.barrier()
        torch.cuda.synchronize()

    max_over_ranks, sum_over_ranks = rank_reducers(dist, "cuda")

    # ---- device-resident timed region ----
    main_lse = None
    if args.lse_supplied:  # the fused form's own line: no end-to-end or CPU arms
        if args.h2o_full_prompt:  # the window kernel's layers (SnapKV) need only the window rows
            Q_win_snap = [Q[l] if wl.route[l] == gen.SNAPKV else None for l in range(wl.L)]
            main_lse = [None] * wl.L
            for l, x in enumerate(window_lse_device(wl, K, Q_win_snap)):
                if wl.route[l] == gen.SNAPKV:
                    main_lse[l] = x
            for l, x in prompt_lse_device(wl, K, Q).items():
                main_lse[l] = x
        else:
            main_lse = window_lse_device(wl, K, Q)
        args.no_e2e = args.no_cpu_baseline = True
    kvev.kvev_plan_enable_timing(plan.handle, True)
    for _ in range(args.warmup):
        plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs, stream, lse=main_lse)
    barrier()
    ms_local, kernel_ms, clocks, kernels_launched = time_prefill(plan, wl, K, V, Q, lens, bufs, stream,
                                                                  args.steps, barrier, kvev, lse=main_lse)
    ms_step = max_over_ranks(ms_local)
    status = plan.status()
    assert status == kvev.OK, f"device status {status}"
    all_bytes = sum_over_ranks(float(tot_bytes))
    all_evicted = sum_over_ranks(float(evicted))
    value = all_bytes / (ms_step / 1e3) / 1e9

    # ---- roofline of the dominant kernel (window scores) ----
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        pass
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    peak_src = "measured" if "hbm_gbs" in peaks else "fallback"
    score_ms = kernel_ms["score"] if kernel_ms["score"] is not None else float("nan")
    achieved = score_bytes / (score_ms / 1e3) / 1e9
    tc_peak = float(peaks.get("bf16_tflops", 1900.0))
    tc_achieved = score_flops(wl) / (score_ms / 1e3) / 1e12
    # MUFU: peak from the unit count and the SM clock sampled under load
    n_sms = torch.cuda.get_device_properties(local_rank).multi_processor_count
    mhz = clocks.get("sm_mhz") or clocks.get("sm_max_mhz") or 2070.0
    mufu_peak = MUFU_EX2_PER_CLK_SM * n_sms * mhz * 1e6 / 1e9
    mufu_achieved = score_exp2(wl) / (score_ms / 1e3) / 1e9
    traffic = None
    traffic_single = None  # the one-sweep form (window normalisers supplied)
    tf = os.path.join(ROOT, "profiles", "score_traffic.json")
    if os.path.exists(tf):
        try:
            t = json.load(open(tf))
            if t.get("workload") == wl.name and t.get("kernel_src_hash") == kernel_hash():
                traffic = t["bytes_per_launch"]
                traffic_single = t.get("single_sweep", {}).get("bytes_per_launch")
        except (OSError, ValueError, KeyError):
            pass
    if args.lse_supplied:
        traffic = traffic_single

    # ---- end to end through the C ABI with host buffers ----
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, wl, plan, dev, lens, stream, tot_bytes, barrier, max_over_ranks,
                      sum_over_ranks)

    # ---- CPU baseline (rank 0, one GPU only) ----
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cores = cpu_cores()
        # one unit per core and call: the oracle runs its units in parallel, one per thread
        units, secs, nb, i = [], 0.0, 0, 0
        while secs < args.cpu_seconds and i < 4096:
            batch = sample_units(wl, cores, seed=100 + i)
            s, b = oracle_sample(wl, batch, cores)
            units += batch
            secs += s
            nb += b
            i += 1
        cpu = {"value": nb / secs / 1e9, "unit": "GB/s", "cores": cores, "kind": "oracle",
               "sample": f"{len(units)} (sequence, layer, KV-head) units of the workload, "
                         f"route mix kept, {secs:.1f} s of oracle time"}

    # ---- sustained: the same step over at least 0.5 s of device time ----
    sustained = None
    if not args.no_extras and not args.h2o_full_prompt:
        n_s = max(args.steps, int(np.ceil(500.0 / max(ms_step, 1e-3))))
        ms_s, _, clk_s, _ = time_prefill(plan, wl, K, V, Q, lens, bufs, stream, n_s, barrier, kvev,
                                         lse=main_lse)
        ms_s = max_over_ranks(ms_s)
        assert plan.status() == kvev.OK
        sustained = {"value": all_bytes / (ms_s / 1e3) / 1e9, "unit": "GB/s", "ms_per_step": ms_s,
                     "steps": n_s, "device_seconds": n_s * ms_s / 1e3, "clocks": clk_s}

    extras = {}
    if not args.no_extras and not args.h2o_full_prompt and not args.lse_supplied:
        # the fused form: the window rows' normalisers come from the caller's own
        # prefill attention (kvev_evict_prefill_lse); one sweep over K
        lse = window_lse_device(wl, K, Q)
        for _ in range(args.warmup):
            plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs, stream, lse=lse)
        barrier()
        n_l = min(args.steps, 20)
        ms_l, kms_l, clk_l, _ = time_prefill(plan, wl, K, V, Q, lens, bufs, stream, n_l, barrier, kvev,
                                             lse=lse)
        ms_l = max_over_ranks(ms_l)
        assert plan.status() == kvev.OK
        ach_l = score_bytes / (kms_l["score"] / 1e3) / 1e9 if kms_l.get("score") else None
        val_l = all_bytes / (ms_l / 1e3) / 1e9
        extras["lse_supplied"] = {
            "value": val_l, "unit": "GB/s", "ms_per_step": ms_l, "steps": n_l,
            "hbm_frac": {"of_measured": val_l / hbm_peak, "of_nominal_8TBs": val_l / NOMINAL_HBM_GBS},
            "kernel_ms": kms_l,
            "roofline": {"kernel": "score_kernel (one sweep)", "bound": "hbm", "achieved": ach_l,
                         "peak": hbm_peak, "unit": "GB/s", "frac": None if ach_l is None else ach_l / hbm_peak,
                         "traffic": traffic_single},
            "clocks": clk_l,
            "how": "kvev_evict_prefill_lse: the window rows' log-sum-exp supplied (as a caller's prefill "
                   "attention returns it; computed once, untimed), the score kernel makes one sweep"}
        del lse
    if not args.no_extras and not args.h2o_full_prompt and args.workload == "long" and not args.batch:
        del dev, K, V, Q, bufs
        plan.close()
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        extras["long32k"] = fixed_length_variant(args, rank, kvev, barrier, max_over_ranks, sum_over_ranks)
        torch.cuda.empty_cache()
        extras["decode"] = decode_measure(args, rank, world, local_rank, B=16, steps=max(args.steps, 50),
                                          warmup=args.warmup, attn_supplied=False)
        torch.cuda.empty_cache()
    if not args.no_extras and not args.h2o_full_prompt:
        extras["host_link"] = host_link_peak()
        if e2e is not None:
            link = e2e["h2d_bytes_per_step"] / (e2e["ms_per_step"] / 1e3) / 1e9
            e2e["host_link_gbs"] = link
            e2e["host_link_frac"] = link / extras["host_link"]["h2d_gbs"]

    if rank == 0 and args.h2o_full_prompt:
        alg, perf = h2o_full_flops(wl)
        tc_ach = alg / (score_ms / 1e3) / 1e12
        out = {
            "metric": "H2O full-prompt prefill eviction: causal attention TFLOP/s of the step",
            "value": sum_over_ranks(alg) / (ms_step / 1e3) / 1e12, "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded; full-prompt queries drawn N(0,1) on the device)",
            "config": workload_config(wl, {"h2o_full_prompt": True, "query_block": max(1, 256 // wl.G)}),
            "kernel_ms": kernel_ms,
            "roofline": {"kernel": "h2o_full_kernel row + key passes (and the window kernel)", "bound": "tensor",
                         "achieved": tc_ach, "peak": tc_peak, "unit": "TFLOP/s", "frac": tc_ach / tc_peak,
                         "traffic": None, "peak_source": "measured" if "bf16_tflops" in peaks else "fallback",
                         "tensor_pipe": {"achieved": perf / (score_ms / 1e3) / 1e12, "peak": tc_peak,
                                         "unit": "TFLOP/s",
                                         "frac": perf / (score_ms / 1e3) / 1e12 / tc_peak,
                                         "work": "row pass + key pass, 256 x 256 tiles"}},
            "clocks": clocks,
            # prologue, window scores, row pass (or, with --lse-supplied, the two normaliser fills
            # instead), key pass, select, gather
            "gpu_launches": args.steps * (7 if args.lse_supplied else 6),
            "e2e": None, "cpu_baseline": None,
        }
        print(json.dumps(out), flush=True)
    elif rank == 0:
        out = {
            "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded; shapes of LLaMA-3.1-8B long-context workloads)",
            "config": workload_config(wl, {"parallelism": f"independent batch per GPU x{world}",
                                           **({"lse_supplied": True} if args.lse_supplied else {})}),
            "hbm_frac": {"of_measured": value / hbm_peak, "of_nominal_8TBs": value / NOMINAL_HBM_GBS},
            # tokens dropped from a layer's cache, counted once per (sequence,
            # layer) and once per (sequence, layer, KV head): every head keeps
            # b_l of the n positions, each its own choice
            "evicted_tokens_per_s": all_evicted / wl.H_kv / (ms_step / 1e3),
            "evicted_rows_per_s": all_evicted / (ms_step / 1e3),
            "kernel_ms": kernel_ms,
            "roofline": {"kernel": "score_kernel", "bound": "hbm", "achieved": achieved,
                         "peak": hbm_peak, "unit": "GB/s", "frac": achieved / hbm_peak,
                         "traffic": traffic, "peak_source": peak_src,
                         "tensor_pipe": {"achieved": tc_achieved, "peak": tc_peak, "unit": "TFLOP/s",
                                         "frac": tc_achieved / tc_peak,
                                         "work": "two sweeps of Q_win K^T (bf16 in, fp32 accumulate)",
                                         "peak_source": "measured" if "bf16_tflops" in peaks
                                         else "fallback"},
                         "mufu": {"achieved": mufu_achieved, "peak": mufu_peak, "unit": "Gexp2/s",
                                  "frac": mufu_achieved / mufu_peak,
                                  "work": "one exp2 per (window row, key) in each of the two sweeps",
                                  "peak_source": f"{MUFU_EX2_PER_CLK_SM} exp2/clock/SM x {n_sms} SMs x "
                                                 f"{mhz:.0f} MHz (median SM clock under load)"}},
            "clocks": clocks,
            "gpu_launches": kernels_launched,
            "e2e": e2e,
            "cpu_baseline": cpu,
            "sustained": sustained,
        }
        out.update(extras)
        print(json.dumps(out), flush=True)


def fixed_length_variant(args, rank, kvev, barrier, max_over_ranks, sum_over_ranks):
    """The headline's fixed-length variant: batch 8, every sequence 32,768
    tokens, same route and allocation; device-resident inputs, same timing."""
    import torch
    wl = make_workload("long32k", rank, kvev.alloc_from_scores)
    tot_bytes, score_bytes, evicted = workload_bytes(wl)
    need_q = lambda l: wl.route[l] in (gen.SNAPKV, gen.H2O)
    dev = {l: gen.device_layer(wl, l, need_q=need_q(l)) for l in range(wl.L)}
    plan = kvev.Plan.from_workload(wl)
    bufs = plan.buffers(wl.B, wl.S_cap)
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    K = [dev[l][0] for l in range(wl.L)]
    V = [dev[l][1] for l in range(wl.L)]
    Q = [dev[l][2] for l in range(wl.L)]
    stream = torch.cuda.current_stream()
    kvev.kvev_plan_enable_timing(plan.handle, True)
    for _ in range(args.warmup):
        plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs, stream)
    barrier()
    steps = max(10, min(args.steps, 40))
    ms, kms, clk, _ = time_prefill(plan, wl, K, V, Q, lens, bufs, stream, steps, barrier, kvev)
    ms = max_over_ranks(ms)
    assert plan.status() == kvev.OK
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        pass
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    value = sum_over_ranks(float(tot_bytes)) / (ms / 1e3) / 1e9
    ach = score_bytes / (kms["score"] / 1e3) / 1e9
    out = {"workload": wl.name, "value": value, "unit": "GB/s", "ms_per_step": ms, "steps": steps,
           "hbm_frac": {"of_measured": value / hbm_peak, "of_nominal_8TBs": value / NOMINAL_HBM_GBS},
           "evicted_tokens_per_s": sum_over_ranks(float(evicted)) / wl.H_kv / (ms / 1e3),
           "kernel_ms": kms,
           "roofline": {"kernel": "score_kernel", "bound": "hbm", "achieved": ach, "peak": hbm_peak,
                        "unit": "GB/s", "frac": ach / hbm_peak, "traffic": None},
           "clocks": clk}
    del dev, K, V, Q, bufs
    plan.close()
    torch.cuda.synchronize()
    return out


def run_e2e(args, wl, plan, dev, lens_dev, stream, tot_bytes, barrier, max_over_ranks,
            sum_over_ranks):
    """Same metric through the public API, starting every step from pinned host
    memory: the inputs the tensor-core path streams (the prompt rows of K and
    Q_win of the SnapKV / H2O layers) are copied to the device on four copy
    streams, and the tensors that are only gathered row by row (V of every
    layer, K of the StreamingLLM layers) stay in pinned host memory, read in
    place over the host link by the gather kernel (by the selection kernel for
    the StreamingLLM layers); the kept indices and counts
    are read back.  Steps alternate between two device copies of the streamed
    inputs, so a step's uploads overlap the previous step's eviction (each step
    still uploads its own inputs and reads back its own result).  The bytes
    that cross the host link either way are counted in h2d_bytes_per_step."""
    import torch
    from paper_2606_15157_gb300 import kvev
    scoring = [int(wl.route[l]) in (gen.SNAPKV, gen.H2O) for l in range(wl.L)]
    pinned = lambda t: None if t is None else torch.empty(t.shape, dtype=t.dtype, pin_memory=True).copy_(t)
    rt = cudart()
    H2D = 1  # cudaMemcpyHostToDevice
    V_arg = []
    K_set, Q_set, copy_set = [[], []], [[], []], [[], []]
    for l in range(wl.L):
        Kd, Vd, Qd = dev[l]
        Kh, Vh, Qh = pinned(Kd), pinned(Vd), pinned(Qd)
        V_arg.append(Vh)
        for b in range(2):
            if scoring[l]:
                Kb = Kd if b == 0 else torch.empty_like(Kd)
                Qb = Qd if b == 0 else torch.empty_like(Qd)
                K_set[b].append(Kb)
                Q_set[b].append(Qb)
                # the prompt rows of a sequence's KV heads: H_kv blocks of n rows,
                # S_cap rows apart in [B][H_kv][S_cap][d], as one 2-D copy (rows
                # past a sequence's length are never read)
                pitch = wl.S_cap * wl.d * Kh.element_size()
                for s in range(wl.B):
                    n = int(wl.lens[s])
                    if n > 0:
                        copy_set[b].append(("2d", Kb[s].data_ptr(), Kh[s].data_ptr(), pitch,
                                            n * wl.d * Kh.element_size(), wl.H_kv))
                copy_set[b].append(("1d", Qh, Qb))
            else:
                K_set[b].append(Kh)
                Q_set[b].append(None)
    lens_h = torch.from_numpy(np.asarray(wl.lens, np.int32)).pin_memory()
    bufs = plan.buffers(wl.B, wl.S_cap)
    idx_h = torch.empty(bufs["out_idx"].shape, dtype=torch.int32, pin_memory=True)
    cnt_h = torch.empty(bufs["out_count"].shape, dtype=torch.int32, pin_memory=True)
    copied = sum(c[4] * c[5] if c[0] == "2d" else c[1].numel() * c[1].element_size()
                 for c in copy_set[0]) + lens_h.numel() * 4
    d2h = idx_h.numel() * 4 + cnt_h.numel() * 4
    copy_streams = [torch.cuda.Stream() for _ in range(4)]
    released = [torch.cuda.Event(), torch.cuda.Event()]  # last eviction that read input set b is done
    for ev in released:
        ev.record(stream)
    step_no = [0]

    def step():
        b = step_no[0] & 1
        step_no[0] += 1
        evs = []
        for i, cs in enumerate(copy_streams):
            cs.wait_event(released[b])
            with torch.cuda.stream(cs):
                for c in copy_set[b][i::len(copy_streams)]:
                    if c[0] == "2d":
                        _, dst, src, pitch, width, height = c
                        rc = rt.cudaMemcpy2DAsync(dst, pitch, src, pitch, width, height, H2D, cs.cuda_stream)
                        assert rc == 0, f"cudaMemcpy2DAsync failed ({rc})"
                    else:
                        c[2].copy_(c[1], non_blocking=True)
            ev = torch.cuda.Event()
            ev.record(cs)
            evs.append(ev)
        for ev in evs:
            stream.wait_event(ev)
        with torch.cuda.stream(stream):
            lens_dev.copy_(lens_h, non_blocking=True)
        plan.evict_prefill(K_set[b], V_arg, Q_set[b], lens_dev, wl.B, wl.S_cap, bufs, stream)
        released[b].record(stream)
        with torch.cuda.stream(stream):
            idx_h.copy_(bufs["out_idx"], non_blocking=True)
            cnt_h.copy_(bufs["out_count"], non_blocking=True)

    kvev.kvev_plan_enable_timing(plan.handle, False)
    for _ in range(args.warmup):
        step()
    stream.synchronize()
    # rows read in place from host memory: every kept row of V, and
    # of K for the layers whose K stays on the host (FULL layers keep nothing)
    row = wl.d * 2
    counts = cnt_h.numpy().reshape(wl.L, -1)
    host_read = 0
    for l in range(wl.L):
        if int(wl.route[l]) == gen.FULL:
            continue
        kept = int(counts[l].sum())
        host_read += kept * row * (1 if scoring[l] else 2)
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n = args.e2e_steps
    for cs in copy_streams:  # the timed region starts with every stream idle
        cs.synchronize()
    e0.record(stream)
    for cs in copy_streams:
        cs.wait_event(e0)
    for _ in range(n):
        step()
    e1.record(stream)
    barrier()
    ms = max_over_ranks(e0.elapsed_time(e1) / n)
    return {"value": sum_over_ranks(float(tot_bytes)) / (ms / 1e3) / 1e9, "unit": "GB/s",
            "h2d_bytes_per_step": int(copied + host_read), "d2h_bytes_per_step": int(d2h),
            "ms_per_step": ms, "steps": n,
            "host_resident": "V of every layer and K of the StreamingLLM layers, read in place",
            "copies_per_step": len(copy_set[0]) + 3,
            "pipelining": "two device copies of the streamed inputs; uploads overlap the previous step"}


def decode_step_bytes(wl, counts, supplied_attention=False):
    """Algorithmic bytes of one decode step: for H2O/TOVA units the retained K rows,
    the new token's k/q, the slots' positions and acc (read and written), or with
    the attention supplied by the caller that attention row (4 B per slot) instead
    of K and q; for every unit the new K/V row written (and StreamingLLM's
    position scan)."""
    row = wl.d * 2
    tot = 0
    for l in range(wl.L):
        md = int(wl.route_decode[l])
        c = counts[l]
        units = wl.B * wl.H_kv
        if md in (gen.H2O, gen.TOVA) and supplied_attention:
            tot += units * (4 * (c + 1) + c * 12 + row + 2 * row)
        elif md in (gen.H2O, gen.TOVA):
            tot += units * (c * row + c * 12 + row * (1 + wl.G) + 2 * row)
        elif md == gen.STREAMING:
            tot += units * (c * 4 + 2 * row)
        elif wl.route[l] != gen.FULL:
            tot += units * 2 * row
    return tot


def run_decode(args, rank, world, local_rank):
    """Decode workload: batch 16, 16K-token caches compacted to 2048 slots by the
    prefill eviction (not timed), then one kvev_decode_step per generated token."""
    out = decode_measure(args, rank, world, local_rank, B=args.batch or 16, steps=args.steps,
                         warmup=args.warmup, attn_supplied=args.decode_attn)
    if rank == 0:
        print(json.dumps(out), flush=True)


def decode_measure(args, rank, world, local_rank, B, steps, warmup, attn_supplied):
    """The decode step's JSON record (see run_decode)."""
    import torch
    from paper_2606_15157_gb300 import kvev

    torch.cuda.set_device(local_rank)
    dist = world > 1
    if dist:
        import torch.distributed as td
    wl = gen.config_decode(seed=rank, B=B)
    total = warmup + steps
    growth = total
    plan = kvev.Plan.from_workload(wl)
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    bufs = plan.buffers(wl.B, wl.S_cap)
    need_q = lambda l: wl.route[l] in (gen.SNAPKV, gen.H2O)
    dev = {l: gen.device_layer(wl, l, need_q=need_q(l)) for l in range(wl.L)}
    plan.evict_prefill([dev[l][0] for l in range(wl.L)], [dev[l][1] for l in range(wl.L)],
                       [dev[l][2] for l in range(wl.L)], lens, wl.B, wl.S_cap, bufs)
    torch.cuda.synchronize()
    del dev
    arena = kvev.DecodeArena(plan, wl.B, growth)
    arena.init_from_prefill(bufs, lens)
    # every step's new tokens, resident in HBM before the timed region
    toks = [[gen.device_decode_tokens(wl, t, l) for l in range(wl.L)] for t in range(total)]
    torch.cuda.synchronize()
    counts = [int(wl.budget[l]) for l in range(wl.L)]
    step_bytes = decode_step_bytes(wl, counts, attn_supplied)
    stream = torch.cuda.current_stream()
    attn = None
    if attn_supplied:
        # the caller's decode attention would supply these every step; any valid
        # rows cost the same, so one seeded set of distributions is reused
        g = torch.Generator(device="cuda")
        g.manual_seed(77 + rank)
        attn = []
        for l, (_, cap, _) in enumerate(arena.layers):
            if cap > 0 and int(wl.route_decode[l]) in (gen.H2O, gen.TOVA):
                a = torch.rand((wl.B, wl.H_kv, cap + 1), generator=g, device="cuda")
                attn.append(a / a.sum(dim=2, keepdim=True))
            else:
                attn.append(None)

    def run(t):
        k = [x[0] for x in toks[t]]
        v = [x[1] for x in toks[t]]
        if attn is not None:
            arena.step_attn(k, v, attn, stream)
            return
        q = [x[2] for x in toks[t]]
        arena.step(k, v, q, stream)

    for t in range(warmup):
        run(t)
    if dist:
        td.barrier()
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    with ClockSampler(local_rank) as clk:
        if dist:
            td.barrier()
        torch.cuda.synchronize()
        evs[0].record(stream)
        for i in range(steps):
            run(warmup + i)
            evs[i + 1].record(stream)
        torch.cuda.synchronize()
        if dist:
            td.barrier()
    per = [evs[i].elapsed_time(evs[i + 1]) for i in range(steps)]
    ms = evs[0].elapsed_time(evs[-1]) / steps
    max_over_ranks, sum_over_ranks = rank_reducers(dist, "cuda")
    ms = max_over_ranks(ms)
    all_bytes = sum_over_ranks(float(step_bytes))
    assert plan.status() == kvev.OK
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        pass
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    value = all_bytes / (ms / 1e3) / 1e9
    achieved = step_bytes / (statistics.median(per) / 1e3) / 1e9
    del toks, arena, bufs
    plan.close()
    torch.cuda.synchronize()
    if True:
        out = {
            "metric": "KV decode-step GB/s (retained-cache update per generated token)",
            "value": value, "unit": "GB/s", "n_gpus": world, "steps": steps,
            "warmup": warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded; shapes of LLaMA-3.1-8B decode with compacted caches)",
            "config": {"workload": wl.name, "layers": wl.L, "batch": wl.B, "cache_slots": 2048,
                       "attention": "supplied by the caller (kvev_decode_step_attn)" if attn_supplied
                       else "computed from q_new and the retained K",
                       "route_decode": {"h2o": int((wl.route_decode == gen.H2O).sum()),
                                        "streaming": int((wl.route_decode == gen.STREAMING).sum()),
                                        "append": int(((wl.route_decode == gen.FULL) &
                                                       (wl.route != gen.FULL)).sum())},
                       "l2": "retained K of the H2O layers (470 MB) larger than L2",
                       "parallelism": f"independent batch per GPU x{world}"},
            "tokens_per_s": world * wl.B / (ms / 1e3),
            "roofline": {"kernel": "decode_step_kernel", "bound": "hbm", "achieved": achieved,
                         "peak": hbm_peak, "unit": "GB/s", "frac": achieved / hbm_peak,
                         "traffic": None},
            "clocks": clk.summary(),
            "gpu_launches": steps,  # one decode_step_kernel per token (it also advances lens)
            "e2e": None, "cpu_baseline": None,
        }
    return out


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="long",
                    choices=["long", "long32k", "homog8k", "hetero8k", "decode"])
    ap.add_argument("--batch", type=int, default=None,
                    help="use only the first B sequences of the 'long' workload, or B sequences "
                         "in the decode workload (profiling)")
    ap.add_argument("--h2o-full-prompt", action="store_true",
                    help="H2O layers score every prompt query row (reports causal-attention TFLOP/s)")
    ap.add_argument("--lse-supplied", action="store_true",
                    help="the window rows' log-sum-exp is supplied (kvev_evict_prefill_lse): one score sweep")
    ap.add_argument("--decode-attn", action="store_true",
                    help="decode workload: the caller supplies the attention (kvev_decode_step_attn)")
    ap.add_argument("--e2e-steps", type=int, default=8)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--ref-units", type=int, default=16)
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the sustained run, the fixed-32K variant, the decode step and the "
                         "host-link peak (profiling runs)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1 and args.impl == "ours":
        import torch
        import torch.distributed as td
        torch.cuda.set_device(local_rank)
        td.init_process_group("nccl")
    if args.impl == "reference":
        run_reference(args, rank, world)
    elif args.workload == "decode":
        run_decode(args, rank, world, local_rank)
    else:
        run_ours(args, rank, world, local_rank)
    if world > 1 and args.impl == "ours":
        import torch.distributed as td
        td.destroy_process_group()


if __name__ == "__main__":
    main()
