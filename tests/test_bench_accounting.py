"""Host-side accounting of bench.py, on CPU.

The benchmark divides algorithmic bytes, tensor-core flops and evicted tokens
by its device time.  These tests write those counts out again from their
per-(sequence, layer) definitions and check the workloads' shapes.
  - Scoring layer (SnapKV, H2O): all of K read, the window queries read, and
    the kept K and V written.  That is 2 d H_kv bytes per key,
    2 d H_q bytes per window row and 4 d H_kv bytes per kept row.
  - StreamingLLM layer: the kept K and V read and written.
  - A layer whose budget covers the sequence: every row of K and V read and
    written.
  - Flops: Q_win K^T over the whole group, 2 W H_q n d per sweep, two sweeps,
    on every layer that scores; one exp2 per (window row, key) per sweep.
The reference arm (the oracle on the host cores) is run briefly in a
subprocess: its JSON line, and silence on ranks other than 0.
"""
import numpy as np

import bench
import oracle
from paper_2606_15157_gb300 import inputs as gen


def _layer_bytes(wl, l, n):
    b = int(wl.budget[l])
    m = int(wl.route[l])
    if m == gen.SNAPKV and n <= b:
        return 8 * wl.d * wl.H_kv * n
    if m in (gen.SNAPKV, gen.H2O):
        return 2 * wl.d * wl.H_kv * n + 2 * wl.d * wl.H_q * wl.W + 4 * wl.d * wl.H_kv * min(n, b)
    if m == gen.STREAMING:
        return 8 * wl.d * wl.H_kv * min(n, b)
    return 0


def test_headline_workload_shape():
    wl = bench.make_workload("long", 0, oracle.alloc_from_scores)
    assert (wl.L, wl.H_q, wl.H_kv, wl.d, wl.B, wl.W) == (32, 32, 8, 128, 8, 64)
    assert wl.pool_type == gen.POOL_AVG and wl.pool_kernel == 7
    assert np.all((wl.lens >= 16384) & (wl.lens <= 32768))
    route = list(wl.route)
    assert (route.count(gen.SNAPKV), route.count(gen.H2O), route.count(gen.STREAMING)) == (18, 7, 7)
    # each method's layers form one contiguous block
    changes = sum(1 for a, b in zip(route, route[1:]) if a != b)
    assert changes == 2
    assert int(np.sum(wl.budget)) == 32 * 1024
    assert int(np.min(wl.budget)) >= max(48, wl.W + 16)


def test_bytes_flops_and_evicted_follow_the_definitions():
    wl = bench.make_workload("long", 1, oracle.alloc_from_scores)
    tot, _, evicted_rows = bench.workload_bytes(wl)
    exp_bytes = sum(_layer_bytes(wl, l, int(n)) for l in range(wl.L) for n in wl.lens)
    assert tot == exp_bytes
    evicted = sum(int(n) - min(int(n), int(wl.budget[l])) for l in range(wl.L) for n in wl.lens
                  if wl.route[l] != gen.FULL)
    assert evicted_rows == wl.H_kv * evicted
    flops = sum(2 * 2 * wl.W * wl.H_q * int(n) * wl.d for l in range(wl.L) for n in wl.lens
                if wl.route[l] == gen.H2O or (wl.route[l] == gen.SNAPKV and n > wl.budget[l]))
    assert bench.score_flops(wl) == flops
    exp2 = sum(2 * wl.G * wl.W * int(n) * wl.H_kv for l in range(wl.L) for n in wl.lens
               if wl.route[l] == gen.H2O or (wl.route[l] == gen.SNAPKV and n > wl.budget[l]))
    assert bench.score_exp2(wl) == exp2


def test_identity_layers_count_every_row():
    # a SnapKV layer whose budget covers the sequence keeps every row: no
    # scoring, every row of K and V read and written; one key more and it scores
    wl = bench.make_workload("hetero8k", 0, oracle.alloc_from_scores)
    for l in range(wl.L):
        if wl.route[l] == gen.SNAPKV:
            n = int(wl.budget[l])
            a, c = bench.unit_bytes(wl, l, n)
            assert a * wl.H_kv == 8 * wl.d * wl.H_kv * n and c == 0
            a, c = bench.unit_bytes(wl, l, n + 1)
            assert a * wl.H_kv == _layer_bytes(wl, l, n + 1) and c > 0


def _run_bench(args, env_extra):
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, **env_extra)
    p = subprocess.run([sys.executable, os.path.join(root, "bench.py")] + args, cwd=root, env=env,
                       capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [ln for ln in p.stdout.splitlines() if ln.startswith("{")]
    return [json.loads(ln) for ln in lines]


def test_reference_arm_prints_the_contract_line():
    # the reference arm is the oracle on the host cores: one JSON line with the
    # ours-arm metric, unit and direction, a cpu_baseline record and a zero-copy e2e
    out = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "3", "--ref-units", "2"], {})
    assert len(out) == 1
    r = out[0]
    assert r["impl"] == "reference" and r["metric"] == bench.METRIC and r["unit"] == "GB/s"
    assert r["higher_is_better"] is True and r["value"] > 0 and r["steps"] == 1 and r["warmup"] == 3
    assert r["cpu_baseline"]["kind"] == "oracle" and r["cpu_baseline"]["cores"] >= 1
    assert r["cpu_baseline"]["value"] == r["value"]
    assert r["e2e"] == {"value": r["value"], "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert r["config"]["workload"] == "long_b8_16k-32k"


def test_reference_arm_other_ranks_do_no_work():
    # under torchrun only rank 0 runs the oracle and prints; the others exit 0
    out = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "3", "--ref-units", "2"],
                     {"WORLD_SIZE": "2", "RANK": "1", "LOCAL_RANK": "1"})
    assert out == []
