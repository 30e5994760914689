"""GPU parity: the CUDA path through the C ABI against the CPU oracle.

Every test runs the library's kernels (libkvev.so) on seeded synthetic inputs
and compares scores, kept positions, gathered K/V bytes and H2O state with the
oracle under the match criteria of ``tests/parity.py``.
"""
import os

import numpy as np
import pytest

from paper_2606_15157_gb300 import inputs as gen

from . import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as t
    if not t.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_15157_gb300 import kvev
    kvev.load()
    return t


def host_to_dev(torch, arrays):
    out = {}
    for l, (K, V, Q) in arrays.items():
        f = lambda a: None if a is None else torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)
        out[l] = (f(K), f(V), f(Q))
    return out


def device_workload(wl, layers=None):
    layers = range(wl.L) if layers is None else layers
    return {l: gen.device_layer(wl, l, need_q=wl.route[l] in (gen.SNAPKV, gen.H2O)) for l in layers}


def oracle_alloc(s, B_total, b_min, transform):
    import oracle
    return oracle.alloc_from_scores(s, B_total, b_min, transform)


def kvev_alloc(s, B_total, b_min, transform):
    from paper_2606_15157_gb300 import kvev
    return kvev.alloc_from_scores(s, B_total, b_min, transform)


# ---------------------------------------------------------------------------

def test_synth_device_matches_host(torch):
    # The device generator reproduces the host generator bit for bit.
    wl = gen.config_tiny(seed=3)
    host = gen.host_tensors(wl, [0, 2])
    for l in (0, 2):
        K, V, Q = gen.device_layer(wl, l)
        assert np.array_equal(parity.to_host_u16(K), host[l][0])
        assert np.array_equal(parity.to_host_u16(V), host[l][1])
        assert np.array_equal(parity.to_host_u16(Q), host[l][2])
    wl2 = gen.config_homog8k(seed=1)
    for l in (0, 13, 31):
        K, V, Q = gen.device_layer(wl2, l)
        pos = np.array([0, 5, wl2.plant["start"][l], wl2.plant["start"][l] + 1, 8191])
        for h in (0, 7):
            assert np.array_equal(parity.to_host_u16(K[0, h])[pos], gen.k_rows(wl2, l, 0, h, pos))
            assert np.array_equal(parity.to_host_u16(Q[0, h * 4:(h + 1) * 4]), gen.q_group(wl2, l, 0, h))
    k, v, q = gen.device_decode_tokens(wl2, 5, 3)
    kh, vh, qh = gen.decode_token(wl2, 5, 3, 0, 6)
    assert np.array_equal(parity.to_host_u16(k[0, 6]), kh)
    assert np.array_equal(parity.to_host_u16(v[0, 6]), vh)
    assert np.array_equal(parity.to_host_u16(q[0, 24:28]), qh)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_tiny_config(torch, orc, seed):
    wl = gen.config_tiny(seed)
    dev = host_to_dev(torch, gen.host_tensors(wl))
    stats = {}
    parity.check_workload(wl, dev, wl.lens, stats=stats)
    assert stats["max_rel_err"] < 2e-3


def test_homogeneous_snapkv_8k(torch, orc):
    wl = gen.config_homog8k(seed=0)
    dev = device_workload(wl)
    stats = {}
    parity.check_workload(wl, dev, wl.lens, stats=stats)
    print("homog8k", stats)


@pytest.mark.parametrize("bbar", [128, 256, 512, 1024, 2048])
def test_heterogeneous_route_8k(torch, orc, bbar):
    wl = gen.config_hetero8k(kvev_alloc, seed=0, bbar=bbar)
    wl_o = gen.config_hetero8k(oracle_alloc, seed=0, bbar=bbar)
    assert np.array_equal(wl.budget, wl_o.budget)
    assert wl.budget.sum() == 32 * bbar
    dev = device_workload(wl)
    stats = {}
    parity.check_workload(wl_o, dev, wl.lens, stats=stats)
    print("hetero8k", bbar, stats)


def _sample_units(wl, k, seed):
    rng = np.random.default_rng(seed)
    units = []
    for op in (gen.SNAPKV, gen.H2O, gen.STREAMING):
        layers = np.nonzero(wl.route == op)[0]
        for _ in range(k):
            units.append((int(rng.choice(layers)), int(rng.integers(wl.B)), int(rng.integers(wl.H_kv))))
    return sorted(set(units))


def test_long_context_batch_every_unit(torch, orc):
    # Full-size headline workload (batch 8, ragged 16K-32K, W=64) in the launch
    # configuration the benchmark times: every (layer, sequence, KV head) unit
    # against the oracle (all host cores), plus properties that hold at any size.
    import oracle
    wl = gen.config_long(kvev_alloc, seed=0)
    wl_o = gen.config_long(oracle_alloc, seed=0)
    assert np.array_equal(wl.budget, wl_o.budget)
    dev = device_workload(wl)
    stats = {}
    plan, bufs, gpu = parity.check_workload(wl_o, dev, wl.lens, stats=stats,
                                            nthreads=os.cpu_count())
    assert stats["units_checked"] == wl.L * wl.B * wl.H_kv
    print("long, every unit", stats)
    # properties over every unit
    for l in range(wl.L):
        b = int(wl.budget[l])
        for s in range(wl.B):
            n = int(wl.lens[s])
            assert np.all(gpu.count[l, s] == min(b, n))
            base0 = plan.layer_offset(wl.B, l)
            blk = gpu.idx[base0 + s * wl.H_kv * b: base0 + (s + 1) * wl.H_kv * b].reshape(wl.H_kv, b)
            assert np.all(np.diff(blk, axis=1) > 0)
            prot = {gen.SNAPKV: wl.W, gen.H2O: b // 2, gen.STREAMING: b - wl.sink}[int(wl.route[l])]
            assert np.all(blk[:, b - prot:] == np.arange(n - prot, n)[None, :])
            if wl.route[l] in (gen.SNAPKV, gen.H2O):
                tot = gpu.scores[l][s, :, :n].astype(np.float64).sum(axis=1)
                assert np.allclose(tot, wl.W, rtol=1e-3)  # each window row's softmax sums to 1
    # gathered rows of every unit equal the source rows (device-side check)
    outK = bufs["out_K"]
    for l in range(wl.L):
        b = int(wl.budget[l])
        base0 = plan.layer_offset(wl.B, l)
        idx = bufs["out_idx"][base0: base0 + wl.B * wl.H_kv * b].view(wl.B, wl.H_kv, b).long()
        src = dev[l][0].view(torch.int16)
        ref = torch.gather(src, 2, idx.unsqueeze(-1).expand(-1, -1, -1, wl.d))
        got = outK[base0: base0 + wl.B * wl.H_kv * b].view(torch.int16).view(wl.B, wl.H_kv, b, wl.d)
        assert torch.equal(ref, got)


def test_long_context_fixed_32k_sampled(torch, orc):
    # The fixed-length variant of the headline (batch 8, every sequence 32,768
    # tokens): sampled units of every rule against the oracle, and every unit's
    # kept count and protected window.
    import oracle
    wl = gen.config_long(kvev_alloc, seed=0, fixed_len=32768)
    wl_o = gen.config_long(oracle_alloc, seed=0, fixed_len=32768)
    assert np.array_equal(wl.budget, wl_o.budget) and np.all(wl.lens == 32768)
    dev = device_workload(wl)
    stats = {}
    plan, bufs, gpu = parity.check_workload(wl_o, dev, wl.lens, units=_sample_units(wl, 6, 1),
                                            stats=stats, nthreads=os.cpu_count())
    print("long fixed 32K, sampled", stats)
    for l in range(wl.L):
        b = int(wl.budget[l])
        assert np.all(gpu.count[l] == min(b, 32768))
        base0 = plan.layer_offset(wl.B, l)
        blk = gpu.idx[base0: base0 + wl.B * wl.H_kv * b].reshape(wl.B * wl.H_kv, b)
        prot = {gen.SNAPKV: wl.W, gen.H2O: b // 2, gen.STREAMING: b - wl.sink}[int(wl.route[l])]
        assert np.all(blk[:, b - prot:] == np.arange(32768 - prot, 32768)[None, :])
        assert np.all(np.diff(blk, axis=1) > 0)


def _window_lse_device(wl, dev, torch):
    """A caller's prefill-attention normalisers at full size: per SnapKV / H2O layer
    fp32 [B][H_q][W] log-sum-exp of each window row over the keys it sees, from a
    plain fp32 torch softmax on the device."""
    import math
    tf32 = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    out = []
    for l in range(wl.L):
        if int(wl.route[l]) not in (gen.SNAPKV, gen.H2O):
            out.append(None)
            continue
        K, _, Q = dev[l]
        lse = torch.zeros((wl.B, wl.H_q, wl.W), dtype=torch.float32, device="cuda")
        for s in range(wl.B):
            n = int(wl.lens[s])
            t = n - wl.W + torch.arange(wl.W, device="cuda")
            mask = torch.arange(n, device="cuda")[None, :] > t[:, None]
            for h in range(wl.H_kv):
                S = torch.matmul(Q[s, h * wl.G:(h + 1) * wl.G].float(), K[s, h, :n].float().T) / math.sqrt(wl.d)
                S.masked_fill_(mask[None], float("-inf"))
                lse[s, h * wl.G:(h + 1) * wl.G] = torch.logsumexp(S, dim=-1)
        out.append(lse)
    torch.backends.cuda.matmul.allow_tf32 = tf32
    return out


def test_long_context_supplied_lse_sampled(torch, orc):
    # The headline workload through kvev_evict_prefill_lse (one score sweep), the
    # window rows' log-sum-exp from the caller's attention (plain fp32 torch on the
    # device): sampled units of every rule against the oracle, which forms its own
    # normalisers, and every scored unit's window-row mass.
    wl = gen.config_long(kvev_alloc, seed=0)
    wl_o = gen.config_long(oracle_alloc, seed=0)
    assert np.array_equal(wl.budget, wl_o.budget)
    dev = device_workload(wl)
    lse = _window_lse_device(wl, dev, torch)
    stats = {}
    plan, bufs, gpu = parity.check_workload(wl_o, dev, wl.lens, units=_sample_units(wl, 8, 2), stats=stats,
                                            nthreads=os.cpu_count(), lse=lse)
    print("long, supplied lse, sampled", stats)
    for l in range(wl.L):
        if wl.route[l] in (gen.SNAPKV, gen.H2O):
            for s in range(wl.B):
                n = int(wl.lens[s])
                tot = gpu.scores[l][s, :, :n].astype(np.float64).sum(axis=1)
                assert np.allclose(tot, wl.W, rtol=1e-3)  # each window row's softmax sums to 1


def _custom(L_routes, budgets, lens, W=16, d=128, H_q=8, H_kv=2, S_cap=None, pool=(5, gen.POOL_MAX),
            seed=7, sink=4, h2o_recent=-1):
    lens = np.asarray(lens, np.int32)
    S_cap = S_cap or int(max(lens.max(), 1))
    return gen.Workload(name="edge", L=len(L_routes), H_q=H_q, H_kv=H_kv, d=d, B=len(lens), lens=lens,
                        S_cap=S_cap, W=W, pool_kernel=pool[0], pool_type=pool[1],
                        route=np.asarray(L_routes, np.int32), budget=np.asarray(budgets, np.int32),
                        sink=sink, seed=seed, sink_tokens=4, h2o_recent=h2o_recent)


@pytest.mark.parametrize("d", [64, 128])
def test_edge_lengths(torch, orc, d):
    # Ragged batch with empty, shorter-than-window, exactly-budget, budget+1,
    # non-multiple-of-tile and full-capacity lengths; FULL layers interleaved.
    b = 40
    lens = [0, 1, 15, 16, 40, 41, 127, 129, 1000, 1031]
    routes = [gen.SNAPKV, gen.H2O, gen.STREAMING, gen.FULL, gen.H2O, gen.SNAPKV]
    wl = _custom(routes, [b, b, b, 0, 7, 130], lens, d=d, S_cap=1031)
    dev = device_workload(wl)
    parity.check_workload(wl, dev, wl.lens)


def test_selection_dispatch_orders(torch, orc):
    # The selection launch takes the SnapKV / H2O units longest sequence first
    # (sequences ranked by warp 0, up to 32 of them; larger batches keep the
    # index order), with the StreamingLLM units (which also copy their kept
    # rows) and FULL units spread between them.  Cases: 40 ragged sequences (the
    # index order), equal lengths (rank ties), a route with no scoring layer
    # and one with no StreamingLLM or FULL layer.
    rng = np.random.default_rng(11)
    lens40 = rng.integers(150, 600, size=40)
    lens40[[3, 17, 31]] = 600  # ties across the first 32 and past them
    cases = [
        ([gen.STREAMING, gen.SNAPKV, gen.FULL, gen.H2O], [40, 64, 0, 90], lens40),
        ([gen.SNAPKV, gen.STREAMING, gen.H2O], [48, 40, 70], [500, 500, 320, 500, 320]),
        ([gen.STREAMING, gen.FULL, gen.STREAMING], [40, 0, 24], [700, 30, 455]),
        ([gen.SNAPKV, gen.H2O], [64, 100], [900, 300, 1200]),
    ]
    for routes, budgets, lens in cases:
        wl = _custom(routes, budgets, lens, H_q=4, H_kv=2, d=64)
        parity.check_workload(wl, device_workload(wl), wl.lens)


def test_edge_window_and_groups(torch, orc):
    # Different GQA group sizes and windows: R = G*W = 16, 48 (a 16-column tail), 128, 192, 256.
    for (H_q, H_kv, W) in [(4, 2, 8), (12, 4, 16), (8, 2, 32), (12, 2, 32), (32, 8, 64)]:
        wl = _custom([gen.SNAPKV, gen.H2O], [W + 37, 100], [700, 3000, 2 * W], W=W, H_q=H_q, H_kv=H_kv,
                     pool=(7, gen.POOL_AVG))
        dev = device_workload(wl)
        parity.check_workload(wl, dev, wl.lens)


def test_h2o_recent_override_and_ties(torch, orc):
    # h2o_recent = 0 (pure heavy hitters) and = b (pure recency); plus all-zero
    # queries so every score in a row ties and the lower-position rule decides.
    wl = _custom([gen.H2O, gen.H2O, gen.SNAPKV], [64, 64, 64], [900, 2000], h2o_recent=0)
    dev = device_workload(wl)
    for l in dev:
        if dev[l][2] is not None:
            dev[l][2].zero_() if l == 2 else None
    parity.check_workload(wl, dev, wl.lens)
    wl2 = _custom([gen.H2O], [50], [600], h2o_recent=50)
    parity.check_workload(wl2, device_workload(wl2), wl2.lens)


def test_select_crowded_first_bin(torch, orc):
    # Long units whose candidate bin can hold more keys than the selection's
    # candidate list.  Layer 0 has zero queries, so all of its prefix scores
    # tie (lower positions win the ties); layer 1 keeps live queries and takes
    # the candidate path at full length.
    wl = _custom([gen.SNAPKV, gen.H2O], [2048, 1024], [38000, 30000], W=8, H_q=4, H_kv=2, S_cap=40000, d=64)
    dev = device_workload(wl)
    dev[0][2].zero_()
    parity.check_workload(wl, dev, wl.lens)


def test_capacity_beyond_shared_memory(torch, orc):
    # Capacities past what one CTA's shared memory could hold as keys (53,504
    # positions at 4 bytes): the selection keeps them in the workspace at any
    # capacity.  Sequences that fill the capacity, against the oracle.
    for s_cap in (53504, 65536):
        wl = _custom([gen.SNAPKV, gen.H2O], [512, 300], [s_cap, s_cap - 777], W=8, H_q=4, H_kv=2,
                     S_cap=s_cap, d=64)
        parity.check_workload(wl, device_workload(wl), wl.lens)


def test_supplied_scores(torch, orc):
    # kvev_evict_prefill_scored: the scores of layer 0 (SnapKV) and layer 1 (H2O)
    # come from the caller -- here the oracle's own window scores rounded to
    # fp32 -- and their Q_win is not passed; layer 3 (SnapKV) is still scored by
    # the library.  Pooling, selection, gather and the H2O decode seed must
    # match the oracle on every unit, as in the scored path.
    import oracle
    from paper_2606_15157_gb300 import kvev
    routes = [gen.SNAPKV, gen.H2O, gen.STREAMING, gen.SNAPKV]
    wl = _custom(routes, [64, 80, 64, 100], [900, 1500, 17], W=16)
    dev = device_workload(wl)
    supplied = (0, 1)
    specs, meta = [], []
    for l in range(wl.L):
        for s in range(wl.B):
            n = int(wl.lens[s])
            Kh, Vh = parity.to_host_u16(dev[l][0][s]), parity.to_host_u16(dev[l][1][s])
            Qh = None if dev[l][2] is None else parity.to_host_u16(dev[l][2][s])
            for h in range(wl.H_kv):
                spec = parity.oracle_spec(wl, l, s, h, Kh[h][:max(n, 1)],
                                          None if Qh is None else Qh[h * wl.G:(h + 1) * wl.G])
                spec["n"] = n
                specs.append(spec)
                meta.append((l, s, h, n, Kh[h], Vh[h]))
    results = oracle.evict_units(specs, d=wl.d, G=wl.G)
    S = {l: np.zeros((wl.B, wl.H_kv, wl.S_cap), np.float32) for l in supplied}
    for (l, s, h, n, _, _), res in zip(meta, results):
        if l in supplied and n > 0:
            S[l][s, h, :n] = res.raw[:n]
    plan = kvev.Plan.from_workload(wl)
    bufs = plan.buffers(wl.B, wl.S_cap)
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    K = [dev[l][0] for l in range(wl.L)]
    V = [dev[l][1] for l in range(wl.L)]
    Q = [None if l in supplied else dev[l][2] for l in range(wl.L)]
    scores = [torch.from_numpy(S[l]).cuda() if l in supplied else None for l in range(wl.L)]
    plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs, scores=scores)
    torch.cuda.synchronize()
    assert plan.status() == kvev.OK
    gpu = parity.GpuRun(plan, wl, bufs, np.asarray(wl.lens))
    for l in supplied:  # the scores the selection read are the supplied ones
        gpu.scores[l] = S[l]
    for (l, s, h, n, Kr, Vr), res in zip(meta, results):
        parity.check_unit(wl, l, s, h, n, res, gpu, Kr, Vr)


def _window_lse(wl, dev, torch):
    """The caller's prefill-attention normalisers: for every SnapKV / H2O layer,
    fp32 [B][H_q][W] log-sum-exp of each window row over the keys it sees, from a
    plain fp64 softmax of the same bf16 rows (the library never computes them in
    this mode)."""
    out = []
    for l in range(wl.L):
        if int(wl.route[l]) not in (gen.SNAPKV, gen.H2O):
            out.append(None)
            continue
        lse = np.zeros((wl.B, wl.H_q, wl.W), np.float32)
        for s in range(wl.B):
            n = int(wl.lens[s])
            if n == 0:
                continue
            Kh = gen.bf16_bits_to_f32(parity.to_host_u16(dev[l][0][s])).astype(np.float64)
            Qh = gen.bf16_bits_to_f32(parity.to_host_u16(dev[l][2][s])).astype(np.float64)
            t = n - wl.W + np.arange(wl.W)                     # positions of the window rows
            for q in range(wl.H_q):
                S = Qh[q] @ Kh[q // wl.G][:n].T / np.sqrt(wl.d)  # [W][n]
                S[np.arange(n)[None, :] > t[:, None]] = -np.inf
                m = S.max(axis=1)
                ok = t >= 0
                lse[s, q, ok] = (m[ok] + np.log(np.exp(S[ok] - m[ok, None]).sum(axis=1)))
        out.append(torch.from_numpy(lse).cuda())
    return out


@pytest.mark.parametrize("d", [64, 128])
def test_supplied_lse(torch, orc, d):
    # kvev_evict_prefill_lse: the window rows' log-sum-exp comes from the caller's
    # own prefill attention, and the score kernel makes a single sweep over K.
    # Ragged lengths (one shorter than the window, one not a multiple of the
    # tile), SnapKV with max and avg pooling, H2O, a StreamingLLM and a FULL
    # layer; every unit against the oracle, which forms its own normalisers.
    routes = [gen.SNAPKV, gen.H2O, gen.STREAMING, gen.FULL, gen.SNAPKV]
    for pool in ((7, gen.POOL_AVG), (5, gen.POOL_MAX)):
        wl = _custom(routes, [64, 80, 64, 0, 100], [900, 1500, 11, 2100], W=16, d=d, pool=pool)
        dev = device_workload(wl)
        parity.check_workload(wl, dev, wl.lens, lse=_window_lse(wl, dev, torch))


def test_supplied_lse_groups_and_windows(torch, orc):
    # The same for R = G*W of 48 (a 16-column tail), 128 and 256 rows.
    for (H_q, H_kv, W) in [(12, 4, 16), (8, 2, 32), (32, 8, 64)]:
        wl = _custom([gen.SNAPKV, gen.H2O], [W + 37, 100], [700, 3000, 2 * W], W=W, H_q=H_q, H_kv=H_kv,
                     pool=(7, gen.POOL_AVG))
        dev = device_workload(wl)
        parity.check_workload(wl, dev, wl.lens, lse=_window_lse(wl, dev, torch))


def test_repeat_calls_identical(torch):
    wl = gen.config_tiny(1)
    dev = host_to_dev(torch, gen.host_tensors(wl))
    plan, bufs = parity.run_gpu(wl, dev, wl.lens)
    first = {k: v.clone() for k, v in bufs.items() if hasattr(v, "clone")}
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    K = [dev[l][0] for l in range(wl.L)]
    V = [dev[l][1] for l in range(wl.L)]
    Q = [dev[l][2] for l in range(wl.L)]
    for _ in range(3):
        plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs)
    torch.cuda.synchronize()
    for k in ("out_K", "out_V", "out_idx", "out_count"):
        assert torch.equal(first[k], bufs[k])


def test_host_resident_gathered_tensors(torch):
    # V of every layer and K of the StreamingLLM layers are only gathered at
    # the kept positions: passed as pinned host memory they are read in place,
    # with outputs identical to the all-device call.
    from paper_2606_15157_gb300 import kvev
    wl = gen.config_tiny(2)
    dev = host_to_dev(torch, gen.host_tensors(wl))
    plan = kvev.Plan.from_workload(wl)
    bufs = plan.buffers(wl.B, wl.S_cap)
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    pin = lambda t: None if t is None else t.cpu().pin_memory()
    scoring = [int(wl.route[l]) in (gen.SNAPKV, gen.H2O) for l in range(wl.L)]
    Q = [dev[l][2] for l in range(wl.L)]
    runs = []
    for host in (False, True):
        for b in bufs.values():
            if hasattr(b, "zero_"):
                b.zero_()
        K = [dev[l][0] if (scoring[l] or not host) else pin(dev[l][0]) for l in range(wl.L)]
        V = [pin(dev[l][1]) if host else dev[l][1] for l in range(wl.L)]
        plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs)
        torch.cuda.synchronize()
        assert plan.status() == kvev.OK
        runs.append({k: bufs[k].clone() for k in ("out_K", "out_V", "out_idx", "out_count", "h2o_state")})
    for k in runs[0]:
        assert torch.equal(runs[0][k], runs[1][k]), k


def test_wait_timeout_reports_status(torch):
    # A unit whose normaliser is never published: every wait on it runs out
    # after the (short) limit, the kernel finishes, the status word says
    # ETIMEOUT, and the context stays usable for the next call.
    from paper_2606_15157_gb300 import kvev
    wl = gen.config_tiny(0)
    dev = host_to_dev(torch, gen.host_tensors(wl))
    plan = kvev.Plan.from_workload(wl)
    kvev.kvev_plan_set_wait_limit(plan.handle, 20_000_000)  # 20 ms
    kvev.kvev_plan_debug_stall_unit(plan.handle, 0)
    bufs = plan.buffers(wl.B, wl.S_cap)
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    K = [dev[l][0] for l in range(wl.L)]
    V = [dev[l][1] for l in range(wl.L)]
    Q = [dev[l][2] for l in range(wl.L)]
    plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs)
    torch.cuda.synchronize()
    assert plan.status() == kvev.ETIMEOUT
    kvev.kvev_plan_debug_stall_unit(plan.handle, -1)
    plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs)
    torch.cuda.synchronize()
    assert plan.status() == kvev.OK


def test_invalid_lengths_flagged(torch):
    from paper_2606_15157_gb300 import kvev
    wl = _custom([gen.SNAPKV, gen.STREAMING], [40, 40], [100, 200], S_cap=200)
    dev = device_workload(wl)
    plan = kvev.Plan.from_workload(wl)
    bufs = plan.buffers(wl.B, wl.S_cap)
    lens = torch.tensor([100, 5000], dtype=torch.int32, device="cuda")  # 5000 > S_cap
    K = [dev[l][0] for l in range(wl.L)]
    V = [dev[l][1] for l in range(wl.L)]
    Q = [dev[l][2] for l in range(wl.L)]
    plan.evict_prefill(K, V, Q, lens, wl.B, wl.S_cap, bufs)
    torch.cuda.synchronize()
    assert plan.status() == kvev.EDEVICE
    cnt = bufs["out_count"].cpu().numpy()
    assert np.all(cnt[:, 1] == 0)  # the invalid sequence is treated as empty
