"""GPU parity of H2O prefill scoring over every prompt query row (H2O's
original accumulated attention, Sec. 2.1): the library computes each row's
normaliser in a row pass and the key sums in a key pass; the oracle evaluates
the definition with the whole prompt as the window.  SnapKV layers of the same
plan keep their observation-window scores, identical to a plan without the
option."""
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


def _bf16_bits(rng, shape, scale=1.0):
    x = (rng.standard_normal(shape) * scale).astype(np.float32)
    u = x.view(np.uint32)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)  # round to nearest even


# (H_q, H_kv, d, lens): G = 4 fills 256-row blocks of 64 positions; G = 3
# leaves a 255-row block of 85 positions; G = 8 gives blocks of 32 positions.
GEOMETRIES = [
    (8, 2, 128, (700, 1000)),
    (8, 2, 128, (16, 1)),
    (12, 4, 64, (300, 0, 517)),
    (16, 2, 64, (450, 129)),
]


def _rows_lse(Kh, Qh, n, t_rows, d):
    """ln sum_{k <= t} exp(q_t . k / sqrt(d)) for the query rows Qh [rows][d] at
    positions t_rows, from the bf16 bits in fp64 (a caller's attention)."""
    Kf = gen.bf16_bits_to_f32(Kh[:n]).astype(np.float64)
    Qf = gen.bf16_bits_to_f32(Qh).astype(np.float64)
    S = Qf @ Kf.T / np.sqrt(d)
    S[np.arange(n)[None, :] > t_rows[:, None]] = -np.inf
    m = S.max(axis=1)
    out = np.zeros(len(t_rows), np.float32)
    ok = t_rows >= 0
    out[ok] = m[ok] + np.log(np.exp(S[ok] - m[ok, None]).sum(axis=1))
    return out


@pytest.mark.parametrize("supplied_lse", [False, True])
@pytest.mark.parametrize("H_q,H_kv,d,lens", GEOMETRIES)
def test_h2o_full_prompt_scores_and_selection(torch, H_q, H_kv, d, lens, supplied_lse):
    from paper_2606_15157_gb300 import kvev
    import oracle
    route = [gen.H2O, gen.SNAPKV, gen.H2O]
    wl = gen.Workload(name="h2o_full", L=3, H_q=H_q, H_kv=H_kv, d=d, B=len(lens), lens=np.asarray(lens, np.int32),
                      S_cap=1024, W=16, pool_kernel=5, pool_type=gen.POOL_MAX,
                      route=np.asarray(route, np.int32), budget=np.asarray([256, 200, 96], np.int32),
                      sink=4, seed=11, sink_tokens=4, h2o_recent=-1)
    rng = np.random.default_rng(5)
    dev, q_full = {}, {}
    for l in range(wl.L):
        K, V, Qw = gen.device_layer(wl, l, need_q=route[l] == gen.SNAPKV)
        if route[l] == gen.H2O:
            qb = _bf16_bits(rng, (wl.B, wl.H_q, wl.S_cap, wl.d))
            q_full[l] = qb
            Qw = torch.from_numpy(qb.view(np.int16)).cuda().view(torch.bfloat16)
        dev[l] = (K, V, Qw)
    lens_dev = torch.from_numpy(np.asarray(lens, np.int32)).cuda()
    K = [dev[l][0] for l in range(wl.L)]
    V = [dev[l][1] for l in range(wl.L)]
    Q = [dev[l][2] for l in range(wl.L)]

    lse = None
    if supplied_lse:
        # kvev_evict_prefill_lse: the caller's attention gives every prompt row's
        # log-sum-exp for the H2O layers ([B][H_q][S_cap]; the row pass is
        # skipped) and the window rows' for the SnapKV layer ([B][H_q][W])
        lse = []
        for l in range(wl.L):
            rows = wl.S_cap if route[l] == gen.H2O else wl.W
            x = np.zeros((wl.B, wl.H_q, rows), np.float32)
            for s in range(wl.B):
                n = int(lens[s])
                if n == 0:
                    continue
                Kh = parity.to_host_u16(dev[l][0][s])
                t = np.arange(n) if route[l] == gen.H2O else n - wl.W + np.arange(wl.W)
                for q in range(wl.H_q):
                    Qq = q_full[l][s, q, :n] if route[l] == gen.H2O else parity.to_host_u16(dev[l][2][s])[q]
                    x[s, q, :len(t)] = _rows_lse(Kh[q // wl.G], Qq, n, t, wl.d)
            lse.append(torch.from_numpy(x).cuda())
    plan = kvev.Plan(wl.L, wl.H_q, wl.H_kv, wl.d, wl.route, wl.budget, wl.W, wl.pool_kernel, wl.pool_type,
                     wl.sink, wl.recent, wl.h2o_recent, h2o_full_prompt=True)
    bufs = plan.buffers(wl.B, wl.S_cap)
    plan.evict_prefill(K, V, Q, lens_dev, wl.B, wl.S_cap, bufs, lse=lse)
    torch.cuda.synchronize()
    assert plan.status() == kvev.OK
    gpu = parity.GpuRun(plan, wl, bufs, np.asarray(lens))

    specs, meta = [], []
    for l in range(wl.L):
        for s in range(wl.B):
            n = int(lens[s])
            Kh = parity.to_host_u16(dev[l][0][s])
            Vh = parity.to_host_u16(dev[l][1][s])
            for h in range(wl.H_kv):
                if route[l] == gen.H2O:
                    # the definition: every prompt position is a query row (window = the prompt)
                    Qg = np.ascontiguousarray(q_full[l][s, h * wl.G:(h + 1) * wl.G, :max(n, 1)])
                    spec = parity.oracle_spec(wl, l, s, h, Kh[h][:max(n, 1)], Qg)
                    spec["W"] = max(n, 1)
                else:
                    Qh = parity.to_host_u16(dev[l][2][s])
                    spec = parity.oracle_spec(wl, l, s, h, Kh[h][:max(n, 1)], Qh[h * wl.G:(h + 1) * wl.G])
                spec["n"] = n
                specs.append(spec)
                meta.append((l, s, h, n, Kh[h], Vh[h]))
    results = oracle.evict_units(specs, d=wl.d, G=wl.G)
    for (l, s, h, n, Kr, Vr), res in zip(meta, results):
        parity.check_unit(wl, l, s, h, n, res, gpu, Kr, Vr)

    if supplied_lse:
        return  # the check below compares two library-formed normalisers bit for bit
    # the SnapKV layer's window scores do not depend on the option
    ref = kvev.Plan(wl.L, wl.H_q, wl.H_kv, wl.d, wl.route, wl.budget, wl.W, wl.pool_kernel, wl.pool_type,
                    wl.sink, wl.recent, wl.h2o_recent)
    rbufs = ref.buffers(wl.B, wl.S_cap)
    Qwin = [dev[l][2] if route[l] == gen.SNAPKV else
            torch.from_numpy(np.ascontiguousarray(q_full[l][:, :, :wl.W]).view(np.int16)).cuda().view(torch.bfloat16)
            for l in range(wl.L)]
    ref.evict_prefill(K, V, Qwin, lens_dev, wl.B, wl.S_cap, rbufs)
    torch.cuda.synchronize()
    for s in range(wl.B):
        n = int(lens[s])
        if n <= wl.budget[1]:  # kept whole: the layer scores nothing for this sequence
            continue
        a = plan.scores(bufs, wl.B, wl.S_cap, 1)[s, :, :n]
        b = ref.scores(rbufs, wl.B, wl.S_cap, 1)[s, :, :n]
        assert torch.equal(a, b)


def _full_prompt_workload(n, seed):
    route = [gen.H2O, gen.SNAPKV, gen.H2O]
    return gen.Workload(name=f"h2o_full_{n}", L=3, H_q=32, H_kv=8, d=128, B=1, lens=np.asarray([n], np.int32),
                        S_cap=n, W=32, pool_kernel=7, pool_type=gen.POOL_AVG,
                        route=np.asarray(route, np.int32), budget=np.asarray([512, 512, 768], np.int32),
                        sink=4, seed=seed, sink_tokens=4, h2o_recent=-1)


def _run_full_prompt(torch, wl, rng):
    from paper_2606_15157_gb300 import kvev
    dev, q_full = {}, {}
    for l in range(wl.L):
        K, V, Qw = gen.device_layer(wl, l, need_q=wl.route[l] == gen.SNAPKV)
        if wl.route[l] == gen.H2O:
            qb = _bf16_bits(rng, (wl.B, wl.H_q, wl.S_cap, wl.d))
            q_full[l] = qb
            Qw = torch.from_numpy(qb.view(np.int16)).cuda().view(torch.bfloat16)
        dev[l] = (K, V, Qw)
    lens_dev = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    plan = kvev.Plan(wl.L, wl.H_q, wl.H_kv, wl.d, wl.route, wl.budget, wl.W, wl.pool_kernel, wl.pool_type,
                     wl.sink, wl.recent, wl.h2o_recent, h2o_full_prompt=True)
    bufs = plan.buffers(wl.B, wl.S_cap)
    plan.evict_prefill([dev[l][0] for l in range(wl.L)], [dev[l][1] for l in range(wl.L)],
                       [dev[l][2] for l in range(wl.L)], lens_dev, wl.B, wl.S_cap, bufs)
    torch.cuda.synchronize()
    assert plan.status() == kvev.OK
    return plan, bufs, dev, q_full, parity.GpuRun(plan, wl, bufs, np.asarray(wl.lens))


def test_h2o_full_prompt_8k_properties(torch):
    # The geometry the full-prompt bench measures (8,192 positions, 32/8 heads,
    # d = 128: 128 query blocks and 32 key super-tiles per unit).  Every H2O
    # unit against the oracle (all host cores), and every H2O unit against
    # properties: each query row's softmax sums to 1, so the scores of a KV head
    # (averaged over its G query heads) sum to n and are positive; the kept
    # set is the recent window plus the top (b - r) of the unit's own scores
    # before it (ties to the lower position); the H2O state holds the kept
    # positions' scores.
    wl = _full_prompt_workload(8192, 21)
    n = int(wl.lens[0])
    plan, bufs, dev, q_full, gpu = _run_full_prompt(torch, wl, np.random.default_rng(8))
    for l in (0, 2):
        sc = gpu.scores[l][0].astype(np.float64)
        np.testing.assert_allclose(sc.sum(axis=1), n, rtol=2e-3)
        assert (sc[:, :n] > 0).all()
        b = int(wl.budget[l])
        r = b // 2
        for h in range(wl.H_kv):
            base, _ = gpu.unit_rows(l, 0, h)
            cnt = int(gpu.count[l, 0, h])
            kept = gpu.idx[base: base + cnt]
            assert cnt == b
            key = gpu.scores[l][0, h, :n - r]
            order = np.lexsort((np.arange(n - r), -key))  # larger score first, then lower position
            expect = set(order[:b - r].tolist()) | set(range(n - r, n))
            assert set(kept.tolist()) == expect
            np.testing.assert_array_equal(gpu.state[base: base + cnt], gpu.scores[l][0, h, kept])
    # and every H2O unit against the oracle
    import os
    import oracle
    specs, meta = [], []
    for (l, h) in [(l, h) for l in (0, 2) for h in range(wl.H_kv)]:
        Kh = parity.to_host_u16(dev[l][0][0])
        Vh = parity.to_host_u16(dev[l][1][0])
        spec = parity.oracle_spec(wl, l, 0, h, Kh[h][:n],
                                  np.ascontiguousarray(q_full[l][0, h * wl.G:(h + 1) * wl.G, :n]))
        spec["W"] = n
        spec["n"] = n
        specs.append(spec)
        meta.append((l, 0, h, n, Kh[h], Vh[h]))
    results = oracle.evict_units(specs, d=wl.d, G=wl.G, nthreads=os.cpu_count())
    for (l, s, h, n_, Kr, Vr), res in zip(meta, results):
        parity.check_unit(wl, l, s, h, n_, res, gpu, Kr, Vr)


def test_h2o_full_prompt_2k_oracle(torch):
    # The same geometry at 2,048 positions (32 query blocks, 8 key super-tiles):
    # every H2O unit against the oracle with the whole prompt as the window.
    import os
    import oracle
    wl = _full_prompt_workload(2048, 22)
    n = int(wl.lens[0])
    plan, bufs, dev, q_full, gpu = _run_full_prompt(torch, wl, np.random.default_rng(9))
    specs, meta = [], []
    for (l, h) in [(l, h) for l in (0, 2) for h in range(wl.H_kv)]:
        Kh = parity.to_host_u16(dev[l][0][0])
        Vh = parity.to_host_u16(dev[l][1][0])
        spec = parity.oracle_spec(wl, l, 0, h, Kh[h][:n],
                                  np.ascontiguousarray(q_full[l][0, h * wl.G:(h + 1) * wl.G, :n]))
        spec["W"] = n
        spec["n"] = n
        specs.append(spec)
        meta.append((l, 0, h, n, Kh[h], Vh[h]))
    results = oracle.evict_units(specs, d=wl.d, G=wl.G, nthreads=os.cpu_count())
    for (l, s, h, n_, Kr, Vr), res in zip(meta, results):
        parity.check_unit(wl, l, s, h, n_, res, gpu, Kr, Vr)


def test_full_prompt_with_one_layer_supplied(torch):
    # A full-prompt plan in which layer 0 (H2O) takes the caller's scores
    # (kvev_evict_prefill_scored; its Q is not passed) while layer 2 (H2O) is
    # scored over the whole prompt by the library: layer 0 selects exactly on
    # the supplied scores, layer 2 matches the plan without supplied scores.
    from paper_2606_15157_gb300 import kvev
    wl = _full_prompt_workload(1024, 31)
    n = int(wl.lens[0])
    plan, bufs, dev, q_full, gpu = _run_full_prompt(torch, wl, np.random.default_rng(10))
    rng = np.random.default_rng(11)
    sup = rng.random((wl.B, wl.H_kv, wl.S_cap)).astype(np.float32)
    plan2 = kvev.Plan(wl.L, wl.H_q, wl.H_kv, wl.d, wl.route, wl.budget, wl.W, wl.pool_kernel, wl.pool_type,
                      wl.sink, wl.recent, wl.h2o_recent, h2o_full_prompt=True)
    bufs2 = plan2.buffers(wl.B, wl.S_cap)
    lens_dev = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    Q = [None] + [dev[l][2] for l in range(1, wl.L)]
    scores = [torch.from_numpy(sup).cuda(), None, None]
    plan2.evict_prefill([dev[l][0] for l in range(wl.L)], [dev[l][1] for l in range(wl.L)], Q, lens_dev,
                        wl.B, wl.S_cap, bufs2, scores=scores)
    torch.cuda.synchronize()
    assert plan2.status() == kvev.OK
    g2 = parity.GpuRun(plan2, wl, bufs2, np.asarray(wl.lens))
    b = int(wl.budget[0])
    r = b // 2
    for h in range(wl.H_kv):
        base, _ = g2.unit_rows(0, 0, h)
        kept = g2.idx[base: base + b]
        key = sup[0, h, :n - r]
        order = np.lexsort((np.arange(n - r), -key))
        assert set(kept.tolist()) == set(order[:b - r].tolist()) | set(range(n - r, n))
        np.testing.assert_array_equal(g2.state[base: base + b], sup[0, h, kept])
    # layer 2: the same as in the plan where the library scores both H2O layers
    assert np.array_equal(g2.scores[2][0, :, :n], gpu.scores[2][0, :, :n])
    for h in range(wl.H_kv):
        b2 = int(wl.budget[2])
        base, _ = g2.unit_rows(2, 0, h)
        base1, _ = gpu.unit_rows(2, 0, h)
        assert np.array_equal(g2.idx[base: base + b2], gpu.idx[base1: base1 + b2])
