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


@pytest.mark.parametrize("H_q,H_kv,d,lens", GEOMETRIES)
def test_h2o_full_prompt_scores_and_selection(torch, H_q, H_kv, d, lens):
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

    plan = kvev.Plan(wl.L, wl.H_q, wl.H_kv, wl.d, wl.route, wl.budget, wl.W, wl.pool_kernel, wl.pool_type,
                     wl.sink, wl.recent, wl.h2o_recent, h2o_full_prompt=True)
    bufs = plan.buffers(wl.B, wl.S_cap)
    plan.evict_prefill(K, V, Q, lens_dev, wl.B, wl.S_cap, bufs)
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
