"""GPU parity of the decode step (kvev_decode_init / kvev_decode_step) against the
oracle, replayed in lock step: the oracle's slot sets start as a copy of the GPU
arena after initialisation and both advance by the same new tokens.  Per step
and unit: the same count, the same set of positions, K/V rows identical byte
for byte by position, acc within the score tolerance.  A different eviction is
accepted only where the two candidates' accumulated attention is a near tie
(within the tolerance); the oracle then continues from the GPU state.
"""
import numpy as np
import pytest

from paper_2606_15157_gb300 import inputs as gen

pytestmark = pytest.mark.gpu

REL = 2e-3  # score tolerance of the parity criteria


@pytest.fixture(scope="module")
def env():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_15157_gb300 import kvev
    from oracle import oracle as orc
    kvev.load()
    return torch, kvev, orc


class Arena:
    """Host copy of a DecodeArena plus unit bookkeeping."""

    def __init__(self, torch, arena, wl):
        self.a, self.wl = arena, wl
        self.units = []  # (layer, s, h, u, rows0, cap)
        for l, (off, cap, u0) in enumerate(arena.layers):
            if cap == 0:
                continue
            for s in range(wl.B):
                for h in range(wl.H_kv):
                    i = s * wl.H_kv + h
                    self.units.append((l, s, h, u0 + i, off + i * cap, cap))
        self.refresh(torch)

    def refresh(self, torch):
        torch.cuda.synchronize()
        self.K = self.a.K.view(torch.int16).cpu().numpy().view(np.uint16)
        self.V = self.a.V.view(torch.int16).cpu().numpy().view(np.uint16)
        self.pos = self.a.pos().cpu().numpy()
        self.acc = self.a.acc().cpu().numpy()
        self.count = self.a.count().cpu().numpy()
        self.lens = self.a.lens().cpu().numpy()
        self.evicted = self.a.evicted().cpu().numpy()

    def unit(self, i):
        l, s, h, u, r0, cap = self.units[i]
        c = int(self.count[u])
        sl = slice(r0, r0 + c)
        return {"count": c, "pos": self.pos[sl], "acc": self.acc[sl].astype(np.float64),
                "K": self.K[sl], "V": self.V[sl]}


def oracle_state(orc, wl, plan_dec, g, i):
    l, s, h, u, r0, cap = g.units[i]
    x = g.unit(i)
    # the oracle appends before it evicts: one slot of working room past the arena
    return orc.DecodeState(int(plan_dec[l]), int(wl.budget[l]), cap + 1, wl.d, int(g.lens[s]),
                           x["pos"], x["K"], x["V"], x["acc"], sink=wl.sink, recent=wl.recent,
                           h2o_recent=wl.h2o_recent)


def resync(st, x):
    c = x["count"]
    st.count = c
    st.pos[:] = -1
    st.pos[:c] = x["pos"]
    st.acc[:] = 0.0
    st.acc[:c] = x["acc"]
    st.K[:c] = x["K"]
    st.V[:c] = x["V"]


def compare_unit(st, x, what):
    """None if the unit matches, 'tie' for a tolerated near-tie eviction; raises otherwise."""
    assert st.count == x["count"], f"{what}: count {x['count']} vs oracle {st.count}"
    c = st.count
    po, pg = st.pos[:c], x["pos"]
    if set(po.tolist()) != set(pg.tolist()):
        only_o = sorted(set(po.tolist()) - set(pg.tolist()))   # the GPU evicted these
        only_g = sorted(set(pg.tolist()) - set(po.tolist()))   # the oracle evicted these
        assert len(only_o) == 1 and len(only_g) == 1, f"{what}: slot sets differ {only_o} {only_g}"
        a_o_gpu_choice = st.acc[:c][po == only_o[0]][0]
        a_g_oracle_choice = x["acc"][pg == only_g[0]][0]
        scale = max(abs(a_o_gpu_choice), abs(a_g_oracle_choice), 1e-30)
        assert abs(a_o_gpu_choice - a_g_oracle_choice) <= REL * scale, \
            f"{what}: evicted {only_o[0]} (acc {a_o_gpu_choice}) instead of {only_g[0]} " \
            f"(acc {a_g_oracle_choice})"
        return "tie"
    oo, og = np.argsort(po), np.argsort(pg)
    assert np.array_equal(st.K[:c][oo], x["K"][og]), f"{what}: K rows differ"
    assert np.array_equal(st.V[:c][oo], x["V"][og]), f"{what}: V rows differ"
    ao, ag = st.acc[:c][oo], x["acc"][og]
    tol = REL * np.maximum(np.abs(ao), 1e-4 * max(np.abs(ao).max(initial=0.0), 1e-30))
    bad = np.abs(ag - ao) > tol
    assert not bad.any(), f"{what}: acc off at positions {po[oo][bad][:5]}: " \
                          f"{ag[bad][:5]} vs {ao[bad][:5]}"
    return None


def prefill_and_arena(torch, kvev, wl, growth):
    plan = kvev.Plan.from_workload(wl)
    lens = torch.from_numpy(np.asarray(wl.lens, np.int32)).cuda()
    dev = {l: gen.device_layer(wl, l) for l in range(wl.L)}
    bufs = plan.buffers(wl.B, wl.S_cap)
    plan.evict_prefill([dev[l][0] for l in range(wl.L)], [dev[l][1] for l in range(wl.L)],
                       [dev[l][2] for l in range(wl.L)], lens, wl.B, wl.S_cap, bufs)
    del dev
    arena = kvev.DecodeArena(plan, wl.B, growth)
    arena.init_from_prefill(bufs, lens)
    torch.cuda.synchronize()
    assert plan.status() == kvev.OK
    return plan, bufs, arena


def step_tokens(wl, step, layers):
    toks = {l: gen.device_decode_tokens(wl, step, l) for l in layers}
    k = [toks[l][0] if l in toks else None for l in range(wl.L)]
    v = [toks[l][1] if l in toks else None for l in range(wl.L)]
    q = [toks[l][2] if l in toks else None for l in range(wl.L)]
    return toks, k, v, q


def host_tokens(torch, toks, wl, units, g):
    kn, vn, qn = [], [], []
    cache = {}
    for i in units:
        l, s, h = g.units[i][:3]
        if l not in cache:
            cache[l] = tuple(t.view(torch.int16).cpu().numpy().view(np.uint16) for t in toks[l])
        k, v, q = cache[l]
        kn.append(k[s, h])
        vn.append(v[s, h])
        qn.append(q[s, h * wl.G:(h + 1) * wl.G])
    return kn, vn, qn


@pytest.mark.parametrize("d", [128, 64])
def test_decode_lockstep_mixed_rules(env, d):
    torch, kvev, orc = env
    wl = gen.config_decode_mixed(seed=3, d=d)
    growth = wl.decode_steps + 8
    plan, bufs, arena = prefill_and_arena(torch, kvev, wl, growth)
    g = Arena(torch, arena, wl)
    all_units = list(range(len(g.units)))
    states = [oracle_state(orc, wl, wl.route_decode, g, i) for i in all_units]
    layers = sorted({g.units[i][0] for i in all_units})
    ties = 0
    for step in range(wl.decode_steps):
        toks, k, v, q = step_tokens(wl, step, layers)
        arena.step(k, v, q)
        kn, vn, qn = host_tokens(torch, toks, wl, all_units, g)
        orc.decode_step(states, kn, vn, qn, wl.d, wl.G)
        g.refresh(torch)
        assert np.array_equal(g.lens, wl.lens + step + 1)
        for i in all_units:
            l, s, h = g.units[i][:3]
            x = g.unit(i)
            if compare_unit(states[i], x, f"step {step} layer {l} seq {s} head {h}") == "tie":
                ties += 1
                resync(states[i], x)
            # the reported eviction is the position that left the unit
            ev = int(g.evicted[g.units[i][3]])
            assert ev == -1 or ev not in set(x["pos"].tolist())
    assert plan.status() == kvev.OK
    assert ties <= len(all_units)  # near ties are rare; a flood would mean a real mismatch
    # every rule has done its job by the end
    for i in all_units:
        l, s = g.units[i][:2]
        x = g.unit(i)
        b, md = int(wl.budget[l]), int(wl.route_decode[l])
        n_now = int(wl.lens[s]) + wl.decode_steps
        if md == kvev.FULL:
            assert x["count"] == min(b, int(wl.lens[s])) + wl.decode_steps
        elif md == kvev.STREAMING:
            cap = wl.sink + b - wl.sink
            assert x["count"] == min(cap, n_now)
            assert set(range(wl.sink)) <= set(x["pos"].tolist())
            assert n_now - 1 in set(x["pos"].tolist())
        else:
            assert x["count"] == min(b, n_now)
            if md == kvev.H2O:  # decode tokens inside the protected window are retained
                r = b // 2
                first = max(n_now - r, int(wl.lens[s]))
                assert set(range(first, n_now)) <= set(x["pos"].tolist())


def _bf16_to_f64(u16):
    return (np.asarray(u16, np.uint32) << 16).view(np.float32).astype(np.float64)


def supplied_attention(torch, wl, g, toks, layers_attend):
    """Per H2O / TOVA layer, fp32 [B][H_kv][cap + 1]: the group-mean softmax of the
    new token's queries over the unit's slots (arena slot order) and the new
    token (last), in fp64 from the definition."""
    attn = {}
    host = {l: tuple(t.view(torch.int16).cpu().numpy().view(np.uint16) for t in toks[l]) for l in layers_attend}
    for i, (l, s, h, u, r0, cap) in enumerate(g.units):
        if l not in layers_attend:
            continue
        a = attn.setdefault(l, np.zeros((wl.B, wl.H_kv, cap + 1), np.float32))
        c = int(g.count[u])
        k, _, q = host[l]
        keys = np.concatenate([_bf16_to_f64(g.K[r0:r0 + c]), _bf16_to_f64(k[s, h])[None, :]], axis=0)
        qg = _bf16_to_f64(q[s, h * wl.G:(h + 1) * wl.G])
        x = qg @ keys.T / np.sqrt(wl.d)                 # [G][c + 1]
        pr = np.exp(x - x.max(axis=1, keepdims=True))
        pr /= pr.sum(axis=1, keepdims=True)
        a[s, h, :c + 1] = pr.mean(axis=0)
    return {l: torch.from_numpy(v).cuda() for l, v in attn.items()}


def test_decode_lockstep_supplied_attention(env):
    # kvev_decode_step_attn (the caller's decode attention supplies p) against
    # the oracle, which computes p from the queries itself: same rules, same
    # lock-step comparison as above.
    torch, kvev, orc = env
    wl = gen.config_decode_mixed(seed=5, d=128)
    growth = wl.decode_steps + 8
    plan, bufs, arena = prefill_and_arena(torch, kvev, wl, growth)
    g = Arena(torch, arena, wl)
    all_units = list(range(len(g.units)))
    states = [oracle_state(orc, wl, wl.route_decode, g, i) for i in all_units]
    layers = sorted({g.units[i][0] for i in all_units})
    attending = {l for l in layers if int(wl.route_decode[l]) in (kvev.H2O, kvev.TOVA)}
    assert attending
    ties = 0
    for step in range(wl.decode_steps):
        toks, k, v, q = step_tokens(wl, step, layers)
        attn = supplied_attention(torch, wl, g, toks, attending)
        arena.step_attn(k, v, [attn.get(l) for l in range(wl.L)])
        kn, vn, qn = host_tokens(torch, toks, wl, all_units, g)
        orc.decode_step(states, kn, vn, qn, wl.d, wl.G)
        g.refresh(torch)
        assert np.array_equal(g.lens, wl.lens + step + 1)
        for i in all_units:
            l, s, h = g.units[i][:3]
            x = g.unit(i)
            if compare_unit(states[i], x, f"step {step} layer {l} seq {s} head {h}") == "tie":
                ties += 1
                resync(states[i], x)
    assert plan.status() == kvev.OK
    assert ties <= len(all_units)


def test_decode_step_attn_rejects_missing_rows(env):
    torch, kvev, orc = env
    wl = gen.config_decode_mixed(seed=5, d=128)
    plan, bufs, arena = prefill_and_arena(torch, kvev, wl, 8)
    layers = [l for l in range(wl.L) if arena.layers[l][1] > 0]
    toks, k, v, q = step_tokens(wl, 0, layers)
    with pytest.raises(kvev.KvevError):
        arena.step_attn(k, v, [None] * wl.L)


def test_decode_full_size_sampled(env):
    """The decode workload at full size (batch 16, 16K caches compacted to 2048,
    32 layers): invariants on every unit over a few steps, and lock-step oracle
    parity on a sample of H2O, StreamingLLM and append-only units."""
    torch, kvev, orc = env
    wl = gen.config_decode(seed=1)
    steps, growth = 3, 8
    plan, bufs, arena = prefill_and_arena(torch, kvev, wl, growth)
    g = Arena(torch, arena, wl)
    rng = np.random.default_rng(5)
    by_rule = {}
    for i, (l, s, h, u, r0, cap) in enumerate(g.units):
        by_rule.setdefault(int(wl.route_decode[l]), []).append(i)
    sample = []
    for md, idx in by_rule.items():
        sample += [int(x) for x in rng.choice(idx, size=min(4, len(idx)), replace=False)]
    states = {i: oracle_state(orc, wl, wl.route_decode, g, i) for i in sample}
    layers = sorted({g.units[i][0] for i in range(len(g.units))})
    for step in range(steps):
        toks, k, v, q = step_tokens(wl, step, layers)
        arena.step(k, v, q)
        kn, vn, qn = host_tokens(torch, toks, wl, sample, g)
        orc.decode_step([states[i] for i in sample], kn, vn, qn, wl.d, wl.G)
        g.refresh(torch)
        for i in sample:
            l, s, h = g.units[i][:3]
            x = g.unit(i)
            if compare_unit(states[i], x, f"step {step} layer {l} seq {s} head {h}") == "tie":
                resync(states[i], x)
        for i, (l, s, h, u, r0, cap) in enumerate(g.units):
            c = int(g.count[u])
            b, md = int(wl.budget[l]), int(wl.route_decode[l])
            exp = b + step + 1 if md == kvev.FULL else b
            assert c == exp, (l, s, h, c, exp)
            p = g.pos[r0:r0 + c]
            assert len(np.unique(p)) == c and p.min() >= 0
            assert int(wl.lens[s]) + step in set(p.tolist()) or md in (kvev.TOVA,)
    assert plan.status() == kvev.OK


class SampledArena:
    """Host copies of a few units of a DecodeArena (the whole arena is several GB)."""

    def __init__(self, torch, arena, wl, units):
        self.a, self.wl, self.units = arena, wl, units  # units: [(l, s, h, u, r0, cap)]
        rows = np.concatenate([np.arange(r0, r0 + cap) for (_, _, _, _, r0, cap) in units])
        self.rows = torch.from_numpy(rows.astype(np.int64)).cuda()
        self.starts = np.cumsum([0] + [cap for (*_, cap) in units])
        self.uidx = torch.tensor([u for (_, _, _, u, _, _) in units], dtype=torch.int64).cuda()

    def refresh(self, torch):
        a = self.a
        self.K = a.K.view(torch.int16).index_select(0, self.rows).cpu().numpy().view(np.uint16)
        self.V = a.V.view(torch.int16).index_select(0, self.rows).cpu().numpy().view(np.uint16)
        self.pos = a.pos().index_select(0, self.rows).cpu().numpy()
        self.acc = a.acc().index_select(0, self.rows).cpu().numpy()
        self.count = a.count().index_select(0, self.uidx).cpu().numpy()
        self.lens = a.lens().cpu().numpy()

    def unit(self, i):
        c = int(self.count[i])
        sl = slice(self.starts[i], self.starts[i] + c)
        return {"count": c, "pos": self.pos[sl], "acc": self.acc[sl].astype(np.float64),
                "K": self.K[sl], "V": self.V[sl]}


def test_decode_all_steps_full_size(env):
    """The decode workload at its full length: batch 16, 16K caches compacted to
    2048 slots, 32 layers (H2O, StreamingLLM and append-only decode rules), all
    256 steps.  Every unit is checked on the device after every step (slot
    count, unique valid positions, the newest token, the sinks and the recent
    window of each rule); 32 sampled units (12 H2O, 10 StreamingLLM, 10
    append-only) are replayed in lock step by the oracle over all 256 steps."""
    torch, kvev, orc = env
    wl = gen.config_decode(seed=2)
    steps = wl.decode_steps
    assert steps == 256 and wl.B == 16
    growth = steps
    plan, bufs, arena = prefill_and_arena(torch, kvev, wl, growth)
    n0 = int(wl.lens[0])
    assert np.all(wl.lens == n0)
    units, layer_info = [], []
    for l, (off, cap, u0) in enumerate(arena.layers):
        if cap == 0:
            continue
        md, b = int(wl.route_decode[l]), int(wl.budget[l])
        layer_info.append((l, off, cap, u0, md, b))
        for s in range(wl.B):
            for h in range(wl.H_kv):
                i = s * wl.H_kv + h
                units.append((l, s, h, u0 + i, off + i * cap, cap))
    rng = np.random.default_rng(11)
    want = {kvev.H2O: 12, kvev.STREAMING: 10, kvev.FULL: 10}
    sample = []
    for md, k in want.items():
        idx = [i for i, un in enumerate(units) if int(wl.route_decode[un[0]]) == md]
        assert len(idx) >= k
        sample += [units[int(j)] for j in rng.choice(idx, size=k, replace=False)]
    g = SampledArena(torch, arena, wl, sample)
    g.refresh(torch)
    full_like = Arena.__new__(Arena)  # oracle_state reads units / unit() / lens from its argument
    full_like.units, full_like.unit, full_like.lens = sample, g.unit, g.lens
    states = [oracle_state(orc, wl, wl.route_decode, full_like, i) for i in range(len(sample))]
    layers = [li[0] for li in layer_info]
    exp_count = torch.zeros(arena.units, dtype=torch.int32, device="cuda")
    ties = 0
    for step in range(steps):
        toks, k, v, q = step_tokens(wl, step, layers)
        arena.step(k, v, q)
        # lock-step replay of the sampled units
        kn, vn, qn = host_tokens(torch, toks, wl, range(len(sample)), full_like)
        orc.decode_step(states, kn, vn, qn, wl.d, wl.G)
        g.refresh(torch)
        assert np.all(g.lens == n0 + step + 1)
        for i, (l, s, h, *_r) in enumerate(sample):
            if compare_unit(states[i], g.unit(i), f"step {step} layer {l} seq {s} head {h}") == "tie":
                ties += 1
                resync(states[i], g.unit(i))
        # every unit, on the device
        n = n0 + step + 1
        pos = arena.pos()
        for (l, off, cap, u0, md, b) in layer_info:
            c = b + step + 1 if md == kvev.FULL else b
            exp_count[u0: u0 + wl.B * wl.H_kv] = c
            P = torch.sort(pos[off: off + wl.B * wl.H_kv * cap].view(wl.B * wl.H_kv, cap), dim=1)[0]
            where = f"step {step} layer {l} rule {md}"
            assert bool((P[:, :cap - c] == -1).all()), where
            val = P[:, cap - c:]
            assert bool((val[:, 0] >= 0).all()) and bool((val[:, 1:] > val[:, :-1]).all()), where
            assert bool((val[:, -1] == n - 1).all()), where  # the newest token is kept
            ar = lambda lo, hi: torch.arange(lo, hi, dtype=torch.int32, device="cuda")[None, :]
            if md == kvev.STREAMING:
                assert bool((val[:, :wl.sink] == ar(0, wl.sink)).all()), where
                assert bool((val[:, wl.sink:] == ar(n - (c - wl.sink), n)).all()), where
            elif md == kvev.H2O:
                r = b // 2
                assert bool((val[:, c - r:] == ar(n - r, n)).all()), where
            else:
                assert bool((val[:, c - (step + 1):] == ar(n0, n)).all()), where
        assert torch.equal(arena.count(), exp_count), f"step {step}: counts"
    assert plan.status() == kvev.OK
    assert ties <= len(sample) * 4
    print("decode 256 steps: near-tie resyncs", ties)
