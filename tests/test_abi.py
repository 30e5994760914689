"""Host-side checks of the C ABI (no GPU needed, no kernel launched).

* the shared libraries load and export every symbol include/*.h declares,
  and the ctypes binding passes each the parameters its prototype lists;
* the library's allocator equals the oracle's bit for bit;
* plan validation, byte accounting (App. E worked example) and layer offsets;
* argument errors are reported before any device work.
"""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2606_15157_gb300 import inputs as gen

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def kv():
    from paper_2606_15157_gb300 import build, kvev
    build.build()
    kvev.load()
    return kvev


def declared(header, macro):
    txt = open(os.path.join(ROOT, "include", header)).read()
    return re.findall(macro + r"\s+[\w\s\*]*?\b(kvev_\w+)\s*\(", txt)


def test_libraries_export_every_declared_symbol(kv):
    names = declared("kvev.h", "KVEV_API")
    assert len(names) >= 10
    lib = C.CDLL(kv.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(kv.EXPORTS)
    synth = declared("kvev_synth.h", "KVEV_SYNTH_API")
    slib = C.CDLL(os.path.join(os.path.dirname(kv.LIB_PATH), "libkvev_synth.so"))
    assert len(synth) == 4
    for n in synth:
        assert hasattr(slib, n), n


def test_operator_ids_match_header(kv):
    txt = open(os.path.join(ROOT, "include", "kvev.h")).read()
    ids = dict(re.findall(r"#define KVEV_(FULL|SNAPKV|H2O|STREAMING|TOVA)\s+(\d+)", txt))
    assert {k: int(v) for k, v in ids.items()} == {
        "FULL": kv.FULL, "SNAPKV": kv.SNAPKV, "H2O": kv.H2O, "STREAMING": kv.STREAMING, "TOVA": kv.TOVA}
    assert (gen.FULL, gen.SNAPKV, gen.H2O, gen.STREAMING) == (kv.FULL, kv.SNAPKV, kv.H2O, kv.STREAMING)


def test_allocator_matches_oracle_bit_exact(kv, orc):
    rng = np.random.default_rng(11)
    for trial in range(500):
        L = int(rng.integers(1, 80))
        b_min = int(rng.integers(0, 100))
        B = L * b_min + int(rng.integers(0, 100000))
        kind = trial % 4
        if kind == 0:
            s = rng.gamma(0.3, size=L)
        elif kind == 1:
            s = rng.standard_normal(L)            # non-positive values: shift rule
        elif kind == 2:
            s = np.round(rng.random(L) * 4) / 4    # many exact ties
        else:
            s = np.exp(rng.standard_normal(L) * 3)  # outliers for the Q95 cap
        for T in (kv.T_IDENTITY, kv.T_CAP_Q95):
            a = kv.alloc_from_scores(s, B, b_min, T)
            b = orc.alloc_from_scores(s, B, b_min, T)
            assert a.tolist() == b.tolist(), (trial, T)
    for trial in range(200):
        b_in = rng.integers(1, 4000, size=int(rng.integers(1, 64))).astype(np.int32)
        T = int(rng.integers(0, 200000))
        assert kv.alloc_rescale(b_in, T).tolist() == orc.alloc_rescale(b_in, T).tolist()


def test_workload_budgets(kv, orc):
    # Pyramidal (decreasing with depth) and Dirichlet allocations of the
    # synthetic workloads: exact totals, b_min respected, same on both sides.
    al = lambda f: (lambda s, B, m, t: f(s, B, m, t))
    for bbar in (128, 256, 512, 1024, 2048):
        wk = gen.config_hetero8k(kv.alloc_from_scores, bbar=bbar)
        wo = gen.config_hetero8k(orc.alloc_from_scores, bbar=bbar)
        assert wk.budget.tolist() == wo.budget.tolist()
        assert wk.budget.sum() == 32 * bbar and wk.budget.min() >= 48
        assert np.all(np.diff(wk.budget) <= 0)
        assert (wk.route == gen.SNAPKV).sum() == 18 and (wk.route == gen.H2O).sum() == 7
    wk = gen.config_long(kv.alloc_from_scores)
    wo = gen.config_long(orc.alloc_from_scores)
    assert wk.budget.tolist() == wo.budget.tolist()
    assert wk.budget.sum() == 32 * 1024 and wk.budget.min() >= 80
    assert np.all((wk.lens >= 16384) & (wk.lens <= 32768))


def test_plan_validation(kv):
    ok = dict(L=2, H_q=8, H_kv=2, d=128, route_prefill=[kv.SNAPKV, kv.STREAMING],
              route_decode=None, budget=[64, 64], window=32, pool_kernel=7, pool_type=kv.POOL_AVG,
              sink=4, recent=-1, h2o_recent=-1)
    h = kv.kvev_plan_create(**ok)
    kv.kvev_plan_destroy(h)

    def bad(code, **kw):
        args = dict(ok)
        args.update(kw)
        with pytest.raises(kv.KvevError) as e:
            kv.kvev_plan_create(**args)
        assert e.value.code == code

    bad(kv.EINVAL, budget=[32, 64])                       # SnapKV b <= W
    bad(kv.EINVAL, budget=[64, 4])                        # StreamingLLM b <= sink
    bad(kv.EINVAL, pool_kernel=4)                         # even pooling width
    bad(kv.EINVAL, H_q=7)                                 # H_q not a multiple of H_kv
    bad(kv.EINVAL, route_prefill=[kv.H2O, 9])             # unknown operator
    bad(kv.EINVAL, route_prefill=[kv.H2O, kv.STREAMING], h2o_recent=100)  # r > b
    bad(kv.EINVAL, route_decode=[kv.SNAPKV, kv.FULL])     # SnapKV is not a decode operator
    bad(kv.ENOTSUP, d=96)                                 # scoring needs d in {64, 128}
    bad(kv.ENOTSUP, window=128, budget=[200, 64])         # G*W = 512 > 256
    # FULL layers ignore their budget; StreamingLLM needs no window
    h = kv.kvev_plan_create(**dict(ok, route_prefill=[kv.FULL, kv.STREAMING], budget=[0, 64],
                                   window=0))
    kv.kvev_plan_destroy(h)


def test_app_e_byte_accounting(kv):
    # App. E: 32 layers x 512 retained tokens, 8 KV heads, d=128, bf16 K and V
    # -> 16,384 layer-token positions, 64.00 MiB of exact KV state.
    h = kv.kvev_plan_create(32, 32, 8, 128, [kv.H2O] * 32, None, [512] * 32, 32, 7, kv.POOL_AVG, 4)
    kv_bytes, idx_bytes, cnt_bytes, ws = kv.kvev_plan_query(h, 1, 32768)
    assert idx_bytes // 4 == 16384 * 8
    assert 2 * kv_bytes == 64 * 2 ** 20
    assert cnt_bytes == 32 * 8 * 4
    assert kv.kvev_plan_layer_offset(h, 1, 0) == 0
    assert kv.kvev_plan_layer_offset(h, 1, 5) == 5 * 512 * 8
    assert kv.kvev_plan_layer_offset(h, 3, 5) == 5 * 512 * 8 * 3
    kv.kvev_plan_destroy(h)


def test_layer_offsets_skip_full_layers(kv):
    routes = [kv.FULL, kv.SNAPKV, kv.FULL, kv.STREAMING, kv.H2O, kv.FULL]
    budget = [999, 100, 999, 50, 70, 999]
    h = kv.kvev_plan_create(6, 4, 2, 64, routes, None, budget, 16, 5, kv.POOL_MAX, 4)
    B, H = 3, 2
    exp = [0, 0, 100 * B * H, 100 * B * H, 150 * B * H, 220 * B * H]
    assert [kv.kvev_plan_layer_offset(h, B, l) for l in range(6)] == exp
    kv_bytes, idx_bytes, _, _ = kv.kvev_plan_query(h, B, 4096)
    assert idx_bytes // 4 == 220 * B * H and kv_bytes == 220 * B * H * 64 * 2
    with pytest.raises(kv.KvevError):
        kv.kvev_plan_scores_offset(h, B, 4096, 3)   # StreamingLLM layer has no scores
    o1 = kv.kvev_plan_scores_offset(h, B, 4096, 1)
    o4 = kv.kvev_plan_scores_offset(h, B, 4096, 4)
    assert o4 - o1 == 4 * B * H * 4096
    kv.kvev_plan_destroy(h)


def test_evict_argument_errors_before_device_work(kv):
    h = kv.kvev_plan_create(2, 4, 2, 64, [kv.SNAPKV, kv.STREAMING], None, [64, 64], 8, 5,
                            kv.POOL_MAX, 4)
    fake = 1 << 20
    args = dict(handle=h, K_ptrs=[fake, fake], V_ptrs=[fake, fake], Q_ptrs=[fake, fake],
                lens_ptr=fake, B=1, S_cap=512, out_K=fake, out_V=fake, out_idx=fake,
                out_count=fake, h2o_state=None, workspace=fake, workspace_bytes=1 << 30, stream=None)
    assert kv.kvev_evict_prefill(**dict(args, B=-1)) == kv.EINVAL
    assert kv.kvev_evict_prefill(**dict(args, S_cap=0)) == kv.EINVAL
    assert kv.kvev_evict_prefill(**dict(args, K_ptrs=[fake + 8, fake])) == kv.EINVAL   # misaligned
    assert kv.kvev_evict_prefill(**dict(args, Q_ptrs=[None, fake])) == kv.EINVAL      # SnapKV needs Q
    assert kv.kvev_evict_prefill(**dict(args, workspace=fake + 16)) == kv.EINVAL      # 256-B alignment
    assert kv.kvev_evict_prefill(**dict(args, workspace_bytes=64)) == kv.ENOMEM
    assert kv.kvev_evict_prefill(**dict(args, B=0)) == kv.OK                          # nothing to do
    # caller-supplied scores: the array itself is required; with a layer's scores given, its Q_win
    # is not, but they must be 4-byte aligned
    sargs = dict(args, score_ptrs=[None, None])
    assert kv.kvev_evict_prefill_scored(**dict(sargs, score_ptrs=None)) == kv.EINVAL
    assert kv.kvev_evict_prefill_scored(**dict(sargs, Q_ptrs=[None, fake])) == kv.EINVAL
    assert kv.kvev_evict_prefill_scored(**dict(sargs, Q_ptrs=[None, fake], score_ptrs=[fake + 2, None])) == kv.EINVAL
    assert kv.kvev_evict_prefill_scored(**dict(sargs, Q_ptrs=[None, fake], score_ptrs=[fake, None],
                                                workspace_bytes=64)) == kv.ENOMEM  # past the checks
    # caller-supplied normalisers: required for the scoring layer (layer 0), 4-byte aligned;
    # the StreamingLLM layer's entry is ignored
    largs = dict(args, lse_ptrs=[fake, None])
    assert kv.kvev_evict_prefill_lse(**dict(largs, lse_ptrs=None)) == kv.EINVAL
    assert kv.kvev_evict_prefill_lse(**dict(largs, lse_ptrs=[None, fake])) == kv.EINVAL
    assert kv.kvev_evict_prefill_lse(**dict(largs, lse_ptrs=[fake + 2, None])) == kv.EINVAL
    assert kv.kvev_evict_prefill_lse(**dict(largs, Q_ptrs=[None, fake])) == kv.EINVAL  # Q_win still read
    assert kv.kvev_evict_prefill_lse(**dict(largs, workspace_bytes=64)) == kv.ENOMEM   # past the checks
    assert kv.kvev_evict_prefill_lse(**dict(largs, B=0)) == kv.OK
    kv.kvev_plan_destroy(h)


def test_decode_step_argument_errors(kv):
    # both decode entry points validate before any device work: the supplied-attention
    # form needs an attention row array for its H2O / TOVA layers instead of q_new
    wl = gen.config_decode_mixed()
    plan = kv.Plan.from_workload(wl)
    fake = 1 << 20
    L = wl.L
    step = dict(handle=plan.handle, B=wl.B, growth=8, dec_K=fake, dec_V=fake, dec_state=fake,
                k_ptrs=[fake] * L, v_ptrs=[fake] * L, stream=None)
    assert kv.kvev_decode_step(**step, q_ptrs=[None] * L) == kv.EINVAL
    assert kv.kvev_decode_step(**dict(step, dec_state=fake + 16), q_ptrs=[fake] * L) == kv.EINVAL
    assert kv.kvev_decode_step_attn(**step, attn_ptrs=[None] * L) == kv.EINVAL
    assert kv.kvev_decode_step_attn(**step, attn_ptrs=[fake + 2] * L) == kv.EINVAL
    assert kv.kvev_decode_step_attn(**dict(step, B=0), attn_ptrs=[fake] * L) == kv.OK
    plan.close()


def test_decode_arena_layout(kv):
    wl = gen.config_decode_mixed()
    plan = kv.Plan.from_workload(wl)
    B, growth, H = wl.B, 32, wl.H_kv
    rows, state = kv.kvev_decode_query(plan.handle, B, growth)
    caps, row_offs, unit_offs = [], [], []
    for l in range(wl.L):
        off, cap, u0 = kv.kvev_decode_layer(plan.handle, B, growth, l)
        row_offs.append(off)
        caps.append(cap)
        unit_offs.append(u0)
    # evicting decode rules keep b slots, append-only layers b + growth
    exp_caps = [int(wl.budget[l]) + (growth if wl.route_decode[l] == kv.FULL else 0)
                for l in range(wl.L)]
    assert caps == exp_caps
    assert row_offs == list(np.cumsum([0] + [B * H * c for c in exp_caps])[:-1])
    assert unit_offs == [B * H * l for l in range(wl.L)]
    assert rows == sum(B * H * c for c in exp_caps)
    offs = kv.kvev_decode_state_offsets(plan.handle, B, growth)
    units = wl.L * B * H
    assert offs["lens"] == 0 and all(v % 256 == 0 for v in offs.values())
    assert offs["count"] >= 4 * B and offs["evicted"] >= offs["count"] + 4 * units
    assert offs["pos"] >= offs["evicted"] + 4 * units and offs["acc"] >= offs["pos"] + 4 * rows
    assert state >= offs["acc"] + 4 * rows
    plan.close()


def test_decode_layout_rejects_rules_without_a_retained_cache(kv):
    # a FULL prefill layer keeps the caller's own cache: no decode-phase rule on it
    h = kv.kvev_plan_create(2, 4, 2, 64, [kv.FULL, kv.H2O], [kv.H2O, kv.H2O], [64, 64], 8, 5,
                            kv.POOL_MAX, 4)
    with pytest.raises(kv.KvevError):
        kv.kvev_decode_query(h, 1, 0)
    kv.kvev_plan_destroy(h)
    h = kv.kvev_plan_create(2, 4, 2, 64, [kv.FULL, kv.H2O], [kv.FULL, kv.TOVA], [64, 64], 8, 5,
                            kv.POOL_MAX, 4)
    rows, _ = kv.kvev_decode_query(h, 3, 10)
    assert rows == 3 * 2 * 64   # the FULL layer has no arena, TOVA keeps b slots
    fake = 1 << 20
    assert kv.kvev_decode_step(h, 3, 10, fake, fake, fake + 16, [None, fake], [None, fake],
                               [None, fake], None) == kv.EINVAL   # state must be 256-B aligned
    assert kv.kvev_decode_step(h, 3, 10, fake, fake, fake, [None, fake], [None, fake],
                               [None, None], None) == kv.EINVAL   # TOVA needs the queries
    assert kv.kvev_decode_step(h, 0, 10, fake, fake, fake, [None, fake], [None, fake],
                               [None, fake], None) == kv.OK       # nothing to do
    kv.kvev_plan_destroy(h)


def _prototypes(header, macro):
    """{name: [parameter declarations]} of every function the header declares."""
    txt = open(os.path.join(ROOT, "include", header)).read()
    txt = re.sub(r"/\*.*?\*/", " ", txt, flags=re.S)
    txt = re.sub(r"//[^\n]*", " ", txt)
    out = {}
    for m in re.finditer(macro + r"\s+[\w\s\*]*?\b(kvev_\w+)\s*\(([^)]*)\)\s*;", txt):
        params = [p.strip() for p in m.group(2).split(",") if p.strip()]
        out[m.group(1)] = [] if params == ["void"] else params
    return out


def _kind(decl):
    """The ctypes class a C parameter declaration marshals to."""
    if "*" in decl:
        return "ptr"
    t = decl.rsplit(None, 1)[0] if len(decl.split()) > 1 else decl
    return {"int": "i32", "int32_t": "i32", "int64_t": "i64", "size_t": "size",
            "double": "f64", "float": "f32"}[t.replace("const ", "").strip()]


def test_binding_argtypes_match_header(kv):
    # every prototype in kvev.h against the ctypes signature the binding
    # installs: same number of parameters, and each of the same kind (pointer,
    # 32- or 64-bit integer, size_t, double, float) on both sides
    protos = _prototypes("kvev.h", "KVEV_API")
    assert set(protos) == set(kv.EXPORTS)
    lib = kv.load()
    ct = {C.c_void_p: "ptr", C.c_int: "i32", C.c_int32: "i32", C.c_int64: "i64", C.c_size_t: "size",
          C.c_double: "f64", C.c_float: "f32"}
    for name, params in protos.items():
        argtypes = getattr(lib, name).argtypes
        assert argtypes is not None and len(argtypes) == len(params), name
        for decl, a in zip(params, argtypes):
            got = "ptr" if (isinstance(a, type) and issubclass(a, C._Pointer)) else ct.get(a)
            want = _kind(decl)
            # size_t and int64_t are both 64-bit on the supported (LP64) hosts
            assert got == want or {got, want} == {"i64", "size"}, (name, decl, a)
