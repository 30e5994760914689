"""Seeded synthetic inputs for the eviction path (shared by the GPU path and the oracle).

This module holds none of the eviction arithmetic: it only draws the synthetic
KV caches, window queries, lengths, routes and allocation scores that stand in
for the paper's LongBench/RULER workloads on LLaMA-3.1-8B-Instruct (Sec. 4.1,
App. E), whose data and weights are not available.  Only the shapes come from
the paper: 32 layers, 32 query / 8 KV heads, head_dim 128, contexts 4K-32K,
budgets 128-2048 tokens per layer.

Every value is a pure function of (seed, tensor, layer, flat element index)
through one counter-based generator, so the host (numpy, here) and the device
(``csrc/synth.cu``) produce bit-identical tensors:

* ``mix64`` is SplitMix64's output function (Steele, Lea & Flood, 2014) applied
  to ``key + (i + 1) * 0x9E3779B97F4A7C15``; ``key`` is derived from the seed,
  a tensor id and the layer by two more SplitMix64 rounds.
* Gaussian-like values: the sum of the four 16-bit fields of one hash (an
  Irwin-Hall(4) variate, exact in integers), centred, converted to fp32 and
  multiplied by 1/sqrt(Var) in fp32 -- mean 0, variance 1, support +-3.46.
  Only exact or correctly rounded fp32 operations are used (no libm), then
  round-to-nearest-even to bf16.
* V rows are raw hash bits with the exponent kept finite; they are only ever
  copied, never used in arithmetic.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

GAMMA = 0x9E3779B97F4A7C15
M1 = 0xBF58476D1CE4E5B9
M2 = 0x94D049BB133111EB
MASK64 = (1 << 64) - 1

# Tensor ids of the generator streams.
T_K, T_V, T_Q, T_U, T_KNEW, T_VNEW, T_QNEW, T_HOST = 1, 2, 3, 4, 5, 6, 7, 8

IH4_MEAN = 131070                       # 4 * 32767.5
IH4_SCALE = np.float32(1.0 / 37837.226)  # 1 / sqrt(4 * (65536^2 - 1) / 12)

# Operator ids as the GPU library numbers them (kept in sync by tests).
FULL, SNAPKV, H2O, STREAMING, TOVA = 0, 1, 2, 3, 4
POOL_MAX, POOL_AVG = 0, 1


def _mix_int(x: int) -> int:
    z = (x + GAMMA) & MASK64
    z = ((z ^ (z >> 30)) * M1) & MASK64
    z = ((z ^ (z >> 27)) * M2) & MASK64
    return z ^ (z >> 31)


def stream_key(seed: int, tensor: int, layer: int) -> int:
    """64-bit key of one generator stream."""
    return _mix_int(_mix_int(seed & MASK64) ^ (((tensor & 0xFFFF) << 32) | (layer & 0xFFFFFFFF)))


def hash64(key: int, idx: np.ndarray) -> np.ndarray:
    """SplitMix64 output for counters key + (idx+1)*GAMMA (uint64, vectorised)."""
    with np.errstate(over="ignore"):
        z = np.uint64(key) + (idx.astype(np.uint64) + np.uint64(1)) * np.uint64(GAMMA)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(M1)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(M2)
        z = z ^ (z >> np.uint64(31))
    return z


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16, nearest-even (inputs are finite)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def gauss_f32(key: int, idx: np.ndarray) -> np.ndarray:
    """Irwin-Hall(4) standardised value in fp32 for each counter."""
    h = hash64(key, idx)
    s = ((h & np.uint64(0xFFFF)) + ((h >> np.uint64(16)) & np.uint64(0xFFFF)) +
         ((h >> np.uint64(32)) & np.uint64(0xFFFF)) + (h >> np.uint64(48)))
    c = (s.astype(np.int64) - IH4_MEAN).astype(np.float32)  # exact: |c| < 2^18
    return c * IH4_SCALE


def gauss_bf16(key: int, idx: np.ndarray) -> np.ndarray:
    return f32_to_bf16_bits(gauss_f32(key, idx))


def value_bits(key: int, idx: np.ndarray) -> np.ndarray:
    """Arbitrary finite bf16 bit patterns (exponent 0xFF is lowered to 0xFE)."""
    b = (hash64(key, idx) & np.uint64(0xFFFF)).astype(np.uint16)
    inf_exp = (b & np.uint16(0x7F80)) == np.uint16(0x7F80)
    b[inf_exp] &= np.uint16(0xFF7F)
    return b


# --------------------------------------------------------------------------
# Small host-side scalar draws (lengths, routes, allocation scores)
# --------------------------------------------------------------------------

def uniform01(seed: int, tensor: int, i: int) -> float:
    """A double in (0, 1) from the top 53 bits of one hash."""
    h = int(hash64(stream_key(seed, tensor, 0), np.array([i], dtype=np.uint64))[0])
    return ((h >> 11) + 0.5) * (1.0 / (1 << 53))


def ragged_lengths(seed: int, B: int, lo: int, hi: int) -> np.ndarray:
    """Lengths uniform on the integers [lo, hi]."""
    key = stream_key(seed, T_HOST, 1)
    h = hash64(key, np.arange(B, dtype=np.uint64))
    return (lo + (h % np.uint64(hi - lo + 1)).astype(np.int64)).astype(np.int32)


def block_route(seed: int, counts: dict[int, int]) -> np.ndarray:
    """Contiguous blocks of operators; the block order is a seeded permutation."""
    ops = list(counts.keys())
    keys = [uniform01(seed, T_HOST, 100 + j) for j in range(len(ops))]
    order = [ops[j] for j in np.argsort(keys, kind="stable")]
    route = []
    for op in order:
        route += [op] * counts[op]
    return np.array(route, dtype=np.int32)


def dirichlet_scores(seed: int, L: int) -> np.ndarray:
    """Dirichlet(1, ..., 1) draw over L layers via normalised Exp(1) variates."""
    e = np.array([-math.log(uniform01(seed, T_HOST, 1000 + l)) for l in range(L)])
    return e / e.sum()


def pyramid_weights(L: int) -> np.ndarray:
    """Linearly decreasing per-layer weights, 1.5 at the first layer to 0.5 at the last."""
    if L == 1:
        return np.ones(1)
    return 1.5 - np.arange(L, dtype=np.float64) / (L - 1)


# --------------------------------------------------------------------------
# Workload descriptions
# --------------------------------------------------------------------------

@dataclass
class Workload:
    """One synthetic eviction workload (shapes, route, budgets, recipe)."""
    name: str
    L: int
    H_q: int
    H_kv: int
    d: int
    B: int
    lens: np.ndarray
    S_cap: int
    W: int
    pool_kernel: int
    pool_type: int
    route: np.ndarray              # prefill operator per layer
    budget: np.ndarray             # nominal capacity per layer
    sink: int = 4
    recent: int = -1
    h2o_recent: int = -1
    seed: int = 0
    sink_tokens: int = 0           # first positions whose keys are scaled by sink_scale
    sink_scale: float = 4.0
    plant: dict | None = None      # planted attention patterns (see plant_recipe)
    route_decode: np.ndarray | None = None
    decode_steps: int = 0
    notes: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def G(self) -> int:
        return self.H_q // self.H_kv


def config_tiny(seed: int = 0) -> Workload:
    """4 layers, GQA 4/2 heads, d=64, batch 1, n=512, W=8, max-pool 5, b=64."""
    return Workload(
        name="tiny", L=4, H_q=4, H_kv=2, d=64, B=1, lens=np.array([512], np.int32), S_cap=512,
        W=8, pool_kernel=5, pool_type=POOL_MAX,
        route=np.array([SNAPKV, STREAMING, H2O, SNAPKV], np.int32),
        budget=np.array([64, 64, 64, 64], np.int32), sink=4, recent=60, seed=seed,
        sink_tokens=4, sink_scale=4.0)


def support_size(l: int, L: int) -> int:
    """Planted support size of layer l: 16 at the first layer to 1600 at the last."""
    return int(round(16.0 * 100.0 ** (l / max(L - 1, 1))))


def plant_recipe(seed: int, L: int, n: int, W: int) -> dict:
    """Per-layer planted set [start, start+size): recent-focused, mid-context band or
    prefix-focused, cycling in blocks of 4 layers; gamma sets the key alignment."""
    starts, sizes, gammas = [], [], []
    for l in range(L):
        s = support_size(l, L)
        kind = (l // 4) % 3
        E = n - W
        if kind == 0:        # recent-focused: the last s prefix positions
            st = E - s
        elif kind == 1:      # mid-context band at a seeded position
            lo, hi = E // 4, (3 * E) // 4 - s
            st = lo + int(uniform01(seed, T_HOST, 2000 + l) * max(hi - lo, 1))
        else:                # prefix-focused, just after the sink tokens
            st = 4
        # attention logit gap that puts ~95% of the mass on the planted set, so
        # that the smallest set covering 90% of it is most of the planted set
        gap = math.log(19.0 * (n - s) / s)
        gammas.append(np.float32(gap * math.sqrt(128.0) / 4.0))
        starts.append(st)
        sizes.append(s)
    return {"start": np.array(starts, np.int32), "size": np.array(sizes, np.int32),
            "gamma": np.array(gammas, np.float32), "alpha": np.float32(4.0)}


def config_homog8k(seed: int = 0) -> Workload:
    L, n, W = 32, 8192, 32
    return Workload(
        name="homog_snapkv_8k", L=L, H_q=32, H_kv=8, d=128, B=1, lens=np.array([n], np.int32),
        S_cap=n, W=W, pool_kernel=7, pool_type=POOL_AVG,
        route=np.full(L, SNAPKV, np.int32), budget=np.full(L, 512, np.int32), seed=seed,
        plant=plant_recipe(seed, L, n, W))


HETERO_COUNTS = {SNAPKV: 18, H2O: 7, STREAMING: 7}


def config_hetero8k(alloc, seed: int = 0, bbar: int = 512) -> Workload:
    """Heterogeneous contiguous-block route, pyramidal allocation (decreasing with depth).

    ``alloc(s, B_total, b_min, transform)`` is the caller's allocator (the library's
    for the GPU side, the oracle's for the reference side)."""
    L, n, W = 32, 8192, 32
    budget = np.asarray(alloc(pyramid_weights(L), L * bbar, max(48, W + 16), 0), np.int32)
    return Workload(
        name=f"hetero_8k_b{bbar}", L=L, H_q=32, H_kv=8, d=128, B=1,
        lens=np.array([n], np.int32), S_cap=n, W=W, pool_kernel=7, pool_type=POOL_AVG,
        route=block_route(seed, HETERO_COUNTS), budget=budget, sink=4, seed=seed,
        sink_tokens=4, sink_scale=4.0)


def config_long(alloc, seed: int = 0, fixed_len: int | None = None) -> Workload:
    """Batch 8, ragged lengths uniform in [16384, 32768], W=64, Dirichlet allocation.

    ``alloc`` as for :func:`config_hetero8k`."""
    L, B, W = 32, 8, 64
    lens = (np.full(B, fixed_len, np.int32) if fixed_len else ragged_lengths(seed, B, 16384, 32768))
    s = dirichlet_scores(seed, L)
    budget = np.asarray(alloc(s, L * 1024, max(48, W + 16), 0), np.int32)
    return Workload(
        name="long_b8_16k-32k" if fixed_len is None else f"long_b8_{fixed_len}",
        L=L, H_q=32, H_kv=8, d=128, B=B, lens=lens, S_cap=32768, W=W, pool_kernel=7,
        pool_type=POOL_AVG, route=block_route(seed, HETERO_COUNTS), budget=budget, sink=4,
        seed=seed, sink_tokens=4, sink_scale=4.0, extra={"scores": s})


def config_decode(seed: int = 0, B: int = 16, n0: int = 16384, steps: int = 256,
                  budget: int = 2048) -> Workload:
    """Prefill-compact n0-token caches to `budget`, then `steps` decode steps."""
    L, W = 32, 32
    route = block_route(seed, HETERO_COUNTS)
    dec = np.where(route == SNAPKV, FULL, route).astype(np.int32)  # SnapKV is prefill-only
    return Workload(
        name=f"decode_b{B}_{n0}_to_{budget}", L=L, H_q=32, H_kv=8, d=128, B=B,
        lens=np.full(B, n0, np.int32), S_cap=n0, W=W, pool_kernel=7, pool_type=POOL_AVG,
        route=route, budget=np.full(L, budget, np.int32), sink=4, seed=seed,
        sink_tokens=4, sink_scale=4.0, route_decode=dec, decode_steps=steps)


def config_decode_mixed(seed: int = 0, steps: int = 24, d: int = 128) -> Workload:
    """Every decode-phase rule at a size the oracle replays step by step: 8 layers,
    GQA 8/2 heads, batch 2 with ragged lengths, W=16.  Prefill -> decode rules:
    SnapKV->append, H2O->H2O, StreamingLLM->StreamingLLM, H2O->TOVA, SnapKV->TOVA,
    StreamingLLM->append, H2O (budget above the length: identity prefill, the
    decode cache fills up to b first)->H2O, SnapKV->H2O (acc starts at 0)."""
    route = np.array([SNAPKV, H2O, STREAMING, H2O, SNAPKV, STREAMING, H2O, SNAPKV], np.int32)
    dec = np.array([FULL, H2O, STREAMING, TOVA, TOVA, FULL, H2O, H2O], np.int32)
    budget = np.array([256, 192, 128, 160, 200, 96, 3000, 144], np.int32)
    return Workload(
        name=f"decode_mixed_d{d}", L=8, H_q=8, H_kv=2, d=d, B=2,
        lens=np.array([2990, 2731], np.int32), S_cap=3072, W=16, pool_kernel=7,
        pool_type=POOL_AVG, route=route, budget=budget, sink=4, seed=seed, sink_tokens=4,
        sink_scale=4.0, route_decode=dec, decode_steps=steps)


# --------------------------------------------------------------------------
# Host tensor generation (small and sampled cases)
# --------------------------------------------------------------------------

def _unit_u(wl: Workload, layer: int, h: int) -> np.ndarray:
    """Planted direction of (layer, kv head): a N(0, I) draw scaled to unit norm in fp32.
    The norm is exact (fsum in double), so every head's planted logit gap is the
    recipe's gap, not gap * |u|^2 with |u|^2 spread by about +-12% at d = 128."""
    idx = np.arange(h * wl.d, (h + 1) * wl.d, dtype=np.uint64)
    x = gauss_f32(stream_key(wl.seed, T_U, layer), idx)
    norm = math.sqrt(math.fsum(float(v) * float(v) for v in x))
    return x * np.float32(1.0 / norm)


def k_rows(wl: Workload, layer: int, s: int, h: int, pos: np.ndarray) -> np.ndarray:
    """K rows (bf16 bits) of positions `pos` of (layer, seq s, kv head h)."""
    d = wl.d
    base = ((s * wl.H_kv + h) * wl.S_cap + pos.astype(np.int64)) * d
    idx = (base[:, None] + np.arange(d)[None, :]).astype(np.uint64)
    x = gauss_f32(stream_key(wl.seed, T_K, layer), idx.ravel()).reshape(len(pos), d)
    if wl.sink_tokens:
        m = pos < wl.sink_tokens
        x[m] = x[m] * np.float32(wl.sink_scale)
    if wl.plant is not None:
        st, sz = int(wl.plant["start"][layer]), int(wl.plant["size"][layer])
        m = (pos >= st) & (pos < st + sz)
        if m.any():
            u = _unit_u(wl, layer, h)
            g = wl.plant["gamma"][layer]
            x[m] = x[m] + (np.float32(g) * u)[None, :]
    return f32_to_bf16_bits(x)


def v_rows(wl: Workload, layer: int, s: int, h: int, pos: np.ndarray) -> np.ndarray:
    d = wl.d
    base = ((s * wl.H_kv + h) * wl.S_cap + pos.astype(np.int64)) * d
    idx = (base[:, None] + np.arange(d)[None, :]).astype(np.uint64)
    return value_bits(stream_key(wl.seed, T_V, layer), idx.ravel()).reshape(len(pos), d)


def q_group(wl: Workload, layer: int, s: int, h: int) -> np.ndarray:
    """Window queries of the G heads of KV group h: uint16 [G][W][d]."""
    G, W, d = wl.G, wl.W, wl.d
    hq0 = h * G
    base = (((s * wl.H_q + hq0 + np.arange(G))[:, None] * W + np.arange(W)[None, :]) * d)
    idx = (base[:, :, None] + np.arange(d)[None, None, :]).astype(np.uint64)
    x = gauss_f32(stream_key(wl.seed, T_Q, layer), idx.ravel()).reshape(G, W, d)
    if wl.plant is not None:
        u = _unit_u(wl, layer, h)
        x = (wl.plant["alpha"] * u)[None, None, :] + np.float32(0.1) * x
    return f32_to_bf16_bits(x.reshape(-1, d)).reshape(G, W, d)


def host_tensors(wl: Workload, layers=None):
    """Full host tensors per layer: K, V [B][H_kv][S_cap][d] and Q [B][H_q][W][d] (uint16)."""
    layers = range(wl.L) if layers is None else layers
    out = {}
    pos = np.arange(wl.S_cap, dtype=np.int64)
    for l in layers:
        K = np.zeros((wl.B, wl.H_kv, wl.S_cap, wl.d), np.uint16)
        V = np.zeros_like(K)
        Q = np.zeros((wl.B, wl.H_q, wl.W, wl.d), np.uint16)
        for s in range(wl.B):
            for h in range(wl.H_kv):
                K[s, h] = k_rows(wl, l, s, h, pos)
                V[s, h] = v_rows(wl, l, s, h, pos)
                Q[s, h * wl.G:(h + 1) * wl.G] = q_group(wl, l, s, h)
        out[l] = (K, V, Q)
    return out


def decode_token(wl: Workload, step: int, layer: int, s: int, h: int):
    """New token of decode step `step`: k, v [d] and the G query rows [G][d]."""
    d = wl.d
    row = ((step * wl.B + s) * wl.H_kv + h)
    idx = (row * d + np.arange(d)).astype(np.uint64)
    k = gauss_bf16(stream_key(wl.seed, T_KNEW, layer), idx)
    v = value_bits(stream_key(wl.seed, T_VNEW, layer), idx)
    qrow = ((step * wl.B + s) * wl.H_q + h * wl.G + np.arange(wl.G))
    qidx = (qrow[:, None] * d + np.arange(d)[None, :]).astype(np.uint64)
    q = gauss_bf16(stream_key(wl.seed, T_QNEW, layer), qidx.ravel()).reshape(wl.G, d)
    return k, v, q


# --------------------------------------------------------------------------
# Device tensor generation (full-size workloads), bit-identical to the above
# --------------------------------------------------------------------------

_synth = None


def synth_lib():
    """ctypes handle of libkvev_synth.so (raises if it was not built)."""
    global _synth
    if _synth is None:
        import ctypes as C
        import os
        path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "lib", "libkvev_synth.so")
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build()")
        lib = C.CDLL(path)
        vp, i, u64, f = C.c_void_p, C.c_int, C.c_uint64, C.c_float
        lib.kvev_synth_k.argtypes = [vp, i, i, i, i, u64, i, f, i, i, f, vp, vp]
        lib.kvev_synth_q.argtypes = [vp, i, i, i, i, i, u64, f, vp, vp]
        lib.kvev_synth_gauss.argtypes = [vp, u64, u64, u64, vp]
        lib.kvev_synth_bits.argtypes = [vp, u64, u64, u64, vp]
        for fn in ("kvev_synth_k", "kvev_synth_q", "kvev_synth_gauss", "kvev_synth_bits"):
            getattr(lib, fn).restype = C.c_int
        _synth = lib
    return _synth


def _stream_ptr(stream):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def device_layer(wl: Workload, layer: int, stream=None, need_q: bool = True):
    """(K, V, Q) CUDA tensors of one layer, bf16; Q is None when need_q is False."""
    import torch
    lib = synth_lib()
    sp = _stream_ptr(stream)
    K = torch.empty((wl.B, wl.H_kv, wl.S_cap, wl.d), dtype=torch.bfloat16, device="cuda")
    V = torch.empty_like(K)
    u_dev, lo, hi, gamma = None, 0, 0, 0.0
    if wl.plant is not None:
        u = np.stack([_unit_u(wl, layer, h) for h in range(wl.H_kv)]).astype(np.float32)
        u_dev = torch.from_numpy(u).cuda()
        lo = int(wl.plant["start"][layer])
        hi = lo + int(wl.plant["size"][layer])
        gamma = float(wl.plant["gamma"][layer])
    rc = lib.kvev_synth_k(K.data_ptr(), wl.B, wl.H_kv, wl.S_cap, wl.d,
                          stream_key(wl.seed, T_K, layer), wl.sink_tokens, float(wl.sink_scale),
                          lo, hi, gamma, None if u_dev is None else u_dev.data_ptr(), sp)
    assert rc == 0, rc
    rc = lib.kvev_synth_bits(V.data_ptr(), V.numel(), stream_key(wl.seed, T_V, layer), 0, sp)
    assert rc == 0, rc
    Q = None
    if need_q:
        Q = torch.empty((wl.B, wl.H_q, wl.W, wl.d), dtype=torch.bfloat16, device="cuda")
        rc = lib.kvev_synth_q(Q.data_ptr(), wl.B, wl.H_q, wl.W, wl.d, wl.G,
                              stream_key(wl.seed, T_Q, layer),
                              float(wl.plant["alpha"]) if wl.plant is not None else 0.0,
                              None if u_dev is None else u_dev.data_ptr(), sp)
        assert rc == 0, rc
    if u_dev is not None:
        torch.cuda.current_stream().synchronize()
    return K, V, Q


def device_decode_tokens(wl: Workload, step: int, layer: int, stream=None):
    """New-token k, v [B][H_kv][d] and q [B][H_q][d] of one decode step (CUDA, bf16)."""
    import torch
    lib = synth_lib()
    sp = _stream_ptr(stream)
    d = wl.d
    k = torch.empty((wl.B, wl.H_kv, d), dtype=torch.bfloat16, device="cuda")
    v = torch.empty_like(k)
    q = torch.empty((wl.B, wl.H_q, d), dtype=torch.bfloat16, device="cuda")
    base_kv = step * wl.B * wl.H_kv * d
    base_q = step * wl.B * wl.H_q * d
    assert lib.kvev_synth_gauss(k.data_ptr(), k.numel(), stream_key(wl.seed, T_KNEW, layer),
                                base_kv, sp) == 0
    assert lib.kvev_synth_bits(v.data_ptr(), v.numel(), stream_key(wl.seed, T_VNEW, layer),
                               base_kv, sp) == 0
    assert lib.kvev_synth_gauss(q.data_ptr(), q.numel(), stream_key(wl.seed, T_QNEW, layer),
                                base_q, sp) == 0
    return k, v, q
