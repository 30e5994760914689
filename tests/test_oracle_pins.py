"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a hand
computation, a closed form, an invariant, a library routine for a special
case, or brute force on a tiny input.  No GPU and no product code is used.
"""
import math
import os

import numpy as np
import pytest

from paper_2606_15157_gb300 import inputs as gen

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def bf16(x):
    """bf16 bit patterns of values that are exactly representable."""
    a = np.atleast_1d(np.asarray(x, dtype=np.float32))
    bits = gen.f32_to_bf16_bits(a)
    assert np.array_equal(gen.bf16_bits_to_f32(bits), a), "test value not exact in bf16"
    return bits if np.ndim(x) else bits[0]


# --------------------------------------------------------------------------
# Allocation (Sec. 3.3, Eq. 3)
# --------------------------------------------------------------------------

def test_alloc_hand_case_proportional(orc):
    # w = [.1,.2,.3,.4], B = 100 -> exactly [10,20,30,40], nothing clamped.
    b = orc.alloc_from_scores([1, 2, 3, 4], 100, 10)
    assert b.tolist() == [10, 20, 30, 40]


def test_alloc_hand_case_clamp_and_largest_remainder(orc):
    # b_min = 15: layer 0 (10) is fixed at 15; the other 85 are re-split in
    # proportion .2:.3:.4 -> 18.89, 28.33, 37.78; floors 15+18+28+37 = 98, the
    # 2 leftover units go to the largest remainders (.89 layer 1, .78 layer 3).
    b = orc.alloc_from_scores([1, 2, 3, 4], 100, 15)
    assert b.tolist() == [15, 19, 28, 38]


def test_alloc_hand_case_iterated_clamping(orc):
    # b~ = [1, 5, 10, 84]: the first clamping pass fixes layers 0,1; the re-split gives layer 2
    # 80*10/94 = 8.5 < 10 so the second pass fixes it too; layer 3 takes the rest.
    b = orc.alloc_from_scores([1, 5, 10, 84], 100, 10)
    assert b.tolist() == [10, 10, 10, 70]


def test_alloc_uniform_is_identity(orc):
    for L, bbar in [(32, 512), (7, 100), (32, 128)]:
        b = orc.alloc_from_scores(np.full(L, 3.7), L * bbar, 48)
        assert b.tolist() == [bbar] * L


def test_alloc_invariants_random(orc):
    rng = np.random.default_rng(0)
    for trial in range(200):
        L = int(rng.integers(1, 48))
        b_min = int(rng.integers(0, 64))
        B = L * b_min + int(rng.integers(0, 40000))
        s = rng.gamma(0.5, size=L) * rng.choice([1e-3, 1.0, 1e3])
        b = orc.alloc_from_scores(s, B, b_min)
        assert b.sum() == B
        assert (b >= b_min).all()
        # Layers above b_min share the rest in proportion to their weights:
        # each lies within one unit of its exact proportional share.
        free = b > b_min
        if free.sum() >= 1:
            rest = B - b_min * (~free).sum()
            share = rest * s[free] / s[free].sum()
            assert np.all(np.abs(b[free] - share) < 1.0 + 1e-9)


def test_alloc_q95_cap_matches_library_percentile(orc):
    # Type-7 quantile is numpy's default 'linear' percentile.
    rng = np.random.default_rng(1)
    for L in [2, 5, 20, 32, 33]:
        s = rng.standard_normal(L) * 3
        assert abs(orc.quantile95(s) - np.percentile(s, 95)) < 1e-12
    # Capping: with one outlier, the capped allocation equals the identity
    # allocation of the explicitly capped scores.
    s = np.concatenate([np.arange(1.0, 32.0), [1000.0]])
    cap = np.percentile(s, 95)
    assert cap < 1000
    a = orc.alloc_from_scores(s, 32 * 512, 48, orc.T_CAP_Q95)
    b = orc.alloc_from_scores(np.minimum(s, cap), 32 * 512, 48, orc.T_IDENTITY)
    assert a.tolist() == b.tolist()


def test_alloc_nonpositive_shift(orc):
    # If min T(s) <= 0 all values are shifted by -min + 1e-6 before Eq. 3.
    s = np.array([-1.0, 0.0, 1.0, 2.5])
    shifted = s + (-s.min() + 1e-6)
    a = orc.alloc_from_scores(s, 4000, 0)
    b = orc.alloc_from_scores(shifted, 4000, 0)
    assert a.tolist() == b.tolist()
    assert a[0] == 0 and abs(a[2] - 4000 * 2 / 6.5) <= 1


def test_alloc_infeasible_rejected(orc):
    with pytest.raises(ValueError):
        orc.alloc_from_scores([1, 1, 1], 100, 40)


def test_alloc_rescale_hand_cases(orc):
    # [10,20,30,40] scaled to 50 is exact; to 51 gives 5.1,10.2,15.3,20.4 whose
    # single leftover unit goes to the largest remainder (layer 3).
    assert orc.alloc_rescale([10, 20, 30, 40], 50).tolist() == [5, 10, 15, 20]
    assert orc.alloc_rescale([10, 20, 30, 40], 51).tolist() == [5, 10, 15, 21]
    rng = np.random.default_rng(2)
    for _ in range(100):
        b_in = rng.integers(1, 3000, size=32).astype(np.int32)
        T = int(rng.integers(32, 100000))
        b = orc.alloc_rescale(b_in, T)
        assert b.sum() == T
        exact = b_in * T / b_in.sum()
        assert np.all(np.abs(b - exact) < 1.0)


# --------------------------------------------------------------------------
# Window scores (SnapKV / H2O prefill rule)
# --------------------------------------------------------------------------

def rand_bf16(rng, shape, scale=1.0):
    return gen.f32_to_bf16_bits((rng.standard_normal(shape) * scale).astype(np.float32))


@pytest.mark.parametrize("n,W,G,d", [(200, 8, 2, 64), (37, 16, 4, 64), (5, 8, 1, 64), (64, 64, 4, 128)])
def test_scores_total_mass_equals_window_rows(orc, n, W, G, d):
    # Every existing window row's softmax sums to 1 over its visible keys, so
    # sum_k raw[k] = (1/G) * G * (number of rows with position >= 0).
    rng = np.random.default_rng(n + W)
    K = rand_bf16(rng, (n, d))
    Q = rand_bf16(rng, (G, W, d))
    raw = orc.window_scores(K, Q, n, W)
    rows = min(W, n)
    assert abs(raw.sum() - rows) < 1e-11 * rows
    assert (raw >= 0).all()


@pytest.mark.parametrize("n", [1, 37, 300])
def test_full_prompt_scores_closed_form_and_mass(orc, n):
    # H2O's full-prompt accumulation is the window score with every prompt
    # position as a query row (W = n).  Equal logits: query t puts 1/(t+1) on
    # keys 0..t, so raw[k] = sum_{t=k}^{n-1} 1/(t+1) = H_n - H_k (harmonic
    # numbers); and every row's distribution sums to 1, so sum_k raw[k] = n.
    rng = np.random.default_rng(9)
    d, G = 64, 3
    K = rand_bf16(rng, (n, d))
    raw = orc.window_scores(K, np.zeros((G, n, d), np.uint16), n, n)
    tail = np.cumsum((1.0 / np.arange(1, n + 1))[::-1])[::-1]  # H_n - H_k without cancellation
    assert np.allclose(raw, tail, rtol=1e-13, atol=0)
    Q = rand_bf16(rng, (G, n, d))
    raw = orc.window_scores(K, Q, n, n)
    assert abs(raw.sum() - n) <= 1e-9 * n


def test_full_prompt_scores_are_sums_of_row_blocks(orc):
    # The accumulation over all rows splits into blocks of W consecutive
    # positions, block j scored as the window of the prompt truncated after it
    # (the row-block decomposition the GPU path uses).
    rng = np.random.default_rng(10)
    n, W, d, G = 96, 16, 64, 2
    K = rand_bf16(rng, (n, d))
    Q = rand_bf16(rng, (G, n, d))
    full = orc.window_scores(K, Q, n, n)
    acc = np.zeros(n)
    for j in range(n // W):
        m = (j + 1) * W
        acc[:m] += orc.window_scores(K[:m], np.ascontiguousarray(Q[:, j * W:m]), m, W)
    assert np.allclose(acc, full, rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("n,W", [(50, 8), (6, 8), (9, 9)])
def test_scores_uniform_logits_closed_form(orc, n, W):
    # Q = 0 gives equal logits: row i (position t_i = n-W+i) puts 1/(t_i+1) on
    # each key 0..t_i, so raw[k] = sum over rows with t_i >= k of 1/(t_i+1).
    rng = np.random.default_rng(3)
    d, G = 64, 2
    K = rand_bf16(rng, (n, d))
    Q = np.zeros((G, W, d), np.uint16)
    raw = orc.window_scores(K, Q, n, W)
    expect = np.zeros(n)
    for i in range(W):
        t = n - W + i
        if t >= 0:
            expect[: t + 1] += 1.0 / (t + 1)
    assert np.allclose(raw, expect, rtol=1e-13, atol=0)


def test_scores_one_dominant_key_closed_form(orc):
    # Every query is 8*e_0 and key j is 8*e_0, all other keys 0: with d = 64
    # the logit of key j is 8*8/sqrt(64) = 8 and every other logit is 0, so a
    # row at position t puts e^8/(e^8+t) on j and 1/(e^8+t) on each other key.
    n, W, G, d, j = 120, 8, 4, 64, 17
    K = np.zeros((n, d), np.uint16)
    K[j, 0] = bf16(8.0)
    Q = np.zeros((G, W, d), np.uint16)
    Q[:, :, 0] = bf16(8.0)
    raw = orc.window_scores(K, Q, n, W)
    e8 = math.exp(8.0)
    rows_t = [n - W + i for i in range(W)]
    assert abs(raw[j] - sum(e8 / (e8 + t) for t in rows_t)) < 1e-12
    k = 50  # another prefix key, seen by every row
    assert abs(raw[k] - sum(1.0 / (e8 + t) for t in rows_t)) < 1e-14
    # a window key is seen only by rows at or after it
    kw = n - 3
    assert abs(raw[kw] - sum(1.0 / (e8 + t) for t in rows_t if t >= kw)) < 1e-14


def test_scores_head_permutation_and_key_permutation(orc):
    rng = np.random.default_rng(4)
    n, W, G, d = 150, 16, 4, 64
    K = rand_bf16(rng, (n, d))
    Q = rand_bf16(rng, (G, W, d))
    raw = orc.window_scores(K, Q, n, W)
    # The group mean does not depend on the order of the G heads.
    raw2 = orc.window_scores(K, Q[::-1].copy(), n, W)
    assert np.allclose(raw, raw2, rtol=1e-12, atol=1e-15)
    # Prefix keys (before the window) are seen by every row: permuting them
    # permutes their scores and leaves the window keys' scores unchanged.
    E = n - W
    perm = rng.permutation(E)
    K2 = K.copy()
    K2[:E] = K[perm]
    raw3 = orc.window_scores(K2, Q, n, W)
    assert np.allclose(raw3[:E], raw[perm], rtol=1e-12, atol=1e-15)
    assert np.allclose(raw3[E:], raw[E:], rtol=1e-12, atol=1e-15)


def test_scores_last_key_seen_only_by_last_row(orc):
    # The causal mask inside the window: key n-1 appears only in row W-1.
    rng = np.random.default_rng(5)
    n, W, G, d = 40, 8, 2, 64
    K = rand_bf16(rng, (n, d))
    Q = rand_bf16(rng, (G, W, d))
    raw = orc.window_scores(K, Q, n, W)
    Kf = gen.bf16_bits_to_f32(K).astype(np.float64)
    Qf = gen.bf16_bits_to_f32(Q).astype(np.float64)
    p_last = 0.0
    for g in range(G):
        lg = Kf @ Qf[g, W - 1] / math.sqrt(d)
        e = np.exp(lg - lg.max())
        p_last += e[-1] / e.sum()
    assert abs(raw[n - 1] - p_last / G) < 1e-13


def test_scores_matrix_form_tiny_config(orc):
    # A second restatement of the window scores in matrix form (numpy, float64):
    # logits = Q K^T / sqrt(d) for all G*W window rows at once, the causal mask
    # as a boolean matrix, a row softmax over the visible keys, and the column
    # sums divided by G.  The oracle's per-row loops must agree with it to
    # 1e-12 on every (layer, KV head) of the tiny config, window keys included.
    wl = gen.config_tiny(seed=0)
    n, W, G, d = int(wl.lens[0]), wl.W, wl.G, wl.d
    pos = np.arange(n, dtype=np.int64)
    t = n - W + np.arange(W)                       # absolute position of window row i
    visible = pos[None, :] <= t[:, None]           # [W][n]
    for l in range(wl.L):
        for h in range(wl.H_kv):
            K = gen.k_rows(wl, l, 0, h, pos)
            Q = gen.q_group(wl, l, 0, h)
            Kf = gen.bf16_bits_to_f32(K).astype(np.float64)
            Qf = gen.bf16_bits_to_f32(Q.reshape(G * W, d)).astype(np.float64)
            S = (Qf @ Kf.T) / math.sqrt(d)                       # [G*W][n]
            S = np.where(np.tile(visible, (G, 1)), S, -np.inf)
            P = np.exp(S - S.max(axis=1, keepdims=True))
            P /= P.sum(axis=1, keepdims=True)
            ref = P.sum(axis=0) / G
            raw = orc.window_scores(K, Q, n, W)
            assert np.allclose(raw, ref, rtol=1e-12, atol=1e-16), (l, h)
            assert abs(raw.sum() - W) < 1e-9


# --------------------------------------------------------------------------
# Pooling and selection
# --------------------------------------------------------------------------

def test_pool_hand_cases(orc):
    x = np.array([0, 0, 0, 1, 0, 0, 0], float)
    assert orc.pool1d(x, 7, 3, orc.POOL_MAX).tolist() == [0, 0, 1, 1, 1, 0, 0]
    assert np.allclose(orc.pool1d(x, 7, 3, orc.POOL_AVG), [0, 0, 1 / 3, 1 / 3, 1 / 3, 0, 0])
    # edges: zero padding counts in the average (divide by p always), max ignores it
    y = np.array([3.0, 1.0, 2.0, 5.0])
    assert np.allclose(orc.pool1d(y, 4, 5, orc.POOL_AVG), [6 / 5, 11 / 5, 11 / 5, 8 / 5])
    assert orc.pool1d(y, 4, 5, orc.POOL_MAX).tolist() == [3, 5, 5, 5]
    # pooling is restricted to the first E entries
    assert orc.pool1d(y, 2, 3, orc.POOL_MAX).tolist() == [3, 3]
    assert np.allclose(orc.pool1d(y, 3, 1, orc.POOL_AVG), y[:3])


def test_topk_brute_force_with_ties(orc):
    rng = np.random.default_rng(6)
    for trial in range(300):
        E = int(rng.integers(1, 200))
        k = int(rng.integers(0, E + 1))
        key = rng.integers(0, 6, size=E).astype(float)  # many ties
        got = orc.topk(key, k)
        order = sorted(range(E), key=lambda p: (-key[p], p))
        assert got.tolist() == sorted(order[:k])


# --------------------------------------------------------------------------
# Retention rules (one unit)
# --------------------------------------------------------------------------

def unit(method, n, b, K=None, Q=None, W=8, **kw):
    d = 64
    if K is None:
        K = np.zeros((max(n, 1), d), np.uint16)
    spec = dict(method=method, n=n, b=b, W=W, K=K, Q=Q, pool_kernel=kw.pop("pool_kernel", 5),
                pool_type=kw.pop("pool_type", 0))
    spec.update(kw)
    return spec


def test_streaming_exact_set(orc):
    res = orc.evict_units([unit(orc.STREAMING, 100, 20, sink=4),
                           unit(orc.STREAMING, 100, 20, sink=4, recent=10),
                           unit(orc.STREAMING, 15, 20, sink=4)], d=64, G=1)
    assert res[0].idx.tolist() == [0, 1, 2, 3] + list(range(84, 100))
    assert res[0].count == 20
    assert res[1].idx.tolist() == [0, 1, 2, 3] + list(range(90, 100)) + [-1] * 6
    assert res[1].count == 14
    assert res[2].idx.tolist() == list(range(15)) + [-1] * 5
    assert res[2].count == 15


@pytest.mark.parametrize("method", [1, 2, 3])
def test_identity_when_budget_covers_sequence(orc, method):
    rng = np.random.default_rng(7)
    n, W, G, d = 30, 8, 2, 64
    K = rand_bf16(rng, (n, d))
    Q = rand_bf16(rng, (G, W, d))
    for b in [n, n + 5]:
        r = orc.evict_units([dict(method=method, n=n, b=b, W=W, K=K, Q=Q, pool_kernel=5,
                                  pool_type=1, sink=4)], d=d, G=G)[0]
        assert r.idx.tolist() == list(range(n)) + [-1] * (b - n)
        assert r.count == n


def test_snapkv_and_h2o_selection_brute_force(orc):
    rng = np.random.default_rng(8)
    for trial in range(20):
        n = int(rng.integers(40, 200))
        W, G, d = 8, 2, 64
        b = int(rng.integers(W + 1, n))
        K = rand_bf16(rng, (n, d), 2.0)
        Q = rand_bf16(rng, (G, W, d), 2.0)
        p = int(rng.choice([1, 3, 5, 7]))
        ptype = int(rng.integers(0, 2))
        r_s, r_h = orc.evict_units(
            [dict(method=orc.SNAPKV, n=n, b=b, W=W, K=K, Q=Q, pool_kernel=p, pool_type=ptype),
             dict(method=orc.H2O, n=n, b=b, W=W, K=K, Q=Q)], d=d, G=G)
        raw = orc.window_scores(K, Q, n, W)
        # SnapKV: last W kept, plus the b-W best pooled prefix scores.
        E = n - W
        pooled = orc.pool1d(raw, E, p, ptype)
        best = sorted(sorted(range(E), key=lambda q: (-pooled[q], q))[: b - W])
        assert r_s.idx.tolist() == best + list(range(E, n))
        assert r_s.count == b
        # H2O: last floor(b/2) kept, plus the best of the rest by raw score.
        rr = b // 2
        E2 = n - rr
        best2 = sorted(sorted(range(E2), key=lambda q: (-raw[q], q))[: b - rr])
        assert r_h.idx.tolist() == best2 + list(range(E2, n))
        assert r_h.count == b
        assert np.allclose(r_h.acc, raw[r_h.idx], rtol=0, atol=0)


def test_rule_parameter_checks(orc):
    with pytest.raises(ValueError):
        orc.evict_units([unit(orc.SNAPKV, 100, 8, W=8)], d=64, G=1)      # b <= W
    with pytest.raises(ValueError):
        orc.evict_units([unit(orc.SNAPKV, 100, 20, pool_kernel=4)], d=64, G=1)  # even pool
    with pytest.raises(ValueError):
        orc.evict_units([unit(orc.STREAMING, 100, 4, sink=4)], d=64, G=1)  # b <= sink


# --------------------------------------------------------------------------
# Decode phase
# --------------------------------------------------------------------------

def test_h2o_decode_hand_case(orc):
    # b = 4, recent r = 2; identical keys make every softmax uniform over the
    # current slots (p = 1/5 after the append).  Step 1: acc = [.7,.3,.5,.4,.2]
    # for positions [0,1,2,3,4]; candidates are positions < 5-2 = 3; the least
    # accumulated is position 1.  Step 2: acc = 0:.9, 2:.7, 3:.6, 4:.4, 5:.2;
    # candidates < 4 -> position 3 (0.6) is evicted.
    d, G = 64, 2
    row = np.zeros(d, np.uint16)
    row[0] = bf16(1.0)
    K = np.tile(row, (4, 1))
    st = orc.DecodeState(orc.H2O, b=4, cap=8, d=d, n=4, pos=[0, 1, 2, 3], K=K, V=K,
                         acc=[0.5, 0.1, 0.3, 0.2], h2o_recent=2)
    q = np.zeros((G, d), np.uint16)
    q[:, 0] = bf16(3.0)
    orc.decode_step([st], [row], [row], [q], d, G)
    assert st.evicted == 1 and st.count == 4
    assert sorted(st.pos[: st.count].tolist()) == [0, 2, 3, 4]
    orc.decode_step([st], [row], [row], [q], d, G)
    assert st.evicted == 3
    got = dict(zip(st.pos[: st.count].tolist(), st.acc[: st.count].tolist()))
    assert sorted(got) == [0, 2, 4, 5]
    assert np.allclose([got[0], got[2], got[4], got[5]], [0.9, 0.7, 0.4, 0.2], atol=1e-12)


def test_h2o_decode_tie_evicts_higher_position(orc):
    d, G = 64, 1
    row = np.zeros(d, np.uint16)
    K = np.tile(row, (3, 1))
    st = orc.DecodeState(orc.H2O, b=3, cap=6, d=d, n=3, pos=[0, 1, 2], K=K, V=K,
                         acc=[0.0, 0.0, 0.0], h2o_recent=0)
    orc.decode_step([st], [row], [row], [np.zeros((G, d), np.uint16)], d, G)
    # all four accumulate 1/4; no recent protection; the tie goes to position 3
    assert st.evicted == 3


def test_tova_decode_hand_case(orc):
    # TOVA keeps only the current step's attention (no accumulation) and may
    # evict the new token itself (no recent window).  q = 8 e0 and k_j = x_j e0
    # with d = 64 make the logits exactly x_j (8 x_j / sqrt(64)).  Step 1: the
    # slots hold positions 0,1,2 with x = [1, 0, 2] and the new token (position
    # 3) has x = 0.5, so p = softmax([1, 0, 2, .5]); the stale acc [9, 9, 9]
    # must be replaced, and position 1 (x = 0) goes.  Step 2: the new token
    # (position 4, x = -3) is the least attended and is the one evicted.
    d, G = 64, 1

    def krow(x):
        r = np.zeros(d, np.uint16)
        r[0] = bf16(x)
        return r

    K = np.stack([krow(1.0), krow(0.0), krow(2.0)])
    st = orc.DecodeState(orc.TOVA, b=3, cap=6, d=d, n=3, pos=[0, 1, 2], K=K, V=K, acc=[9.0, 9.0, 9.0])
    q = np.zeros((G, d), np.uint16)
    q[0, 0] = bf16(8.0)
    orc.decode_step([st], [krow(0.5)], [krow(0.5)], [q], d, G)
    x = np.array([1.0, 0.0, 2.0, 0.5])
    p = np.exp(x - x.max()) / np.exp(x - x.max()).sum()
    assert st.evicted == 1 and st.count == 3
    got = dict(zip(st.pos[: st.count].tolist(), st.acc[: st.count].tolist()))
    assert sorted(got) == [0, 2, 3]
    assert np.allclose([got[0], got[2], got[3]], p[[0, 2, 3]], rtol=0, atol=1e-12)
    orc.decode_step([st], [krow(-3.0)], [krow(-3.0)], [q], d, G)
    x2 = np.array([1.0, 2.0, 0.5, -3.0])
    p2 = np.exp(x2 - x2.max()) / np.exp(x2 - x2.max()).sum()
    assert st.evicted == 4 and st.count == 3
    got = dict(zip(st.pos[: st.count].tolist(), st.acc[: st.count].tolist()))
    assert sorted(got) == [0, 2, 3]
    assert np.allclose([got[0], got[2], got[3]], p2[:3], rtol=0, atol=1e-12)


def test_streaming_decode_rolls_oldest_non_sink(orc):
    d, G = 64, 1
    pos = [0, 1, 6, 7, 8, 9]
    rows = np.zeros((6, d), np.uint16)
    st = orc.DecodeState(orc.STREAMING, b=6, cap=8, d=d, n=10, pos=pos, K=rows, V=rows, sink=2)
    z = np.zeros(d, np.uint16)
    for step, expect in enumerate([6, 7, 8]):
        orc.decode_step([st], [z], [z], [np.zeros((G, d), np.uint16)], d, G)
        assert st.evicted == expect
        assert st.count == 6
        assert {0, 1} <= set(st.pos[: st.count].tolist())


def test_decode_invariants_random(orc):
    rng = np.random.default_rng(9)
    d, G = 64, 4
    for method in (orc.H2O, orc.TOVA, orc.STREAMING, orc.FULL):
        b, n0 = 32, 32
        K = rand_bf16(rng, (n0, d))
        st = orc.DecodeState(method, b=b, cap=b + 40, d=d, n=n0, pos=list(range(n0)), K=K, V=K,
                             acc=rng.random(n0), sink=4, h2o_recent=8)
        for step in range(30):
            k = rand_bf16(rng, (d,))
            q = rand_bf16(rng, (G, d))
            orc.decode_step([st], [k], [k], [q], d, G)
            pos = set(st.pos[: st.count].tolist())
            new = n0 + step
            if method != orc.TOVA:  # TOVA has no recent window: the new token may go
                assert new in pos
            if method == orc.FULL:
                assert st.count == n0 + step + 1
                continue
            assert st.count == b
            if method == orc.H2O:
                assert set(range(new + 1 - 8, new + 1)) <= pos       # recent window kept
            if method == orc.STREAMING:
                assert set(range(4)) <= pos                          # sinks kept
                assert pos == set(range(4)) | set(range(new + 1 - (b - 4), new + 1))


# --------------------------------------------------------------------------
# Paper-printed worked example
# --------------------------------------------------------------------------

def read_golden(name):
    vals = {}
    with open(os.path.join(ROOT, "tests", "golden", name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                vals[k] = float(v)
    return vals


def test_app_e_retained_kv_bytes():
    g = read_golden("app_e_retained_kv.txt")
    positions = g["layers"] * g["budget_per_layer"] * g["batch"]
    assert positions == g["layer_token_positions"]
    nbytes = positions * g["kv_heads"] * g["head_dim"] * g["bytes_per_element"] * 2  # K and V
    assert round(nbytes / 2 ** 20, 2) == g["retained_kv_mib"]
