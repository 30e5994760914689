"""Plan constructor (Sec. 3.2-3.4), host only: the oracle pinned to closed
forms and library routines, the library checked against the oracle, the
error paths, and the plan serialisation."""
import math
import struct

import numpy as np
import pytest

from oracle import planner as orc
from paper_2606_15157_gb300 import kvev


@pytest.fixture(scope="module", autouse=True)
def lib():
    kvev.load()


# ---- oracle pins ----------------------------------------------------------

def test_oracle_entropy_closed_forms():
    K = 7
    uniform = [[1.0 / K] * K]
    one_hot = [[0.0, 1.0, 0.0]]
    p = 0.3
    two = [[p, 1 - p, 0.0]]
    assert orc.entropy_score([uniform])[0] == pytest.approx(math.log(K), rel=1e-15)
    assert orc.entropy_score([one_hot])[0] == 0.0
    assert orc.entropy_score([two])[0] == pytest.approx(-p * math.log(p) - (1 - p) * math.log(1 - p), rel=1e-15)
    # the mean is over rows: two rows with entropies log 2 and 0
    assert orc.entropy_score([[[0.5, 0.5], [1.0, 0.0]]])[0] == pytest.approx(math.log(2) / 2, rel=1e-15)


def test_oracle_entropy_matches_scipy():
    stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(0)
    A = rng.dirichlet(np.full(33, 0.3), size=(3, 5))
    A[:, :, 20:] = 0.0  # a causal mask
    A /= A.sum(-1, keepdims=True)
    ref = [float(np.mean([stats.entropy(row) for row in A[l]])) for l in range(3)]
    assert orc.entropy_score(A.tolist()) == pytest.approx(ref, rel=1e-12)


def test_oracle_cosine_closed_forms_and_scipy():
    dist = pytest.importorskip("scipy.spatial.distance")
    a = [1.0, 2.0, -3.0]
    C = orc.cosine_profile([a], [[a], [[-2.0, -4.0, 6.0]], [[2.0, -1.0, 0.0]]])
    assert C[0] == pytest.approx([1.0, -1.0, 0.0], abs=1e-15)
    rng = np.random.default_rng(1)
    hf, hc = rng.normal(size=(4, 9)), rng.normal(size=(3, 4, 9))
    C = orc.cosine_profile(hf.tolist(), hc.tolist())
    for l in range(4):
        for r in range(3):
            assert C[l][r] == pytest.approx(1.0 - dist.cosine(hf[l], hc[r][l]), rel=1e-12)


def test_oracle_toprank_hand_cases():
    ops = [orc.SNAPKV, orc.H2O, orc.STREAMING]
    g = [[0.9, 0.95, 0.1], [0.5, 0.5, 0.4], [0.2, 0.3, 0.3]]
    assert orc.toprank(g, ops, True) == [orc.H2O, orc.SNAPKV, orc.H2O]  # ties keep the first
    assert orc.toprank(g, ops, False) == [orc.STREAMING, orc.STREAMING, orc.SNAPKV]
    cov = [[1, 0, 1], [0, 0, 0], [1, 1, 1]]
    assert orc.toprank(g, ops, True, cov) == [orc.SNAPKV, orc.FULL, orc.H2O]


def test_oracle_ppl_and_install():
    assert orc.ppl_score([[10.0, 12.5], [11.0, 9.5]], 10.0) == [2.5, 1.0]
    assert orc.install([orc.SNAPKV, orc.H2O], orc.SCOPE_PREFILL) == ([orc.SNAPKV, orc.H2O], [0, 0])
    assert orc.install([orc.TOVA, orc.H2O], orc.SCOPE_DECODE) == ([0, 0], [orc.TOVA, orc.H2O])
    assert orc.install([orc.STREAMING, orc.H2O], orc.SCOPE_BOTH) == ([orc.STREAMING, orc.H2O],) * 2
    assert orc.install([orc.SNAPKV], orc.SCOPE_DECODE) is None
    assert orc.install([orc.TOVA], orc.SCOPE_BOTH) is None


# ---- library against the oracle --------------------------------------------

@pytest.mark.parametrize("seed", range(5))
def test_library_matches_oracle_random(seed):
    rng = np.random.default_rng(seed)
    L, R, D, rows, K = 6, 4, 17, 9, 40
    hf = rng.normal(size=(L, D)).astype(np.float32)
    hc = rng.normal(size=(R, L, D)).astype(np.float32)
    np.testing.assert_allclose(kvev.kvev_profile_cosine(hf, hc),
                               orc.cosine_profile(hf.astype(np.float64).tolist(),
                                                  hc.astype(np.float64).tolist()), rtol=1e-12, atol=1e-15)
    ppl = rng.uniform(5, 30, size=(L, R))
    np.testing.assert_allclose(kvev.kvev_score_ppl(ppl, 7.0), orc.ppl_score(ppl.tolist(), 7.0), rtol=0, atol=0)
    A = rng.dirichlet(np.full(K, 0.5), size=(L, rows))
    A[:, :, K // 2:] *= rng.integers(0, 2, size=(L, rows, 1))  # some rows causally masked
    A = (A / A.sum(-1, keepdims=True)).astype(np.float32)
    np.testing.assert_allclose(kvev.kvev_score_entropy(A),
                               orc.entropy_score(A.astype(np.float64).tolist()), rtol=1e-12)
    ops = [kvev.SNAPKV, kvev.H2O, kvev.STREAMING, kvev.TOVA]
    g = rng.integers(0, 4, size=(L, R)).astype(np.float64)  # many ties
    cov = rng.integers(0, 2, size=(L, R)).astype(np.uint8)
    for hib in (True, False):
        for c in (None, cov):
            got = kvev.kvev_route_toprank(g, ops, hib, c)
            ref = orc.toprank(g.tolist(), ops, hib, None if c is None else c.tolist())
            assert got.tolist() == ref


def test_library_install_scopes():
    r = np.array([kvev.H2O, kvev.STREAMING, kvev.FULL], np.int32)
    for scope in (kvev.SCOPE_PREFILL, kvev.SCOPE_DECODE, kvev.SCOPE_BOTH):
        pre, dec = kvev.kvev_route_install(r, scope)
        ref = orc.install(r.tolist(), scope)
        assert (pre.tolist(), dec.tolist()) == (list(ref[0]), list(ref[1]))
    with pytest.raises(kvev.KvevError):
        kvev.kvev_route_install([kvev.SNAPKV], kvev.SCOPE_DECODE)
    with pytest.raises(kvev.KvevError):
        kvev.kvev_route_install([kvev.TOVA], kvev.SCOPE_PREFILL)
    with pytest.raises(kvev.KvevError):
        kvev.kvev_route_install([kvev.H2O], 0)


def test_library_rejects_bad_inputs():
    with pytest.raises(kvev.KvevError):
        kvev.kvev_score_entropy(np.array([[[0.5, 0.6]]], np.float32))  # not a distribution
    with pytest.raises(kvev.KvevError):
        kvev.kvev_score_entropy(np.array([[[1.5, -0.5]]], np.float32))  # negative entry
    with pytest.raises(kvev.KvevError):
        kvev.kvev_profile_cosine(np.zeros((1, 3)), np.ones((1, 1, 3)))  # zero norm
    with pytest.raises(kvev.KvevError):
        kvev.kvev_route_toprank([[np.nan]], [kvev.H2O], True)
    with pytest.raises(kvev.KvevError):
        kvev.kvev_route_toprank([[1.0]], [99], True)
    with pytest.raises(kvev.KvevError):
        kvev.kvev_score_ppl([[np.inf]], 1.0)


# ---- plan serialisation (Sec. 3.4) ------------------------------------------

def _fnv1a(b: bytes) -> int:
    h = 1469598103934665603
    for x in b:
        h = ((h ^ x) * 1099511628211) & 0xFFFFFFFFFFFFFFFF
    return h


def _plan():
    route = [kvev.SNAPKV, kvev.STREAMING, kvev.H2O, kvev.FULL, kvev.H2O]
    dec = [kvev.FULL, kvev.STREAMING, kvev.H2O, kvev.FULL, kvev.TOVA]
    return kvev.Plan(5, 8, 2, 128, route, [100, 64, 80, 0, 50], 16, 5, kvev.POOL_MAX, sink=4,
                     recent=-1, h2o_recent=20, route_decode=dec)


def test_plan_save_load_round_trip():
    p = _plan()
    b = p.save()
    L = 5
    assert len(b) == 8 + 4 * (10 + 3 * L) + 8
    assert b[:8] == b"KVEVPLN1"
    words = struct.unpack(f"<{10 + 3 * L}i", b[8:-8])
    assert words[:10] == (5, 8, 2, 128, 16, 5, kvev.POOL_MAX, 4, -1, 20)
    assert list(words[10:15]) == [1, 3, 2, 0, 2] and list(words[20:25]) == [100, 64, 80, 0, 50]
    assert struct.unpack("<Q", b[-8:])[0] == _fnv1a(b[:-8])
    q = kvev.Plan.load(b)
    assert q.save() == b
    assert q.query(4, 4096) == p.query(4, 4096)
    for l in range(L):
        assert q.layer_offset(4, l) == p.layer_offset(4, l)


def test_plan_load_rejects_corrupt_buffers():
    b = bytearray(_plan().save())
    for bad in (bytes(b[:-1]), b"XXXXXXXX" + bytes(b[8:]), bytes(b[:20])):
        with pytest.raises(kvev.KvevError):
            kvev.Plan.load(bad)
    flipped = bytearray(b)
    flipped[40] ^= 1  # a body byte: the checksum no longer matches
    with pytest.raises(kvev.KvevError):
        kvev.Plan.load(bytes(flipped))
    # a well-formed buffer whose plan fails kvev_plan_create's checks
    words = list(struct.unpack("<25i", bytes(b[8:-8])))
    words[20] = 10  # SnapKV budget below its window
    body = b"KVEVPLN1" + struct.pack("<25i", *words)
    with pytest.raises(kvev.KvevError):
        kvev.Plan.load(body + struct.pack("<Q", _fnv1a(body)))
