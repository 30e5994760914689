"""ctypes front end of the CPU oracle (``oracle/kvev_oracle.c``).

TEST INFRASTRUCTURE ONLY: the plain double-precision reference that the GPU
library is checked against.  Only the test suite, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU-baseline leg may import it; the product library never
does, and this module never touches the product library.

Building the oracle is part of ``__graft_entry__.build()``: the shared object
is compiled here with gcc (plain C99 + OpenMP, no fused multiply-add
contraction so both hosts round the same way).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "kvev_oracle.c")
_LIBDIR = os.path.join(_HERE, "lib")
_LIB = os.path.join(_LIBDIR, "libkvev_oracle.so")

# Operator numbering of the oracle (its own; the GPU library has its own enum).
FULL, SNAPKV, H2O, STREAMING, TOVA = 0, 1, 2, 3, 4
POOL_MAX, POOL_AVG = 0, 1
T_IDENTITY, T_CAP_Q95 = 0, 1

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle shared object (idempotent unless ``force``)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-std=c99", "-O2", "-ffp-contract=off", "-fopenmp", "-fPIC", "-shared",
           _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


class OracleUnit(C.Structure):
    _fields_ = [
        ("method", C.c_int), ("n", C.c_int), ("b", C.c_int), ("W", C.c_int),
        ("pool_kernel", C.c_int), ("pool_type", C.c_int), ("sink", C.c_int),
        ("recent", C.c_int), ("h2o_recent", C.c_int),
        ("K", C.c_void_p), ("Q", C.c_void_p),
        ("raw", C.c_void_p), ("pooled", C.c_void_p),
        ("idx", C.c_void_p), ("count", C.c_void_p), ("acc", C.c_void_p),
    ]


class OracleDecUnit(C.Structure):
    _fields_ = [
        ("method", C.c_int), ("b", C.c_int), ("sink", C.c_int), ("recent", C.c_int),
        ("h2o_recent", C.c_int), ("n", C.c_int), ("cap", C.c_int), ("count", C.c_int),
        ("pos", C.c_void_p), ("acc", C.c_void_p), ("K", C.c_void_p), ("V", C.c_void_p),
        ("k_new", C.c_void_p), ("v_new", C.c_void_p), ("q_new", C.c_void_p),
        ("evicted", C.c_int),
    ]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            L = C.CDLL(path)
            L.oracle_alloc_from_scores.argtypes = [C.c_void_p, C.c_void_p, C.c_int, C.c_int64,
                                                   C.c_int, C.c_int]
            L.oracle_alloc_from_scores.restype = C.c_int
            L.oracle_alloc_rescale.argtypes = [C.c_void_p, C.c_void_p, C.c_int, C.c_int64]
            L.oracle_alloc_rescale.restype = C.c_int
            L.oracle_quantile95.argtypes = [C.c_void_p, C.c_int]
            L.oracle_quantile95.restype = C.c_double
            L.oracle_window_scores.argtypes = [C.c_void_p, C.c_void_p, C.c_int, C.c_int, C.c_int,
                                               C.c_int, C.c_void_p]
            L.oracle_window_scores.restype = None
            L.oracle_pool1d.argtypes = [C.c_void_p, C.c_int, C.c_int, C.c_int, C.c_void_p]
            L.oracle_pool1d.restype = None
            L.oracle_topk.argtypes = [C.c_void_p, C.c_int, C.c_int, C.c_void_p]
            L.oracle_topk.restype = None
            L.oracle_evict_unit.argtypes = [C.POINTER(OracleUnit), C.c_int, C.c_int]
            L.oracle_evict_unit.restype = C.c_int
            L.oracle_evict_units.argtypes = [C.POINTER(OracleUnit), C.c_int, C.c_int, C.c_int,
                                             C.c_int]
            L.oracle_evict_units.restype = C.c_int
            L.oracle_decode_units.argtypes = [C.POINTER(OracleDecUnit), C.c_int, C.c_int, C.c_int,
                                              C.c_int]
            L.oracle_decode_units.restype = C.c_int
            L.oracle_max_threads.argtypes = []
            L.oracle_max_threads.restype = C.c_int
            _lib = L
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data


def max_threads() -> int:
    return int(lib().oracle_max_threads())


# --------------------------------------------------------------------------
# Allocation (Sec. 3.3, Eq. 3)
# --------------------------------------------------------------------------

def alloc_from_scores(s, B_total: int, b_min: int, transform: int = T_IDENTITY) -> np.ndarray:
    s = np.ascontiguousarray(s, dtype=np.float64)
    out = np.zeros(len(s), dtype=np.int32)
    rc = lib().oracle_alloc_from_scores(_ptr(out), _ptr(s), len(s), int(B_total), int(b_min),
                                        int(transform))
    if rc != 0:
        raise ValueError("infeasible allocation request")
    return out


def alloc_rescale(b_in, B_target: int) -> np.ndarray:
    b_in = np.ascontiguousarray(b_in, dtype=np.int32)
    out = np.zeros(len(b_in), dtype=np.int32)
    rc = lib().oracle_alloc_rescale(_ptr(out), _ptr(b_in), len(b_in), int(B_target))
    if rc != 0:
        raise ValueError("invalid rescale request")
    return out


def quantile95(s) -> float:
    s = np.ascontiguousarray(s, dtype=np.float64)
    return float(lib().oracle_quantile95(_ptr(s), len(s)))


# --------------------------------------------------------------------------
# Scoring, pooling, selection
# --------------------------------------------------------------------------

def window_scores(K: np.ndarray, Q: np.ndarray, n: int, W: int) -> np.ndarray:
    """K: uint16 bf16 bits [>=n][d]; Q: uint16 [G][W][d].  Returns raw[n]."""
    K = np.ascontiguousarray(K, dtype=np.uint16)
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    G, Wq, d = Q.shape
    assert Wq == W and K.shape[1] == d
    raw = np.zeros(max(n, 1), dtype=np.float64)
    lib().oracle_window_scores(_ptr(K), _ptr(Q), n, d, G, W, _ptr(raw))
    return raw[:n]


def pool1d(raw: np.ndarray, E: int, p: int, pool_type: int) -> np.ndarray:
    raw = np.ascontiguousarray(raw, dtype=np.float64)
    out = np.zeros(max(E, 1), dtype=np.float64)
    lib().oracle_pool1d(_ptr(raw), E, p, pool_type, _ptr(out))
    return out[:E]


def topk(key: np.ndarray, k: int) -> np.ndarray:
    key = np.ascontiguousarray(key, dtype=np.float64)
    out = np.zeros(max(k, 1), dtype=np.int32)
    lib().oracle_topk(_ptr(key), len(key), k, _ptr(out))
    return out[:k]


class UnitResult:
    """Outputs of one prefill-eviction unit."""

    def __init__(self, n: int, b: int):
        self.raw = np.zeros(max(n, 1), dtype=np.float64)
        self.pooled = np.zeros(max(n, 1), dtype=np.float64)
        self.idx = np.full(max(b, 1), -1, dtype=np.int32)
        self.count = np.zeros(1, dtype=np.int32)
        self.acc = np.zeros(max(b, 1), dtype=np.float64)


def evict_units(specs, d: int, G: int, nthreads: int = 0):
    """Run prefill eviction on independent units.

    ``specs``: list of dicts with keys method, n, b, W, pool_kernel, pool_type,
    sink, recent, h2o_recent, K (uint16 [>=n][d]), Q (uint16 [G][W][d] or None).
    Returns a list of UnitResult (idx/acc arrays are length b).
    """
    n_units = len(specs)
    arr = (OracleUnit * max(n_units, 1))()
    keep = []
    results = []
    for i, s in enumerate(specs):
        res = UnitResult(s["n"], s["b"])
        results.append(res)
        K = np.ascontiguousarray(s["K"], dtype=np.uint16)
        Q = None if s.get("Q") is None else np.ascontiguousarray(s["Q"], dtype=np.uint16)
        keep.append((K, Q))
        u = arr[i]
        u.method = s["method"]
        u.n = s["n"]
        u.b = s["b"]
        u.W = s.get("W", 0)
        u.pool_kernel = s.get("pool_kernel", 1)
        u.pool_type = s.get("pool_type", POOL_MAX)
        u.sink = s.get("sink", 0)
        u.recent = s.get("recent", -1)
        u.h2o_recent = s.get("h2o_recent", -1)
        u.K = _ptr(K)
        u.Q = _ptr(Q)
        u.raw = _ptr(res.raw)
        u.pooled = _ptr(res.pooled)
        u.idx = _ptr(res.idx)
        u.count = _ptr(res.count)
        u.acc = _ptr(res.acc)
    failed = lib().oracle_evict_units(arr, n_units, d, G, nthreads)
    if failed:
        raise ValueError(f"{failed} oracle units rejected their parameters")
    for r, s in zip(results, specs):
        r.raw = r.raw[: s["n"]]
        r.pooled = r.pooled[: max(s["n"] - s.get("W", 0), 0)]
        r.idx = r.idx[: s["b"]]
        r.acc = r.acc[: s["b"]]
        r.count = int(r.count[0])
    return results


# --------------------------------------------------------------------------
# Decode phase
# --------------------------------------------------------------------------

class DecodeState:
    """Slot set of one unit in the decode phase (positions, scores, rows)."""

    def __init__(self, method: int, b: int, cap: int, d: int, n: int, pos, K, V, acc=None,
                 sink: int = 0, recent: int = -1, h2o_recent: int = -1):
        self.method, self.b, self.cap, self.d, self.n = method, b, cap, d, n
        self.sink, self.recent, self.h2o_recent = sink, recent, h2o_recent
        cnt = len(pos)
        self.pos = np.full(cap, -1, dtype=np.int32)
        self.pos[:cnt] = pos
        self.acc = np.zeros(cap, dtype=np.float64)
        if acc is not None:
            self.acc[:cnt] = acc
        self.K = np.zeros((cap, d), dtype=np.uint16)
        self.K[:cnt] = K
        self.V = np.zeros((cap, d), dtype=np.uint16)
        self.V[:cnt] = V
        self.count = cnt
        self.evicted = -1

    def as_dict(self):
        c = self.count
        order = np.argsort(self.pos[:c], kind="stable")
        return {"pos": self.pos[:c][order].copy(), "acc": self.acc[:c][order].copy(),
                "K": self.K[:c][order].copy(), "V": self.V[:c][order].copy()}


def decode_step(states, k_new, v_new, q_new, d: int, G: int, nthreads: int = 0):
    """Advance every DecodeState by one token.  k_new/v_new: list of uint16 [d];
    q_new: list of uint16 [G][d]."""
    n_units = len(states)
    arr = (OracleDecUnit * max(n_units, 1))()
    keep = []
    for i, st in enumerate(states):
        kn = np.ascontiguousarray(k_new[i], dtype=np.uint16)
        vn = np.ascontiguousarray(v_new[i], dtype=np.uint16)
        qn = np.ascontiguousarray(q_new[i], dtype=np.uint16)
        keep.append((kn, vn, qn))
        u = arr[i]
        u.method, u.b, u.sink, u.recent = st.method, st.b, st.sink, st.recent
        u.h2o_recent, u.n, u.cap, u.count = st.h2o_recent, st.n, st.cap, st.count
        u.pos, u.acc, u.K, u.V = _ptr(st.pos), _ptr(st.acc), _ptr(st.K), _ptr(st.V)
        u.k_new, u.v_new, u.q_new = _ptr(kn), _ptr(vn), _ptr(qn)
        u.evicted = -1
    failed = lib().oracle_decode_units(arr, n_units, d, G, nthreads)
    if failed:
        raise ValueError(f"{failed} oracle decode units failed")
    for i, st in enumerate(states):
        st.count = arr[i].count
        st.n = arr[i].n
        st.evicted = arr[i].evicted
    return states
