"""ctypes binding of ``libkvev.so`` (C ABI in ``include/kvev.h``).

Argument marshalling only: every step of the eviction runs in the library's
kernels.  Functions keep the C names; :class:`Plan` is a small convenience
wrapper that owns a plan handle and sizes the buffers.  If the library has not
been built, loading raises -- there is no fallback implementation.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "lib", "libkvev.so")

OK, EINVAL, ENOMEM, ECUDA, ETIMEOUT, EDEVICE, ENOTSUP = range(7)
FULL, SNAPKV, H2O, STREAMING, TOVA = 0, 1, 2, 3, 4
POOL_MAX, POOL_AVG = 0, 1
T_IDENTITY, T_CAP_Q95 = 0, 1
SCOPE_PREFILL, SCOPE_DECODE, SCOPE_BOTH = 1, 2, 3

STATUS_NAMES = {OK: "OK", EINVAL: "EINVAL", ENOMEM: "ENOMEM", ECUDA: "ECUDA",
                ETIMEOUT: "ETIMEOUT", EDEVICE: "EDEVICE", ENOTSUP: "ENOTSUP"}

EXPORTS = ["kvev_alloc_from_scores", "kvev_alloc_rescale", "kvev_plan_create",
           "kvev_plan_destroy", "kvev_plan_query", "kvev_plan_layer_offset",
           "kvev_evict_prefill", "kvev_status", "kvev_plan_set_wait_limit",
           "kvev_plan_debug_stall_unit", "kvev_plan_scores_offset", "kvev_plan_enable_timing",
           "kvev_plan_last_timings", "kvev_evict_prefill_noalloc", "kvev_decode_query",
           "kvev_decode_layer", "kvev_decode_state_offsets", "kvev_decode_init",
           "kvev_decode_step", "kvev_decode_step_attn", "kvev_evict_prefill_scored", "kvev_evict_prefill_lse",
           "kvev_profile_cosine", "kvev_score_ppl", "kvev_score_entropy",
           "kvev_route_toprank", "kvev_route_install", "kvev_plan_save", "kvev_plan_load",
           "kvev_plan_set_h2o_full_prompt"]
KERNEL_NAMES = ["prologue", "score", "select", "gather"]


class KvevError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {STATUS_NAMES.get(code, code)}")
        self.code = code


_lock = threading.Lock()
_lib = None


def load(path: str = LIB_PATH):
    """Load the library (once).  Raises if it is missing."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build()")
        L = C.CDLL(path)
        vp, i32, i64, sz = C.c_void_p, C.c_int32, C.c_int64, C.c_size_t
        P = C.POINTER
        L.kvev_alloc_from_scores.argtypes = [vp, vp, C.c_int, i64, C.c_int, C.c_int]
        L.kvev_alloc_rescale.argtypes = [vp, vp, C.c_int, i64]
        L.kvev_plan_create.argtypes = [P(vp), C.c_int, C.c_int, C.c_int, C.c_int, vp, vp, vp,
                                       C.c_int, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int]
        L.kvev_plan_destroy.argtypes = [vp]
        L.kvev_plan_destroy.restype = None
        L.kvev_plan_query.argtypes = [vp, C.c_int, C.c_int, P(sz), P(sz), P(sz), P(sz)]
        L.kvev_plan_layer_offset.argtypes = [vp, C.c_int, C.c_int, P(i64)]
        L.kvev_evict_prefill.argtypes = [vp, vp, vp, vp, vp, C.c_int, C.c_int, vp, vp, vp, vp, vp,
                                         vp, sz, vp]
        L.kvev_evict_prefill_scored.argtypes = [vp, vp, vp, vp, vp, vp, C.c_int, C.c_int, vp, vp, vp,
                                                vp, vp, vp, sz, vp]
        L.kvev_evict_prefill_lse.argtypes = [vp, vp, vp, vp, vp, vp, C.c_int, C.c_int, vp, vp, vp,
                                             vp, vp, vp, sz, vp]
        L.kvev_status.argtypes = [vp, P(C.c_int)]
        L.kvev_plan_set_wait_limit.argtypes = [vp, i64]
        L.kvev_plan_debug_stall_unit.argtypes = [vp, C.c_int]
        L.kvev_plan_scores_offset.argtypes = [vp, C.c_int, C.c_int, C.c_int, P(sz)]
        L.kvev_plan_enable_timing.argtypes = [vp, C.c_int]
        L.kvev_evict_prefill_noalloc.argtypes = [vp, vp, vp, vp, vp, C.c_int, C.c_int, vp, vp,
                                                 vp, vp, vp, vp, vp]
        L.kvev_plan_last_timings.argtypes = [vp, vp, C.c_int]
        L.kvev_decode_query.argtypes = [vp, C.c_int, C.c_int, P(i64), P(sz)]
        L.kvev_decode_layer.argtypes = [vp, C.c_int, C.c_int, C.c_int, P(i64), P(C.c_int),
                                        P(C.c_int)]
        L.kvev_decode_state_offsets.argtypes = [vp, C.c_int, C.c_int, P(sz)]
        L.kvev_decode_init.argtypes = [vp, C.c_int, C.c_int, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
        L.kvev_decode_step.argtypes = [vp, C.c_int, C.c_int, vp, vp, vp, vp, vp, vp, vp]
        L.kvev_decode_step_attn.argtypes = [vp, C.c_int, C.c_int, vp, vp, vp, vp, vp, vp, vp]
        L.kvev_profile_cosine.argtypes = [vp, vp, vp, C.c_int, C.c_int, i64]
        L.kvev_score_ppl.argtypes = [vp, vp, C.c_double, C.c_int, C.c_int]
        L.kvev_score_entropy.argtypes = [vp, vp, C.c_int, i64, C.c_int]
        L.kvev_route_toprank.argtypes = [vp, vp, C.c_int, C.c_int, vp, vp, C.c_int]
        L.kvev_route_install.argtypes = [vp, vp, vp, C.c_int, C.c_int]
        L.kvev_plan_save.argtypes = [vp, vp, P(sz)]
        L.kvev_plan_load.argtypes = [P(vp), vp, sz]
        L.kvev_plan_set_h2o_full_prompt.argtypes = [vp, C.c_int]
        for name in EXPORTS:
            if name != "kvev_plan_destroy":
                getattr(L, name).restype = C.c_int
        _lib = L
    return _lib


def _check(rc: int, what: str):
    if rc != OK:
        raise KvevError(rc, what)


# ---------------------------------------------------------------------------
# C-named wrappers
# ---------------------------------------------------------------------------

def kvev_alloc_from_scores(s, B_total: int, b_min: int, transform: int = T_IDENTITY) -> np.ndarray:
    s = np.ascontiguousarray(s, dtype=np.float64)
    out = np.zeros(len(s), np.int32)
    _check(load().kvev_alloc_from_scores(out.ctypes.data, s.ctypes.data, len(s), int(B_total),
                                         int(b_min), int(transform)), "kvev_alloc_from_scores")
    return out


def kvev_alloc_rescale(b_in, B_target: int) -> np.ndarray:
    b_in = np.ascontiguousarray(b_in, dtype=np.int32)
    out = np.zeros(len(b_in), np.int32)
    _check(load().kvev_alloc_rescale(out.ctypes.data, b_in.ctypes.data, len(b_in), int(B_target)),
           "kvev_alloc_rescale")
    return out


alloc_from_scores = kvev_alloc_from_scores
alloc_rescale = kvev_alloc_rescale


def kvev_plan_create(L, H_q, H_kv, d, route_prefill, route_decode, budget, window, pool_kernel,
                     pool_type, sink, recent=-1, h2o_recent=-1) -> int:
    rp = np.ascontiguousarray(route_prefill, np.int32)
    rd = None if route_decode is None else np.ascontiguousarray(route_decode, np.int32)
    b = np.ascontiguousarray(budget, np.int32)
    h = C.c_void_p()
    rc = load().kvev_plan_create(C.byref(h), L, H_q, H_kv, d, rp.ctypes.data,
                                 None if rd is None else rd.ctypes.data, b.ctypes.data, window,
                                 pool_kernel, pool_type, sink, recent, h2o_recent)
    _check(rc, "kvev_plan_create")
    return h.value


def kvev_plan_destroy(handle: int):
    load().kvev_plan_destroy(handle)


def kvev_plan_query(handle: int, B: int, S_cap: int):
    vals = [C.c_size_t() for _ in range(4)]
    _check(load().kvev_plan_query(handle, B, S_cap, *[C.byref(v) for v in vals]),
           "kvev_plan_query")
    return tuple(v.value for v in vals)


def kvev_plan_layer_offset(handle: int, B: int, layer: int) -> int:
    v = C.c_int64()
    _check(load().kvev_plan_layer_offset(handle, B, layer, C.byref(v)), "kvev_plan_layer_offset")
    return v.value


def kvev_evict_prefill(handle, K_ptrs, V_ptrs, Q_ptrs, lens_ptr, B, S_cap, out_K, out_V, out_idx,
                       out_count, h2o_state, workspace, workspace_bytes, stream) -> int:
    """Pointer-level call; returns the status code (does not raise)."""
    Ln = len(K_ptrs)
    arr = C.c_void_p * Ln
    Ka, Va = arr(*K_ptrs), arr(*V_ptrs)
    Qa = arr(*Q_ptrs) if Q_ptrs is not None else None
    return load().kvev_evict_prefill(handle, Ka, Va, Qa, lens_ptr, B, S_cap, out_K, out_V,
                                     out_idx, out_count, h2o_state, workspace, workspace_bytes,
                                     stream)


def kvev_evict_prefill_scored(handle, K_ptrs, V_ptrs, Q_ptrs, score_ptrs, lens_ptr, B, S_cap, out_K, out_V,
                              out_idx, out_count, h2o_state, workspace, workspace_bytes, stream) -> int:
    """Pointer-level call with caller-supplied scores; returns the status code."""
    Ln = len(K_ptrs)
    arr = C.c_void_p * Ln
    Ka, Va = arr(*K_ptrs), arr(*V_ptrs)
    Sa = arr(*score_ptrs) if score_ptrs is not None else None
    Qa = arr(*Q_ptrs) if Q_ptrs is not None else None
    return load().kvev_evict_prefill_scored(handle, Ka, Va, Qa, Sa, lens_ptr, B, S_cap, out_K, out_V,
                                            out_idx, out_count, h2o_state, workspace, workspace_bytes,
                                            stream)


def kvev_evict_prefill_lse(handle, K_ptrs, V_ptrs, Q_ptrs, lse_ptrs, lens_ptr, B, S_cap, out_K, out_V,
                           out_idx, out_count, h2o_state, workspace, workspace_bytes, stream) -> int:
    """Pointer-level call with the caller's window-row log-sum-exp; returns the status code."""
    Ln = len(K_ptrs)
    arr = C.c_void_p * Ln
    Ka, Va = arr(*K_ptrs), arr(*V_ptrs)
    La = arr(*lse_ptrs) if lse_ptrs is not None else None
    Qa = arr(*Q_ptrs) if Q_ptrs is not None else None
    return load().kvev_evict_prefill_lse(handle, Ka, Va, Qa, La, lens_ptr, B, S_cap, out_K, out_V,
                                         out_idx, out_count, h2o_state, workspace, workspace_bytes,
                                         stream)


NOALLOC_SCRATCH_BYTES = 32 << 20


def kvev_evict_prefill_noalloc(handle, K_ptrs, V_ptrs, Q_ptrs, lens_ptr, B, S_cap, out_K, out_V,
                               out_idx, out_count, h2o_state, device_status, stream) -> int:
    """Pointer-level call of the entry point that allocates nothing (its scratch is
    a fixed library-owned device array); returns the status code."""
    arr = C.c_void_p * len(K_ptrs)
    Ka, Va = arr(*K_ptrs), arr(*V_ptrs)
    Qa = arr(*Q_ptrs) if Q_ptrs is not None else None
    return load().kvev_evict_prefill_noalloc(handle, Ka, Va, Qa, lens_ptr, B, S_cap, out_K, out_V,
                                             out_idx, out_count, h2o_state, device_status, stream)


def kvev_decode_query(handle: int, B: int, growth: int):
    rows, state = C.c_int64(), C.c_size_t()
    _check(load().kvev_decode_query(handle, B, growth, C.byref(rows), C.byref(state)),
           "kvev_decode_query")
    return rows.value, state.value


def kvev_decode_layer(handle: int, B: int, growth: int, layer: int):
    """(first arena row, slots per unit, first unit) of a layer."""
    off, cap, u0 = C.c_int64(), C.c_int(), C.c_int()
    _check(load().kvev_decode_layer(handle, B, growth, layer, C.byref(off), C.byref(cap),
                                    C.byref(u0)), "kvev_decode_layer")
    return off.value, cap.value, u0.value


def kvev_decode_state_offsets(handle: int, B: int, growth: int):
    """Byte offsets of lens, count, evicted, pos, acc in the state buffer."""
    offs = (C.c_size_t * 5)()
    _check(load().kvev_decode_state_offsets(handle, B, growth, offs), "kvev_decode_state_offsets")
    return dict(zip(("lens", "count", "evicted", "pos", "acc"), list(offs)))


def kvev_decode_init(handle, B, growth, pre_K, pre_V, pre_idx, pre_count, h2o_state, lens_ptr,
                     dec_K, dec_V, dec_state, stream) -> int:
    return load().kvev_decode_init(handle, B, growth, pre_K, pre_V, pre_idx, pre_count, h2o_state,
                                   lens_ptr, dec_K, dec_V, dec_state, stream)


def kvev_decode_step(handle, B, growth, dec_K, dec_V, dec_state, k_ptrs, v_ptrs, q_ptrs,
                     stream) -> int:
    arr = C.c_void_p * len(k_ptrs)
    return load().kvev_decode_step(handle, B, growth, dec_K, dec_V, dec_state, arr(*k_ptrs),
                                   arr(*v_ptrs), arr(*q_ptrs), stream)


def kvev_decode_step_attn(handle, B, growth, dec_K, dec_V, dec_state, k_ptrs, v_ptrs, attn_ptrs,
                          stream) -> int:
    """Pointer-level call; returns the status code (does not raise)."""
    arr = C.c_void_p * len(k_ptrs)
    return load().kvev_decode_step_attn(handle, B, growth, dec_K, dec_V, dec_state, arr(*k_ptrs),
                                        arr(*v_ptrs), arr(*attn_ptrs), stream)


def kvev_status(handle: int) -> int:
    v = C.c_int()
    _check(load().kvev_status(handle, C.byref(v)), "kvev_status")
    return v.value


def kvev_plan_scores_offset(handle: int, B: int, S_cap: int, layer: int) -> int:
    v = C.c_size_t()
    _check(load().kvev_plan_scores_offset(handle, B, S_cap, layer, C.byref(v)),
           "kvev_plan_scores_offset")
    return v.value


def kvev_plan_enable_timing(handle: int, on: bool = True):
    _check(load().kvev_plan_enable_timing(handle, int(bool(on))), "kvev_plan_enable_timing")


def kvev_plan_last_timings(handle: int) -> dict:
    """Per-kernel device milliseconds of the last timed call ({name: ms}, -1 if not launched)."""
    ms = np.zeros(len(KERNEL_NAMES), np.float32)
    _check(load().kvev_plan_last_timings(handle, ms.ctypes.data, len(ms)), "kvev_plan_last_timings")
    return {k: float(v) for k, v in zip(KERNEL_NAMES, ms)}


def kvev_plan_set_wait_limit(handle: int, ns: int):
    _check(load().kvev_plan_set_wait_limit(handle, int(ns)), "kvev_plan_set_wait_limit")


def kvev_plan_debug_stall_unit(handle: int, unit: int):
    _check(load().kvev_plan_debug_stall_unit(handle, int(unit)), "kvev_plan_debug_stall_unit")


def kvev_profile_cosine(h_full, h_cand) -> np.ndarray:
    """Sec. 3.2 cosine profile: h_full [L, D], h_cand [R, L, D] -> C [L, R] (fp64)."""
    hf = np.ascontiguousarray(h_full, np.float32)
    hc = np.ascontiguousarray(h_cand, np.float32)
    L, D = hf.shape
    R = hc.shape[0]
    assert hc.shape == (R, L, D)
    out = np.zeros((L, R), np.float64)
    _check(load().kvev_profile_cosine(out.ctypes.data, hf.ctypes.data, hc.ctypes.data, L, R, D),
           "kvev_profile_cosine")
    return out


def kvev_score_ppl(ppl, ppl_full: float) -> np.ndarray:
    """Sec. 3.3 PPL allocation score: max_r (ppl[l, r] - ppl_full)."""
    p = np.ascontiguousarray(ppl, np.float64)
    L, R = p.shape
    out = np.zeros(L, np.float64)
    _check(load().kvev_score_ppl(out.ctypes.data, p.ctypes.data, float(ppl_full), L, R), "kvev_score_ppl")
    return out


def kvev_score_entropy(A) -> np.ndarray:
    """Sec. 3.3 entropy allocation score of attention rows A [L, rows, K] (nats)."""
    a = np.ascontiguousarray(A, np.float32)
    L, rows, K = a.shape
    out = np.zeros(L, np.float64)
    _check(load().kvev_score_entropy(out.ctypes.data, a.ctypes.data, L, rows, K), "kvev_score_entropy")
    return out


def kvev_route_toprank(g, ops, higher_is_better: bool, covered=None) -> np.ndarray:
    """Eq. (policy_routing): per layer, the operator of the best covered column of g [L, R]."""
    gg = np.ascontiguousarray(g, np.float64)
    L, R = gg.shape
    o = np.ascontiguousarray(ops, np.int32)
    cv = None if covered is None else np.ascontiguousarray(covered, np.uint8)
    out = np.zeros(L, np.int32)
    _check(load().kvev_route_toprank(out.ctypes.data, gg.ctypes.data, L, R, o.ctypes.data,
                                     None if cv is None else cv.ctypes.data, int(bool(higher_is_better))),
           "kvev_route_toprank")
    return out


def kvev_route_install(route, scope: int):
    """Active phases of the scope take route[l], the others FULL: (route_prefill, route_decode)."""
    r = np.ascontiguousarray(route, np.int32)
    pre, dec = np.zeros(len(r), np.int32), np.zeros(len(r), np.int32)
    _check(load().kvev_route_install(pre.ctypes.data, dec.ctypes.data, r.ctypes.data, len(r), int(scope)),
           "kvev_route_install")
    return pre, dec


def kvev_plan_save(handle: int) -> bytes:
    n = C.c_size_t(0)
    _check(load().kvev_plan_save(handle, None, C.byref(n)), "kvev_plan_save")
    buf = C.create_string_buffer(n.value)
    _check(load().kvev_plan_save(handle, buf, C.byref(n)), "kvev_plan_save")
    return buf.raw[:n.value]


def kvev_plan_load(data: bytes) -> int:
    h = C.c_void_p()
    buf = C.create_string_buffer(bytes(data), len(data))
    _check(load().kvev_plan_load(C.byref(h), buf, len(data)), "kvev_plan_load")
    return h.value


# ---------------------------------------------------------------------------
# Convenience: a plan plus its buffers, with torch tensors as device memory
# ---------------------------------------------------------------------------

class Plan:
    """Owns a kvev plan; allocates outputs/workspace as torch CUDA tensors."""

    def __init__(self, L, H_q, H_kv, d, route, budget, window, pool_kernel=7, pool_type=POOL_AVG,
                 sink=4, recent=-1, h2o_recent=-1, route_decode=None, h2o_full_prompt=False):
        self.L, self.H_q, self.H_kv, self.d = L, H_q, H_kv, d
        self.route = np.asarray(route, np.int32)
        self.budget = np.asarray(budget, np.int32)
        self.window = window
        self.handle = kvev_plan_create(L, H_q, H_kv, d, self.route, route_decode, self.budget,
                                       window, pool_kernel, pool_type, sink, recent, h2o_recent)
        if h2o_full_prompt:
            _check(load().kvev_plan_set_h2o_full_prompt(self.handle, 1), "kvev_plan_set_h2o_full_prompt")

    def set_h2o_full_prompt(self, on: bool = True):
        """H2O layers score every prompt query row (their Q_win is then the
        whole prompt's queries, [B][H_q][S_cap][d])."""
        _check(load().kvev_plan_set_h2o_full_prompt(self.handle, 1 if on else 0),
               "kvev_plan_set_h2o_full_prompt")

    @classmethod
    def from_workload(cls, wl):
        return cls(wl.L, wl.H_q, wl.H_kv, wl.d, wl.route, wl.budget, wl.W, wl.pool_kernel,
                   wl.pool_type, wl.sink, wl.recent, wl.h2o_recent, wl.route_decode)

    def close(self):
        if self.handle:
            kvev_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def query(self, B, S_cap):
        return kvev_plan_query(self.handle, B, S_cap)

    def save(self) -> bytes:
        """The plan's serialised definition (Sec. 3.4)."""
        return kvev_plan_save(self.handle)

    @classmethod
    def load(cls, data: bytes) -> "Plan":
        """A plan recreated from kvev_plan_save bytes."""
        obj = cls.__new__(cls)
        obj.handle = kvev_plan_load(data)
        words = np.frombuffer(bytes(data)[8:-8], dtype="<i4")
        L = int(words[0])
        obj.L, obj.H_q, obj.H_kv, obj.d, obj.window = L, int(words[1]), int(words[2]), int(words[3]), int(words[4])
        obj.route = words[10:10 + L].astype(np.int32)
        obj.budget = words[10 + 2 * L:10 + 3 * L].astype(np.int32)
        return obj

    def layer_offset(self, B, layer):
        return kvev_plan_layer_offset(self.handle, B, layer)

    def buffers(self, B, S_cap, device="cuda"):
        import torch
        kv_bytes, idx_bytes, cnt_bytes, ws_bytes = self.query(B, S_cap)
        rows = idx_bytes // 4
        return {
            "out_K": torch.empty((max(rows, 1), self.d), dtype=torch.bfloat16, device=device),
            "out_V": torch.empty((max(rows, 1), self.d), dtype=torch.bfloat16, device=device),
            "out_idx": torch.empty(max(rows, 1), dtype=torch.int32, device=device),
            "out_count": torch.empty((self.L, B, self.H_kv), dtype=torch.int32, device=device),
            "h2o_state": torch.empty(max(rows, 1), dtype=torch.float32, device=device),
            "workspace": torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=device),
            "rows": rows,
        }

    def evict_prefill(self, K, V, Q, lens, B, S_cap, bufs, stream=None, check=True, scores=None,
                      lse=None) -> int:
        """K, V, Q: lists (per layer) of CUDA tensors or None; lens: int32 CUDA tensor.
        scores: optional per-layer fp32 [B][H_kv][S_cap] CUDA tensors (or None) that a
        caller's own attention produced for SnapKV / H2O layers (kvev_evict_prefill_scored).
        lse: optional per-layer fp32 [B][H_q][W] CUDA tensors (or None): the window rows'
        log-sum-exp from the caller's prefill attention (kvev_evict_prefill_lse)."""
        import torch
        if stream is None:
            stream = torch.cuda.current_stream()
        ptr = lambda t: None if t is None else t.data_ptr()
        if lse is not None:
            rc = kvev_evict_prefill_lse(
                self.handle, [ptr(k) for k in K], [ptr(v) for v in V],
                [ptr(q) for q in Q] if Q is not None else None, [ptr(x) for x in lse], lens.data_ptr(),
                B, S_cap, bufs["out_K"].data_ptr(), bufs["out_V"].data_ptr(), bufs["out_idx"].data_ptr(),
                bufs["out_count"].data_ptr(), bufs["h2o_state"].data_ptr(), bufs["workspace"].data_ptr(),
                bufs["workspace"].numel(), stream.cuda_stream)
            if check:
                _check(rc, "kvev_evict_prefill_lse")
            return rc
        if scores is not None:
            rc = kvev_evict_prefill_scored(
                self.handle, [ptr(k) for k in K], [ptr(v) for v in V],
                [ptr(q) for q in Q] if Q is not None else None, [ptr(x) for x in scores], lens.data_ptr(),
                B, S_cap, bufs["out_K"].data_ptr(), bufs["out_V"].data_ptr(), bufs["out_idx"].data_ptr(),
                bufs["out_count"].data_ptr(), bufs["h2o_state"].data_ptr(), bufs["workspace"].data_ptr(),
                bufs["workspace"].numel(), stream.cuda_stream)
            if check:
                _check(rc, "kvev_evict_prefill_scored")
            return rc
        rc = kvev_evict_prefill(
            self.handle, [ptr(k) for k in K], [ptr(v) for v in V],
            [ptr(q) for q in Q] if Q is not None else None, lens.data_ptr(), B, S_cap,
            bufs["out_K"].data_ptr(), bufs["out_V"].data_ptr(), bufs["out_idx"].data_ptr(),
            bufs["out_count"].data_ptr(), bufs["h2o_state"].data_ptr(),
            bufs["workspace"].data_ptr(), bufs["workspace"].numel(), stream.cuda_stream)
        if check:
            _check(rc, "kvev_evict_prefill")
        return rc

    def status(self) -> int:
        return kvev_status(self.handle)

    def scores(self, bufs, B, S_cap, layer):
        """fp32 window scores [B][H_kv][S_cap] of a SnapKV/H2O layer (a view of the workspace)."""
        import torch
        off = kvev_plan_scores_offset(self.handle, B, S_cap, layer)
        n = B * self.H_kv * S_cap
        return bufs["workspace"][off: off + 4 * n].view(torch.float32).view(B, self.H_kv, S_cap)


class DecodeArena:
    """Decode-phase caches of a Plan for B sequences (torch CUDA tensors as memory)."""

    def __init__(self, plan: "Plan", B: int, growth: int = 0, device="cuda"):
        import torch
        self.plan, self.B, self.growth = plan, B, growth
        self.rows, state_bytes = kvev_decode_query(plan.handle, B, growth)
        self.K = torch.empty((max(self.rows, 1), plan.d), dtype=torch.bfloat16, device=device)
        self.V = torch.empty_like(self.K)
        self.state = torch.zeros(max(state_bytes, 256), dtype=torch.uint8, device=device)
        self.off = kvev_decode_state_offsets(plan.handle, B, growth)
        self.layers = [kvev_decode_layer(plan.handle, B, growth, l) for l in range(plan.L)]
        self.units = sum(B * plan.H_kv for (_, cap, _) in self.layers if cap > 0)

    def _view(self, name, dtype, n):
        import torch
        o = self.off[name]
        return self.state[o: o + 4 * n].view(dtype)

    def lens(self):
        import torch
        return self._view("lens", torch.int32, self.B)

    def count(self):
        import torch
        return self._view("count", torch.int32, self.units)

    def evicted(self):
        import torch
        return self._view("evicted", torch.int32, self.units)

    def pos(self):
        import torch
        return self._view("pos", torch.int32, self.rows)

    def acc(self):
        import torch
        return self._view("acc", torch.float32, self.rows)

    def init_from_prefill(self, bufs, lens, stream=None):
        import torch
        if stream is None:
            stream = torch.cuda.current_stream()
        _check(kvev_decode_init(self.plan.handle, self.B, self.growth, bufs["out_K"].data_ptr(),
                                bufs["out_V"].data_ptr(), bufs["out_idx"].data_ptr(),
                                bufs["out_count"].data_ptr(), bufs["h2o_state"].data_ptr(),
                                lens.data_ptr(), self.K.data_ptr(), self.V.data_ptr(),
                                self.state.data_ptr(), stream.cuda_stream), "kvev_decode_init")

    def step_attn(self, k_new, v_new, attn, stream=None):
        """Decode step with caller-supplied attention: attn[l] fp32 [B][H_kv][cap_l + 1]
        CUDA tensors for H2O / TOVA layers (None elsewhere)."""
        import torch
        if stream is None:
            stream = torch.cuda.current_stream()
        ptr = lambda t: None if t is None else t.data_ptr()
        _check(kvev_decode_step_attn(self.plan.handle, self.B, self.growth, self.K.data_ptr(),
                                     self.V.data_ptr(), self.state.data_ptr(), [ptr(t) for t in k_new],
                                     [ptr(t) for t in v_new], [ptr(t) for t in attn],
                                     stream.cuda_stream), "kvev_decode_step_attn")

    def step(self, k_new, v_new, q_new, stream=None):
        """k_new, v_new, q_new: per-layer CUDA tensors (or None for layers without an arena)."""
        import torch
        if stream is None:
            stream = torch.cuda.current_stream()
        ptr = lambda t: None if t is None else t.data_ptr()
        _check(kvev_decode_step(self.plan.handle, self.B, self.growth, self.K.data_ptr(),
                                self.V.data_ptr(), self.state.data_ptr(), [ptr(t) for t in k_new],
                                [ptr(t) for t in v_new], [ptr(t) for t in q_new],
                                stream.cuda_stream), "kvev_decode_step")
