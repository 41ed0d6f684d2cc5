"""DeltaS CPU oracle: plain fp64 reference of the hot path (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
this package.  It shares no code with the CUDA library and never imports it; the two meet only
through the seeded input generators, which hold none of the method's arithmetic.

The arithmetic lives in ``deltas_oracle.c`` (compiled with gcc into ``oracle/_build``); this file
only marshals numpy arrays.  Each wrapper names the paper passage its C function follows:

* :func:`gdn_recurrence` — gated delta rule, residual form (Sec. 3.2, Eq. 2), token by token.
* :func:`gdn_recurrence_product_form` — the same rule in product form (Eq. 1), a self-check.
* :func:`drift_partials`, :func:`chunk_score` — state drift (Eq. 3; Alg. 1).
* :func:`select_retain` — sink / window / temporal spans / quota + fill (Sec. 3.3; Alg. 1).
* :func:`row_norm_scores`, :func:`select_retain_tokens`, :func:`compact_kv_heads` — the
  cache-internal token signals of the controlled comparison (Sec. 4.3: key norm, value norm; per KV
  head, per token) ranked under the same policy, and the per-head gather that follows.
* :func:`compact_rows`, :func:`compact_kv` — KV gather in stream order (Alg. 1; Sec. 3.3).
* :func:`stream` (in :mod:`oracle.stream`) — the Alg. 1 loop over a whole stream.

Parity status: the recurrence, drift, selection and compaction are each pinned by
``tests/test_oracle_pins.py`` (closed forms, exact-arithmetic brute force, a second formulation,
invariants).  Per-chunk drift values on real video are "parity unpinned": the paper prints none.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "deltas_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libdeltas_oracle.so")
_lock = threading.Lock()
_lib = None

_P = ctypes.c_void_p
_I = ctypes.c_int


def build(force: bool = False) -> str:
    """Compile ``deltas_oracle.c`` into ``oracle/_build/libdeltas_oracle.so`` (gcc -O2)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.oracle_gdn_recurrence.argtypes = [_I] * 6 + [_P] * 7 + [ctypes.c_double, _P]
            lib.oracle_gdn_recurrence.restype = _I
            lib.oracle_gdn_recurrence_product_form.argtypes = [_I] * 6 + [_P] * 5
            lib.oracle_gdn_recurrence_product_form.restype = _I
            lib.oracle_drift_partials.argtypes = [_I] * 4 + [_P] * 3
            lib.oracle_drift_partials.restype = _I
            lib.oracle_chunk_score.argtypes = [_I, _I, _P]
            lib.oracle_chunk_score.restype = ctypes.c_double
            lib.oracle_write_norm_score.argtypes = [_I, _I, _I, _P]
            lib.oracle_write_norm_score.restype = ctypes.c_double
            lib.oracle_select_retain.argtypes = [_I] * 6 + [_P] * 5
            lib.oracle_select_retain.restype = _I
            lib.oracle_compact_rows.argtypes = [_I] * 4 + [_P] * 3 + [_I]
            lib.oracle_compact_rows.restype = _I
            lib.oracle_row_norm_scores.argtypes = [_I, _I, _P, _I, _P]
            lib.oracle_row_norm_scores.restype = _I
            lib.oracle_select_retain_tokens.argtypes = [_I] * 5 + [_P] * 5
            lib.oracle_select_retain_tokens.restype = _I
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def _check(rc: int, what: str):
    if rc != 0:
        raise ValueError(f"oracle {what} rejected its arguments (code {rc})")


def gdn_recurrence(q, k, v, g, beta, state, q_scale: float | None = None, want_out: bool = False,
                   want_write_norms: bool = False):
    """Eq. 2 token loop.  Shapes: q,k [L,T,Hk,dk]; v [L,T,Hv,dv]; g,beta [L,T,Hv];
    state [L,Hv,dv,dk] (copied, not modified).  Returns ``(S_after, out_or_None)`` in fp64, and
    with ``want_write_norms`` a third item: [L,Hv] sums over the tokens of
    beta_t ||v_t - alpha_t S_{t-1} k_t||_2."""
    k = _f32(k)
    v = _f32(v)
    g = _f32(g)
    beta = _f32(beta)
    L, T, Hk, dk = k.shape
    Hv, dv = v.shape[2], v.shape[3]
    assert v.shape[:2] == (L, T) and g.shape == (L, T, Hv) and beta.shape == (L, T, Hv)
    S = np.array(state, dtype=np.float64, copy=True, order="C")
    assert S.shape == (L, Hv, dv, dk)
    qa = _f32(q) if q is not None else None
    out = np.zeros((L, T, Hv, dv), dtype=np.float64) if want_out else None
    if q_scale is None:
        q_scale = 1.0 / np.sqrt(dk)
    wn = np.zeros((L, Hv), dtype=np.float64) if want_write_norms else None
    rc = _load().oracle_gdn_recurrence(L, Hk, Hv, dk, dv, T, _ptr(qa), _ptr(k), _ptr(v), _ptr(g),
                                       _ptr(beta), _ptr(S), _ptr(out), float(q_scale), _ptr(wn))
    _check(rc, "gdn_recurrence")
    return (S, out, wn) if want_write_norms else (S, out)


def write_norm_score(write_norms, n_tokens: int) -> float:
    """The comparison signal's chunk score: write sizes averaged over heads, layers and tokens."""
    wn = np.ascontiguousarray(write_norms, dtype=np.float64)
    L, Hv = wn.shape
    return float(_load().oracle_write_norm_score(L, Hv, int(n_tokens), _ptr(wn)))


def gdn_recurrence_product_form(k, v, g, beta, state):
    """Eq. 1 token loop with an explicit transition matrix (self-check; small sizes only)."""
    k = _f32(k)
    v = _f32(v)
    g = _f32(g)
    beta = _f32(beta)
    L, T, Hk, dk = k.shape
    Hv, dv = v.shape[2], v.shape[3]
    S = np.array(state, dtype=np.float64, copy=True, order="C")
    rc = _load().oracle_gdn_recurrence_product_form(L, Hk, Hv, dk, dv, T, _ptr(k), _ptr(v), _ptr(g),
                                                    _ptr(beta), _ptr(S))
    _check(rc, "gdn_recurrence_product_form")
    return S


def drift_partials(s_before, s_after) -> np.ndarray:
    """Per (layer, head) [sum (S_after - S_before)^2, sum S_before^2] in fp64 (Eq. 3 parts)."""
    sb = np.ascontiguousarray(np.asarray(s_before, dtype=np.float64))
    sa = np.ascontiguousarray(np.asarray(s_after, dtype=np.float64))
    assert sb.shape == sa.shape and sb.ndim == 4
    L, Hv, dv, dk = sb.shape
    part = np.zeros((L, Hv, 2), dtype=np.float64)
    _check(_load().oracle_drift_partials(L, Hv, dv, dk, _ptr(sb), _ptr(sa), _ptr(part)), "drift_partials")
    return part


def chunk_score(partials) -> float:
    """Delta S of Eq. 3 from per (layer, head) partials, in fp64, with the zero-norm reading."""
    p = np.ascontiguousarray(np.asarray(partials, dtype=np.float64))
    L, Hv, two = p.shape
    assert two == 2
    return float(_load().oracle_chunk_score(L, Hv, _ptr(p)))


def state_drift(s_before, s_after) -> float:
    """Delta S straight from two states [L,Hv,dv,dk] (Eq. 3)."""
    return chunk_score(drift_partials(s_before, s_after))


def select_retain(budget_M: int, n_sink: int, n_window: int, n_buckets: int, tok_chunk, chunk_scores):
    """Sec. 3.3 / Alg. 1 retention.  Returns ``(retain_idx int32[n], mask uint8[T])``."""
    tc = np.ascontiguousarray(np.asarray(tok_chunk, dtype=np.int32))
    sc = _f32(chunk_scores)
    T = tc.shape[0]
    idx = np.zeros(max(T, 1), dtype=np.int32)
    mask = np.zeros(max(T, 1), dtype=np.uint8)
    n = ctypes.c_int32(0)
    rc = _load().oracle_select_retain(int(budget_M), int(n_sink), int(n_window), int(n_buckets), T,
                                      int(sc.shape[0]), _ptr(tc), _ptr(sc), _ptr(idx),
                                      ctypes.cast(ctypes.pointer(n), ctypes.c_void_p), _ptr(mask))
    _check(rc, "select_retain")
    return idx[: n.value].copy(), mask[:T].copy()


def compact_rows(planes: np.ndarray, retain_idx, cache_len: int) -> np.ndarray:
    """Out-of-place gather of rows: ``planes`` is [P, capacity, ...] of any dtype."""
    a = np.ascontiguousarray(planes)
    P, cap = a.shape[0], a.shape[1]
    row_bytes = a.dtype.itemsize * int(np.prod(a.shape[2:], dtype=np.int64))
    ri = np.ascontiguousarray(np.asarray(retain_idx, dtype=np.int32))
    out = np.empty_like(a)
    rc = _load().oracle_compact_rows(P, cap, row_bytes, int(cache_len), _ptr(a), _ptr(out), _ptr(ri),
                                     int(ri.shape[0]))
    _check(rc, "compact_rows")
    return out


def compact_kv(k_cache, v_cache, tok_chunk, tok_pos, retain_idx, cache_len: int):
    """Gather K [Lf,Hkv,cap,D], V (same), tok_chunk [cap], tok_pos [cap] by ``retain_idx``."""
    kc = np.asarray(k_cache)
    vc = np.asarray(v_cache)
    Lf, Hkv, cap = kc.shape[:3]
    k2 = compact_rows(kc.reshape(Lf * Hkv, cap, -1), retain_idx, cache_len).reshape(kc.shape)
    v2 = compact_rows(vc.reshape(Lf * Hkv, cap, -1), retain_idx, cache_len).reshape(vc.shape)
    tc = compact_rows(np.asarray(tok_chunk, dtype=np.int32).reshape(1, cap, 1), retain_idx, cache_len)
    tp = compact_rows(np.asarray(tok_pos, dtype=np.int32).reshape(1, cap, 1), retain_idx, cache_len)
    return k2, v2, tc.reshape(cap), tp.reshape(cap)


TOKEN_SIGNALS = ("key_norm", "value_norm")


def row_norm_scores(rows, signal: str) -> np.ndarray:
    """Token scores of the cache-internal signals (Sec. 4.3, appendix table of signals):
    ``key_norm`` -> -||k||_2 of each key row, ``value_norm`` -> ||v||_2 of each value row.
    ``rows`` is [..., D] (bf16 values widened exactly by the caller); the fp64 result is rounded
    to float32, the precision the paper computes every score in."""
    if signal not in TOKEN_SIGNALS:
        raise ValueError(f"unknown token signal {signal!r}")
    r = np.asarray(rows)
    shape = r.shape[:-1]
    D = r.shape[-1]
    a = _f32(r.reshape(-1, D))
    out = np.zeros(max(a.shape[0], 1), dtype=np.float64)
    rc = _load().oracle_row_norm_scores(int(a.shape[0]), int(D), _ptr(a), 1 if signal == "key_norm" else 0,
                                        _ptr(out))
    _check(rc, "row_norm_scores")
    return out[: a.shape[0]].astype(np.float32).reshape(shape)


def select_retain_tokens(budget_M: int, n_sink: int, n_window: int, n_buckets: int, tok_chunk, tok_scores):
    """Sec. 3.3 retention with one float32 score per slot (the token signals of Sec. 4.3).
    Returns ``(retain_idx int32[n], mask uint8[T])``."""
    tc = np.ascontiguousarray(np.asarray(tok_chunk, dtype=np.int32))
    sc = _f32(tok_scores)
    T = tc.shape[0]
    if sc.shape[0] != T:
        raise ValueError("one score per slot expected")
    idx = np.zeros(max(T, 1), dtype=np.int32)
    mask = np.zeros(max(T, 1), dtype=np.uint8)
    n = ctypes.c_int32(0)
    rc = _load().oracle_select_retain_tokens(int(budget_M), int(n_sink), int(n_window), int(n_buckets), T,
                                             _ptr(tc), _ptr(sc), _ptr(idx),
                                             ctypes.cast(ctypes.pointer(n), ctypes.c_void_p), _ptr(mask))
    _check(rc, "select_retain_tokens")
    return idx[: n.value].copy(), mask[:T].copy()


def compact_kv_heads(k_cache, v_cache, tok_chunk, tok_pos, tok_score, retain_lists, cache_len: int):
    """Per-head gather (each KV head keeps its own tokens): plane p = (layer, KV head) of K, V and
    of the per-head metadata tok_chunk / tok_pos / tok_score [Lf, Hkv, cap] is gathered by its own
    list ``retain_lists[p]`` (all lists have the same length)."""
    kc, vc = np.asarray(k_cache), np.asarray(v_cache)
    Lf, Hkv, cap = kc.shape[:3]
    P = Lf * Hkv
    if len(retain_lists) != P:
        raise ValueError("one retain list per (layer, KV head) plane expected")
    outs = []
    for arr in (kc, vc, tok_chunk, tok_pos, tok_score):
        a = np.asarray(arr).reshape(P, cap, -1)
        o = np.stack([compact_rows(a[p:p + 1], retain_lists[p], cache_len)[0] for p in range(P)])
        outs.append(o.reshape(np.asarray(arr).shape))
    return tuple(outs)
