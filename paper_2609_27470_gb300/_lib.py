"""ctypes binding of libdeltas (include/deltas.h): same names, argument marshalling only.

Tensors are torch CUDA tensors; each function checks device, dtype, shape and contiguity, passes
``data_ptr()`` values and the current CUDA stream to the C entry point, and raises
:class:`DeltasError` on a non-OK status.  All arithmetic happens in the library's kernels.
There is no fallback: importing this module fails if ``libdeltas.so`` has not been built.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdeltas.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it first (python -m paper_2609_27470_gb300.build)")

_lib = ctypes.CDLL(LIB_PATH)

DELTAS_OK = 0
DELTAS_ERR_INVALID_ARGUMENT = 1
DELTAS_ERR_UNSUPPORTED = 2
DELTAS_ERR_WORKSPACE = 3
DELTAS_ERR_CUDA = 4
DELTAS_ERR_TIMEOUT = 5
DELTAS_ERR_DEVICE_INDEX = 6
DELTAS_F32 = 0
DELTAS_BF16 = 1

EXPORTED = (
    "deltas_version", "deltas_status_string",
    "deltas_gdn_chunk_update_workspace_size", "deltas_gdn_chunk_update_readout_workspace_size",
    "deltas_gdn_chunk_update",
    "deltas_state_drift_workspace_size", "deltas_state_drift",
    "deltas_score_chunks", "deltas_gdn_chunk_update_write_norms", "deltas_score_write_norms",
    "deltas_select_retain_workspace_size", "deltas_select_retain", "deltas_select_retain_static",
    "deltas_compact_kv_workspace_size", "deltas_compact_kv",
    "deltas_append_kv", "deltas_copy_stream_state",
    "deltas_append_kv_heads", "deltas_select_retain_heads_workspace_size", "deltas_select_retain_heads",
    "deltas_compact_kv_heads_workspace_size", "deltas_compact_kv_heads", "deltas_copy_stream_state_heads",
    "deltas_clear_device_status", "deltas_set_wait_budget", "deltas_get_device_status",
)


class DeltasError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {deltas_status_string(status)} (status {status})")


class GdnDesc(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_k_heads", ctypes.c_int32),
                ("num_v_heads", ctypes.c_int32), ("key_dim", ctypes.c_int32),
                ("value_dim", ctypes.c_int32), ("dtype", ctypes.c_int32), ("q_scale", ctypes.c_float)]


class Policy(ctypes.Structure):
    _fields_ = [("budget_M", ctypes.c_int32), ("n_sink", ctypes.c_int32),
                ("n_window", ctypes.c_int32), ("n_buckets", ctypes.c_int32)]


class KvDesc(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("dtype", ctypes.c_int32), ("capacity", ctypes.c_int32)]


_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_SZ = ctypes.c_size_t


def _sig(name, res, *args):
    f = getattr(_lib, name)
    f.restype = res
    f.argtypes = list(args)
    return f


_sig("deltas_version", ctypes.c_char_p)
_sig("deltas_status_string", ctypes.c_char_p, _I32)
_sig("deltas_gdn_chunk_update_workspace_size", _SZ, _P, _I32)
_sig("deltas_gdn_chunk_update_readout_workspace_size", _SZ, _P, _I32)
_sig("deltas_gdn_chunk_update", ctypes.c_int, _P, _I32, _P, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P)
_sig("deltas_state_drift_workspace_size", _SZ, _P)
_sig("deltas_state_drift", ctypes.c_int, _P, _P, _P, _P, _P, _SZ, _P)
_sig("deltas_score_chunks", ctypes.c_int, _I32, _I32, _P, _I32, _P, _P)
_sig("deltas_gdn_chunk_update_write_norms", ctypes.c_int, _P, _I32, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P)
_sig("deltas_score_write_norms", ctypes.c_int, _I32, _I32, _P, _I32, _I32, _P, _P)
_sig("deltas_select_retain_workspace_size", _SZ, _I32)
_sig("deltas_select_retain", ctypes.c_int, _P, _I32, _I32, _P, _P, _P, _P, _P, _P, _SZ, _P)
_sig("deltas_select_retain_static", ctypes.c_int, _P, _I32, _I32, _P, _P, _P, _P, _P, _P)
_sig("deltas_compact_kv_workspace_size", _SZ, _P, _I32)
_sig("deltas_compact_kv", ctypes.c_int, _P, _P, _P, _P, _P, _P, _P, _I32, _P, _SZ, _P)
_sig("deltas_append_kv", ctypes.c_int, _P, _P, _P, _P, _P, _I32, _P, _P, _I32, _I32, _I32, _P)
_sig("deltas_copy_stream_state", ctypes.c_int, _P, _P, _I32, _I32, _P, _P, _P)
_sig("deltas_copy_stream_state_heads", ctypes.c_int, _P, _P, _I32, _I32, _P, _P, _P, _P, _P)
_sig("deltas_append_kv_heads", ctypes.c_int, _P, _I32, _P, _P, _P, _P, _P, _I32, _P, _P, _I32, _I32, _I32, _P)
_sig("deltas_select_retain_heads_workspace_size", _SZ, _I32, _I32)
_sig("deltas_select_retain_heads", ctypes.c_int, _P, _I32, _I32, _I32, _P, _P, _P, _P, _P, _P, _SZ, _P)
_sig("deltas_compact_kv_heads_workspace_size", _SZ, _P, _I32)
_sig("deltas_compact_kv_heads", ctypes.c_int, _P, _P, _P, _P, _P, _P, _P, _I32, _P, _I32, _P, _SZ, _P)
_sig("deltas_clear_device_status", ctypes.c_int, _P, _P)
_sig("deltas_set_wait_budget", ctypes.c_int, _P, ctypes.c_uint32, _P)
_sig("deltas_get_device_status", ctypes.c_int, _P, _P, _P, _P)

_TORCH_DT = {DELTAS_F32: torch.float32, DELTAS_BF16: torch.bfloat16}


def dtype_code(dt: torch.dtype) -> int:
    if dt == torch.float32:
        return DELTAS_F32
    if dt == torch.bfloat16:
        return DELTAS_BF16
    raise TypeError(f"unsupported dtype {dt}")


def deltas_version() -> str:
    return _lib.deltas_version().decode()


def deltas_status_string(status: int) -> str:
    return _lib.deltas_status_string(int(status)).decode()


def _stream(stream) -> int | None:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _ptr(t: torch.Tensor | None, dtype=None, shape=None, name="tensor"):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    return t.data_ptr()


def _check(status: int, where: str):
    if status != DELTAS_OK:
        raise DeltasError(status, where)


def gdn_desc(L, Hk, Hv, d, dtype: torch.dtype, q_scale: float | None = None) -> GdnDesc:
    return GdnDesc(L, Hk, Hv, d, d, dtype_code(dtype), float(q_scale if q_scale is not None else d ** -0.5))


def policy(budget_M, n_sink=0, n_window=0, n_buckets=1) -> Policy:
    return Policy(int(budget_M), int(n_sink), int(n_window), int(n_buckets))


def kv_desc(Lf, Hkv, D, dtype: torch.dtype, capacity) -> KvDesc:
    return KvDesc(int(Lf), int(Hkv), int(D), dtype_code(dtype), int(capacity))


def alloc_workspace(nbytes: int, device=None) -> torch.Tensor:
    """A zeroed uint8 workspace (the caching allocator returns 512-byte aligned blocks)."""
    ws = torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device or "cuda")
    assert ws.data_ptr() % 256 == 0
    return ws


def deltas_gdn_chunk_update_workspace_size(desc: GdnDesc, n_tokens: int) -> int:
    return int(_lib.deltas_gdn_chunk_update_workspace_size(ctypes.byref(desc), int(n_tokens)))


def deltas_gdn_chunk_update_readout_workspace_size(desc: GdnDesc, n_tokens: int) -> int:
    return int(_lib.deltas_gdn_chunk_update_readout_workspace_size(ctypes.byref(desc), int(n_tokens)))


def deltas_gdn_chunk_update(desc: GdnDesc, n_tokens: int, q, k, v, g, beta, state, out, drift_partials,
                            workspace, stream=None, write_norms=None):
    """The chunk update; with ``write_norms`` ([L, Hv] float32) the call is
    deltas_gdn_chunk_update_write_norms and also sums the tokens' write sizes."""
    L, Hk, Hv, dk, dv = desc.num_layers, desc.num_k_heads, desc.num_v_heads, desc.key_dim, desc.value_dim
    adt = _TORCH_DT[desc.dtype]
    T = int(n_tokens)
    args = [_ptr(q, adt, (L, T, Hk, dk), "q"), _ptr(k, adt, (L, T, Hk, dk), "k"),
            _ptr(v, adt, (L, T, Hv, dv), "v"), _ptr(g, torch.float32, (L, T, Hv), "g"),
            _ptr(beta, torch.float32, (L, T, Hv), "beta"),
            _ptr(state, torch.float32, (L, Hv, dv, dk), "state"),
            _ptr(out, adt, (L, T, Hv, dv), "out"),
            _ptr(drift_partials, torch.float32, (L, Hv, 2), "drift_partials")]
    tail = [_ptr(workspace, torch.uint8, None, "workspace"), workspace.numel(), _stream(stream)]
    if write_norms is None:
        st = _lib.deltas_gdn_chunk_update(ctypes.byref(desc), T, *args, *tail)
        _check(st, "deltas_gdn_chunk_update")
    else:
        st = _lib.deltas_gdn_chunk_update_write_norms(ctypes.byref(desc), T, *args,
                                                      _ptr(write_norms, torch.float32, (L, Hv), "write_norms"),
                                                      *tail)
        _check(st, "deltas_gdn_chunk_update_write_norms")


def deltas_score_write_norms(num_layers: int, num_v_heads: int, write_norms, n_tokens: int, chunk_id: int,
                             chunk_scores, stream=None):
    if chunk_scores.numel() <= chunk_id:
        raise ValueError("chunk_scores too short for chunk_id")
    st = _lib.deltas_score_write_norms(int(num_layers), int(num_v_heads),
                                       _ptr(write_norms, torch.float32, (num_layers, num_v_heads), "write_norms"),
                                       int(n_tokens), int(chunk_id),
                                       _ptr(chunk_scores, torch.float32, None, "chunk_scores"), _stream(stream))
    _check(st, "deltas_score_write_norms")


def deltas_state_drift_workspace_size(desc: GdnDesc) -> int:
    return int(_lib.deltas_state_drift_workspace_size(ctypes.byref(desc)))


def deltas_state_drift(desc: GdnDesc, s_before, s_after, drift_partials, workspace, stream=None):
    shp = (desc.num_layers, desc.num_v_heads, desc.value_dim, desc.key_dim)
    st = _lib.deltas_state_drift(ctypes.byref(desc), _ptr(s_before, torch.float32, shp, "s_before"),
                                 _ptr(s_after, torch.float32, shp, "s_after"),
                                 _ptr(drift_partials, torch.float32, (shp[0], shp[1], 2), "drift_partials"),
                                 _ptr(workspace, torch.uint8, None, "workspace"), workspace.numel(),
                                 _stream(stream))
    _check(st, "deltas_state_drift")


def deltas_score_chunks(num_layers: int, num_v_heads: int, drift_partials, chunk_id: int, chunk_scores,
                        stream=None):
    if chunk_scores.numel() <= chunk_id:
        raise ValueError("chunk_scores too short for chunk_id")
    st = _lib.deltas_score_chunks(int(num_layers), int(num_v_heads),
                                  _ptr(drift_partials, torch.float32, (num_layers, num_v_heads, 2), "drift_partials"),
                                  int(chunk_id), _ptr(chunk_scores, torch.float32, None, "chunk_scores"),
                                  _stream(stream))
    _check(st, "deltas_score_chunks")


def deltas_select_retain_workspace_size(cache_len: int) -> int:
    return int(_lib.deltas_select_retain_workspace_size(int(cache_len)))


def deltas_select_retain(pol: Policy, cache_len: int, tok_chunk, chunk_scores, retain_idx, n_retained,
                         mask, workspace, stream=None):
    T = int(cache_len)
    if tok_chunk.numel() < T or retain_idx.numel() < min(T, pol.budget_M) or (mask is not None and mask.numel() < T):
        raise ValueError("select_retain: an output or input is shorter than cache_len / budget")
    st = _lib.deltas_select_retain(ctypes.byref(pol), T, int(chunk_scores.numel()),
                                   _ptr(tok_chunk, torch.int32, None, "tok_chunk"),
                                   _ptr(chunk_scores, torch.float32, None, "chunk_scores"),
                                   _ptr(retain_idx, torch.int32, None, "retain_idx"),
                                   _ptr(n_retained, torch.int32, None, "n_retained"),
                                   _ptr(mask, torch.uint8, None, "mask"),
                                   _ptr(workspace, torch.uint8, None, "workspace"), workspace.numel(),
                                   _stream(stream))
    _check(st, "deltas_select_retain")


SELECT_STATIC_MAX_CACHE_LEN = 65536   # DELTAS_SELECT_STATIC_MAX_CACHE_LEN


def deltas_select_retain_static(pol: Policy, cache_len: int, tok_chunk, chunk_scores, retain_idx, n_retained,
                                mask, stream=None):
    """deltas_select_retain with the library's own fixed scratch: no workspace and no allocation."""
    T = int(cache_len)
    if tok_chunk.numel() < T or retain_idx.numel() < min(T, pol.budget_M) or (mask is not None and mask.numel() < T):
        raise ValueError("select_retain_static: an output or input is shorter than cache_len / budget")
    st = _lib.deltas_select_retain_static(ctypes.byref(pol), T, int(chunk_scores.numel()),
                                          _ptr(tok_chunk, torch.int32, None, "tok_chunk"),
                                          _ptr(chunk_scores, torch.float32, None, "chunk_scores"),
                                          _ptr(retain_idx, torch.int32, None, "retain_idx"),
                                          _ptr(n_retained, torch.int32, None, "n_retained"),
                                          _ptr(mask, torch.uint8, None, "mask"),
                                          _stream(stream))
    _check(st, "deltas_select_retain_static")


def deltas_compact_kv_workspace_size(desc: KvDesc, cache_len: int) -> int:
    return int(_lib.deltas_compact_kv_workspace_size(ctypes.byref(desc), int(cache_len)))


def deltas_compact_kv(desc: KvDesc, k_cache, v_cache, tok_chunk, tok_pos, retain_idx, n_retained,
                      cache_len: int, workspace, stream=None):
    dt = _TORCH_DT[desc.dtype]
    shp = (desc.num_layers, desc.num_kv_heads, desc.capacity, desc.head_dim)
    st = _lib.deltas_compact_kv(ctypes.byref(desc), _ptr(k_cache, dt, shp, "k_cache"), _ptr(v_cache, dt, shp, "v_cache"),
                                _ptr(tok_chunk, torch.int32, (desc.capacity,), "tok_chunk"),
                                _ptr(tok_pos, torch.int32, (desc.capacity,), "tok_pos"),
                                _ptr(retain_idx, torch.int32, None, "retain_idx"),
                                _ptr(n_retained, torch.int32, None, "n_retained"), int(cache_len),
                                _ptr(workspace, torch.uint8, None, "workspace"), workspace.numel(),
                                _stream(stream))
    _check(st, "deltas_compact_kv")


def deltas_append_kv(desc: KvDesc, k_cache, v_cache, tok_chunk, tok_pos, cache_len: int, k_new, v_new,
                     chunk_id: int, first_pos: int, stream=None):
    dt = _TORCH_DT[desc.dtype]
    shp = (desc.num_layers, desc.num_kv_heads, desc.capacity, desc.head_dim)
    n_new = int(k_new.shape[2])
    nshp = (desc.num_layers, desc.num_kv_heads, n_new, desc.head_dim)
    st = _lib.deltas_append_kv(ctypes.byref(desc), _ptr(k_cache, dt, shp, "k_cache"), _ptr(v_cache, dt, shp, "v_cache"),
                               _ptr(tok_chunk, torch.int32, (desc.capacity,), "tok_chunk"),
                               _ptr(tok_pos, torch.int32, (desc.capacity,), "tok_pos"), int(cache_len),
                               _ptr(k_new, dt, nshp, "k_new"), _ptr(v_new, dt, nshp, "v_new"), n_new,
                               int(chunk_id), int(first_pos), _stream(stream))
    _check(st, "deltas_append_kv")


# Per-head token signals (Sec. 4.3): the key norm scores -||k||, the value norm ||v||
DELTAS_SIGNAL_KEY_NORM = 1
DELTAS_SIGNAL_VALUE_NORM = 2
SIGNALS = {"key_norm": DELTAS_SIGNAL_KEY_NORM, "value_norm": DELTAS_SIGNAL_VALUE_NORM}


def deltas_append_kv_heads(desc: KvDesc, signal: str, k_cache, v_cache, tok_chunk, tok_pos, tok_score,
                           cache_len: int, k_new, v_new, chunk_id: int, first_pos: int, stream=None):
    """Append a chunk and score its tokens per (layer, KV head); metadata is [Lf, Hkv, capacity]."""
    dt = _TORCH_DT[desc.dtype]
    shp = (desc.num_layers, desc.num_kv_heads, desc.capacity, desc.head_dim)
    mshp = shp[:3]
    n_new = int(k_new.shape[2])
    nshp = (desc.num_layers, desc.num_kv_heads, n_new, desc.head_dim)
    st = _lib.deltas_append_kv_heads(ctypes.byref(desc), SIGNALS[signal], _ptr(k_cache, dt, shp, "k_cache"),
                                     _ptr(v_cache, dt, shp, "v_cache"), _ptr(tok_chunk, torch.int32, mshp, "tok_chunk"),
                                     _ptr(tok_pos, torch.int32, mshp, "tok_pos"),
                                     _ptr(tok_score, torch.float32, mshp, "tok_score"), int(cache_len),
                                     _ptr(k_new, dt, nshp, "k_new"), _ptr(v_new, dt, nshp, "v_new"), n_new,
                                     int(chunk_id), int(first_pos), _stream(stream))
    _check(st, "deltas_append_kv_heads")


def deltas_select_retain_heads_workspace_size(num_planes: int, cache_len: int) -> int:
    return int(_lib.deltas_select_retain_heads_workspace_size(int(num_planes), int(cache_len)))


def deltas_select_retain_heads(pol: Policy, cache_len: int, tok_chunk, tok_score, retain_idx, n_retained, mask,
                               workspace, stream=None):
    """Per-plane selection: tok_chunk / tok_score [..., plane_stride] (planes flattened), retain_idx
    [planes, M], mask [planes, plane_stride] or None."""
    T = int(cache_len)
    stride = int(tok_chunk.shape[-1])
    planes = tok_chunk.numel() // max(stride, 1)
    if tok_score.shape != tok_chunk.shape or stride < T:
        raise ValueError("select_retain_heads: tok_score must match tok_chunk, with at least cache_len slots")
    if retain_idx.numel() < planes * pol.budget_M or (mask is not None and tuple(mask.shape) != tuple(tok_chunk.shape)):
        raise ValueError("select_retain_heads: retain_idx needs [planes, M], mask the shape of tok_chunk")
    st = _lib.deltas_select_retain_heads(ctypes.byref(pol), planes, T, stride,
                                         _ptr(tok_chunk, torch.int32, None, "tok_chunk"),
                                         _ptr(tok_score, torch.float32, None, "tok_score"),
                                         _ptr(retain_idx, torch.int32, None, "retain_idx"),
                                         _ptr(n_retained, torch.int32, None, "n_retained"),
                                         _ptr(mask, torch.uint8, None, "mask"),
                                         _ptr(workspace, torch.uint8, None, "workspace"), workspace.numel(),
                                         _stream(stream))
    _check(st, "deltas_select_retain_heads")


def deltas_compact_kv_heads_workspace_size(desc: KvDesc, cache_len: int) -> int:
    return int(_lib.deltas_compact_kv_heads_workspace_size(ctypes.byref(desc), int(cache_len)))


def deltas_compact_kv_heads(desc: KvDesc, k_cache, v_cache, tok_chunk, tok_pos, tok_score, retain_idx, n_retained,
                            cache_len: int, workspace, stream=None):
    """Gather every (layer, KV head) plane by its own row of retain_idx [Lf * Hkv, list_stride]."""
    dt = _TORCH_DT[desc.dtype]
    shp = (desc.num_layers, desc.num_kv_heads, desc.capacity, desc.head_dim)
    mshp = shp[:3]
    planes = desc.num_layers * desc.num_kv_heads
    if retain_idx.dim() != 2 or retain_idx.shape[0] != planes:
        raise ValueError("compact_kv_heads: retain_idx must be [Lf * Hkv, list_stride]")
    st = _lib.deltas_compact_kv_heads(ctypes.byref(desc), _ptr(k_cache, dt, shp, "k_cache"),
                                      _ptr(v_cache, dt, shp, "v_cache"),
                                      _ptr(tok_chunk, torch.int32, mshp, "tok_chunk"),
                                      _ptr(tok_pos, torch.int32, mshp, "tok_pos"),
                                      _ptr(tok_score, torch.float32, mshp, "tok_score"),
                                      _ptr(retain_idx, torch.int32, None, "retain_idx"), int(retain_idx.shape[1]),
                                      _ptr(n_retained, torch.int32, None, "n_retained"), int(cache_len),
                                      _ptr(workspace, torch.uint8, None, "workspace"), workspace.numel(),
                                      _stream(stream))
    _check(st, "deltas_compact_kv_heads")


STREAM_BUFFERS = ("state", "chunk_scores", "k_cache", "v_cache", "tok_chunk", "tok_pos")


class StreamBuffers(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in STREAM_BUFFERS]


def deltas_copy_stream_state(gdn: GdnDesc, kv: KvDesc | None, cache_len: int, n_chunks: int, src: dict, dst: dict,
                             stream=None, per_head: bool = False):
    """Copy a stream state between two buffer sets (dicts keyed by STREAM_BUFFERS; the cache
    entries None when kv is None).  per_head: the metadata is [Lf, Hkv, capacity] and both dicts
    also hold "tok_score" (deltas_copy_stream_state_heads)."""
    sshape = (gdn.num_layers, gdn.num_v_heads, gdn.value_dim, gdn.key_dim)
    mshape = None if kv is None else ((kv.num_layers, kv.num_kv_heads, kv.capacity) if per_head else (kv.capacity,))
    shapes = {"state": (torch.float32, sshape), "chunk_scores": (torch.float32, None),
              "tok_chunk": (torch.int32, mshape), "tok_pos": (torch.int32, mshape)}
    if kv is not None:
        cshape = (kv.num_layers, kv.num_kv_heads, kv.capacity, kv.head_dim)
        shapes["k_cache"] = shapes["v_cache"] = (_TORCH_DT[kv.dtype], cshape)

    def pack(d, side):
        vals = []
        for n in STREAM_BUFFERS:
            t = d.get(n)
            if t is not None and n == "chunk_scores" and t.numel() < n_chunks:
                raise ValueError(f"{side} chunk_scores holds fewer than {n_chunks} entries")
            dt, shp = shapes.get(n, (None, None))
            vals.append(_ptr(t, dt, shp, f"{side} {n}"))
        return StreamBuffers(*vals)

    s, d = pack(src, "src"), pack(dst, "dst")
    if per_head:
        if kv is None:
            raise ValueError("a per-head stream state needs the kv descriptor")
        st = _lib.deltas_copy_stream_state_heads(ctypes.byref(gdn), ctypes.byref(kv), int(cache_len), int(n_chunks),
                                                 ctypes.byref(s), ctypes.byref(d),
                                                 _ptr(src["tok_score"], torch.float32, mshape, "src tok_score"),
                                                 _ptr(dst["tok_score"], torch.float32, mshape, "dst tok_score"),
                                                 _stream(stream))
        _check(st, "deltas_copy_stream_state_heads")
        return
    st = _lib.deltas_copy_stream_state(ctypes.byref(gdn), ctypes.byref(kv) if kv is not None else None,
                                       int(cache_len), int(n_chunks), ctypes.byref(s), ctypes.byref(d),
                                       _stream(stream))
    _check(st, "deltas_copy_stream_state")


def deltas_clear_device_status(workspace, stream=None):
    _check(_lib.deltas_clear_device_status(_ptr(workspace, torch.uint8, None, "workspace"), _stream(stream)),
           "deltas_clear_device_status")


def deltas_set_wait_budget(workspace, budget_ns: int, stream=None):
    """Bounded-wait budget of the kernels that run with this workspace (0: about one second)."""
    _check(_lib.deltas_set_wait_budget(_ptr(workspace, torch.uint8, None, "workspace"), int(budget_ns),
                                       _stream(stream)), "deltas_set_wait_budget")


def deltas_get_device_status(workspace, stream=None):
    s = ctypes.c_int32(0)
    d = ctypes.c_int32(0)
    _check(_lib.deltas_get_device_status(_ptr(workspace, torch.uint8, None, "workspace"), _stream(stream),
                                         ctypes.byref(s), ctypes.byref(d)), "deltas_get_device_status")
    return int(s.value), int(d.value)


def raw():
    """The underlying ctypes CDLL (for tests that call entry points with raw arguments)."""
    return _lib
