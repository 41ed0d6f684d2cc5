"""Host-side checks of the C ABI (no GPU): the library loads, exports every entry point that
include/deltas.h declares, sizes workspaces, and rejects bad arguments before enqueueing
anything (so these calls never touch a device)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    from paper_2609_27470_gb300 import build
    build.build()
    from paper_2609_27470_gb300 import _lib
    return _lib


def _declared():
    src = open(os.path.join(ROOT, "include", "deltas.h")).read()
    return sorted(set(re.findall(r"DELTAS_API\s+[\w\s\*]+?\b(deltas_\w+)\s*\(", src)))


def test_every_declared_symbol_is_exported(L):
    names = _declared()
    assert len(names) == 26, names
    lib = ctypes.CDLL(L.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(L.EXPORTED)


def test_version_and_status_strings(L):
    assert L.deltas_version().startswith("deltas ") and "sm_103a" in L.deltas_version()
    for code in range(0, 7):
        assert L.deltas_status_string(code) != "unknown status"
    assert L.deltas_status_string(99) == "unknown status"


def test_workspace_sizes(L):
    d = L.GdnDesc(24, 16, 32, 128, 128, L.DELTAS_BF16, 0.088)
    assert L.deltas_gdn_chunk_update_workspace_size(d, 1024) >= 16
    # the read-out keeps each token's write (512 B per token-head) and every 128-token block's
    # starting state (64 KiB per block-head) beyond the factor records; only d = 128 bf16 has them
    plain, ro = (L.deltas_gdn_chunk_update_workspace_size(d, 1024),
                 L.deltas_gdn_chunk_update_readout_workspace_size(d, 1024))
    assert ro - plain >= 24 * 32 * (1024 * 512 + 8 * 65536)
    d64 = L.GdnDesc(2, 2, 4, 64, 64, L.DELTAS_BF16, 0.125)
    assert (L.deltas_gdn_chunk_update_readout_workspace_size(d64, 100) ==
            L.deltas_gdn_chunk_update_workspace_size(d64, 100))
    assert L.deltas_state_drift_workspace_size(d) >= 16
    a = L.deltas_select_retain_workspace_size(1000)
    b = L.deltas_select_retain_workspace_size(100000)
    assert 16 <= a < b
    kv = L.KvDesc(8, 2, 256, L.DELTAS_BF16, 65536)
    assert L.deltas_compact_kv_workspace_size(kv, 65536) > L.deltas_compact_kv_workspace_size(kv, 1024) > 0
    bad = L.KvDesc(8, 2, 3, L.DELTAS_BF16, 100)   # 6-byte rows: not a multiple of 16 bytes
    assert L.deltas_compact_kv_workspace_size(bad, 10) == 0


FAKE = 0x10000   # a 256-byte aligned non-NULL address: every call below must reject before using it


def test_gdn_update_argument_checks(L):
    raw = L.raw()
    ok = L.GdnDesc(1, 2, 4, 16, 16, L.DELTAS_F32, 0.25)
    args = lambda desc, T=8, ws=FAKE, wsb=1 << 20: (ctypes.byref(desc) if desc else None, T, FAKE, FAKE, FAKE,
                                                     FAKE, FAKE, FAKE, None, None, ws, wsb, None)
    assert raw.deltas_gdn_chunk_update(*args(None)) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert raw.deltas_gdn_chunk_update(*args(L.GdnDesc(1, 3, 4, 16, 16, 0, 1.0))) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert raw.deltas_gdn_chunk_update(*args(L.GdnDesc(1, 2, 4, 48, 48, 0, 1.0))) == L.DELTAS_ERR_UNSUPPORTED
    assert raw.deltas_gdn_chunk_update(*args(L.GdnDesc(1, 2, 4, 64, 32, 0, 1.0))) == L.DELTAS_ERR_UNSUPPORTED
    assert raw.deltas_gdn_chunk_update(*args(L.GdnDesc(1, 2, 4, 16, 16, 7, 1.0))) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert raw.deltas_gdn_chunk_update(*args(ok, T=-1)) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert raw.deltas_gdn_chunk_update(*args(ok, ws=None)) == L.DELTAS_ERR_WORKSPACE
    assert raw.deltas_gdn_chunk_update(*args(ok, ws=FAKE + 8)) == L.DELTAS_ERR_WORKSPACE
    assert raw.deltas_gdn_chunk_update(*args(ok, wsb=4)) == L.DELTAS_ERR_WORKSPACE
    # misaligned key pointer
    assert raw.deltas_gdn_chunk_update(ctypes.byref(ok), 8, FAKE, FAKE + 4, FAKE, FAKE, FAKE, FAKE, None, None,
                                       FAKE, 1 << 20, None) == L.DELTAS_ERR_INVALID_ARGUMENT
    # output requested without q
    assert raw.deltas_gdn_chunk_update(ctypes.byref(ok), 8, None, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None,
                                       FAKE, 1 << 20, None) == L.DELTAS_ERR_INVALID_ARGUMENT


def test_select_argument_checks(L):
    raw = L.raw()

    def call(pol, T=100, nch=10, ws=FAKE, wsb=1 << 24):
        return raw.deltas_select_retain(ctypes.byref(pol) if pol else None, T, nch, FAKE, FAKE, FAKE, FAKE,
                                        None, ws, wsb, None)
    assert call(None) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert call(L.Policy(10, 5, 5, 1)) == L.DELTAS_ERR_INVALID_ARGUMENT     # M < n_s + n_w + 1
    assert call(L.Policy(10, 0, 0, 33)) == L.DELTAS_ERR_UNSUPPORTED
    assert call(L.Policy(10, 0, 0, -1)) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert call(L.Policy(10, 0, 0, 1), T=-5) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert call(L.Policy(10, 0, 0, 1), wsb=16) == L.DELTAS_ERR_WORKSPACE
    assert call(L.Policy(10, 0, 0, 1), T=(1 << 20) + 1) == L.DELTAS_ERR_UNSUPPORTED   # beyond the run scan


def test_compact_and_append_argument_checks(L):
    raw = L.raw()
    kv = L.KvDesc(2, 2, 64, L.DELTAS_BF16, 1000)
    assert raw.deltas_compact_kv(ctypes.byref(kv), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1001, FAKE, 1 << 24,
                                 None) == L.DELTAS_ERR_INVALID_ARGUMENT      # cache_len > capacity
    assert raw.deltas_compact_kv(ctypes.byref(kv), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 500, FAKE, 64,
                                 None) == L.DELTAS_ERR_WORKSPACE
    bad = L.KvDesc(2, 2, 7, L.DELTAS_F32, 1000)
    assert raw.deltas_compact_kv(ctypes.byref(bad), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 500, FAKE, 1 << 24,
                                 None) == L.DELTAS_ERR_UNSUPPORTED
    assert raw.deltas_append_kv(ctypes.byref(kv), FAKE, FAKE, FAKE, FAKE, 990, FAKE, FAKE, 20, 0, 0,
                                None) == L.DELTAS_ERR_INVALID_ARGUMENT       # overflows capacity
    assert raw.deltas_score_chunks(0, 4, FAKE, 0, FAKE, None) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert raw.deltas_score_chunks(2, 4, FAKE, -1, FAKE, None) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert raw.deltas_clear_device_status(None, None) == L.DELTAS_ERR_WORKSPACE


def test_binding_refuses_cpu_tensors(L):
    import torch
    d = L.gdn_desc(1, 1, 1, 16, torch.float32)
    x = torch.zeros(1, 4, 1, 16)
    with pytest.raises(ValueError):
        L.deltas_gdn_chunk_update(d, 4, x, x, x, torch.zeros(1, 4, 1), torch.zeros(1, 4, 1),
                                  torch.zeros(1, 1, 16, 16), None, None, torch.zeros(256, dtype=torch.uint8))


def test_copy_stream_state_argument_checks(L):
    """Snapshot / restore (deltas_copy_stream_state): every bad argument is refused on the host
    before anything is enqueued (the addresses below are never dereferenced)."""
    raw = L.raw()
    gdn = L.GdnDesc(2, 2, 4, 16, 16, L.DELTAS_F32, 0.25)
    kv = L.KvDesc(2, 2, 64, L.DELTAS_BF16, 1000)
    MB = 1 << 20
    full = lambda base: L.StreamBuffers(base, base + MB, base + 2 * MB, base + 3 * MB, base + 4 * MB, base + 5 * MB)
    light = lambda base: L.StreamBuffers(base, base + MB, None, None, None, None)

    def call(src, dst, kvd=kv, cache_len=500, n_chunks=7, desc=gdn):
        return raw.deltas_copy_stream_state(ctypes.byref(desc) if desc else None,
                                            ctypes.byref(kvd) if kvd else None, cache_len, n_chunks,
                                            ctypes.byref(src) if src else None, ctypes.byref(dst) if dst else None,
                                            None)
    A, B = 1 << 28, 1 << 30
    bad = L.DELTAS_ERR_INVALID_ARGUMENT
    assert call(full(A), full(B), desc=None) == bad
    assert call(None, full(B)) == bad
    assert call(full(A), None) == bad
    assert call(full(A), full(B), n_chunks=-1) == bad
    assert call(full(A), full(B), cache_len=1001) == bad                 # past the capacity
    assert call(full(A), full(B), cache_len=-1) == bad
    assert call(full(A), full(B), kvd=None) == bad                       # cache pointers without a kv desc
    assert call(light(A), light(B), kvd=kv) == bad                       # a kv desc without cache pointers
    mis = full(A)
    mis.v_cache = A + 3 * MB + 8                                          # not 16-byte aligned
    assert call(mis, full(B)) == bad
    assert call(full(A), full(A)) == bad                                 # a set copied onto itself
    ov = full(B)
    ov.state = A + 2 * MB + 4096                                          # inside the source k_cache
    assert call(full(A), ov) == bad
    assert call(full(A), full(B), kvd=L.KvDesc(2, 2, 7, L.DELTAS_F32, 1000)) == L.DELTAS_ERR_UNSUPPORTED
    assert call(full(A), full(B), desc=L.GdnDesc(2, 2, 4, 24, 24, L.DELTAS_F32, 0.25)) == L.DELTAS_ERR_UNSUPPORTED

    # the per-head variant (per-plane metadata and token scores)
    def heads(src, dst, kvd=kv, ss=A + 6 * MB, ds=B + 6 * MB):
        return raw.deltas_copy_stream_state_heads(ctypes.byref(gdn), ctypes.byref(kvd) if kvd else None, 500, 7,
                                                  ctypes.byref(src), ctypes.byref(dst), ss, ds, None)
    assert heads(full(A), full(B), kvd=None) == bad                       # the kv desc is required
    assert heads(full(A), full(B), ss=None) == bad
    assert heads(full(A), full(B), ds=B + 6 * MB + 4) == bad              # not 16-byte aligned
    assert heads(full(A), full(B), kvd=L.KvDesc(2, 2, 64, L.DELTAS_BF16, 1002)) == bad   # capacity % 4
    assert heads(full(A), full(B), ds=A + 6 * MB) == bad                  # scores copied onto themselves


def test_write_norm_argument_checks(L):
    """The comparison-signal entry points refuse bad arguments on the host."""
    raw = L.raw()
    ok = L.GdnDesc(1, 2, 4, 16, 16, L.DELTAS_F32, 0.25)
    bad = L.DELTAS_ERR_INVALID_ARGUMENT
    call = lambda wn: raw.deltas_gdn_chunk_update_write_norms(ctypes.byref(ok), 8, None, FAKE, FAKE, FAKE, FAKE,
                                                              FAKE, None, None, wn, FAKE, 1 << 20, None)
    assert call(None) == bad                                            # the output is required here
    assert call(FAKE + 4) == bad                                        # misaligned
    assert raw.deltas_score_write_norms(0, 4, FAKE, 10, 0, FAKE, None) == bad
    assert raw.deltas_score_write_norms(2, 4, FAKE, -1, 0, FAKE, None) == bad
    assert raw.deltas_score_write_norms(2, 4, FAKE, 10, -1, FAKE, None) == bad
    assert raw.deltas_score_write_norms(2, 4, None, 10, 0, FAKE, None) == bad


def test_token_signal_argument_checks(L):
    """The per-head calls of the Sec. 4.3 token signals reject bad arguments on the host."""
    raw = L.raw()
    kv = L.KvDesc(2, 2, 64, L.DELTAS_BF16, 1000)
    K = L.DELTAS_SIGNAL_KEY_NORM

    def append(signal=K, score=FAKE, cache_len=10, n_new=20):
        return raw.deltas_append_kv_heads(ctypes.byref(kv), signal, FAKE, FAKE, FAKE, FAKE, score, cache_len,
                                          FAKE, FAKE, n_new, 0, 0, None)
    assert append(signal=0) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert append(signal=3) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert append(score=None) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert append(cache_len=990) == L.DELTAS_ERR_INVALID_ARGUMENT           # past capacity
    assert append(n_new=-1) == L.DELTAS_ERR_INVALID_ARGUMENT

    def select(pol, planes=4, T=100, stride=100, ws=FAKE, wsb=1 << 24):
        return raw.deltas_select_retain_heads(ctypes.byref(pol) if pol else None, planes, T, stride, FAKE, FAKE,
                                              FAKE, FAKE, None, ws, wsb, None)
    ok = L.Policy(10, 0, 0, 1)
    assert select(None) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert select(L.Policy(10, 5, 5, 1)) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert select(L.Policy(10, 0, 0, 33)) == L.DELTAS_ERR_UNSUPPORTED
    assert select(ok, planes=0) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert select(ok, stride=99) == L.DELTAS_ERR_INVALID_ARGUMENT          # plane_stride < cache_len
    assert select(ok, T=(1 << 20) + 1, stride=(1 << 20) + 1) == L.DELTAS_ERR_UNSUPPORTED
    assert select(ok, wsb=16) == L.DELTAS_ERR_WORKSPACE
    small = L.deltas_select_retain_heads_workspace_size(4, 100)
    assert 16 < small < L.deltas_select_retain_heads_workspace_size(4, 10000)

    def compact(cache_len=500, stride=600, score=FAKE, wsb=1 << 24):
        return raw.deltas_compact_kv_heads(ctypes.byref(kv), FAKE, FAKE, FAKE, FAKE, score, FAKE, stride, FAKE,
                                           cache_len, FAKE, wsb, None)
    assert compact(cache_len=1001) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert compact(score=None) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert compact(stride=0) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert compact(wsb=64) == L.DELTAS_ERR_WORKSPACE
    big = L.KvDesc(8, 2, 256, L.DELTAS_BF16, 65536)
    assert L.deltas_compact_kv_heads_workspace_size(big, 65536) > L.deltas_compact_kv_workspace_size(big, 65536) > 0
