"""GPU parity of retain selection (Sec. 3.3, Alg. 1) and in-place KV compaction / append
(Alg. 1, Sec. 3.3) against the CPU oracle: bit-exact, given identical float32 scores."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2609_27470_gb300 import inputs

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def L():
    from paper_2609_27470_gb300 import _lib
    return _lib


def gpu_select(L, M, n_s, n_w, N, tok_chunk, scores):
    tc = torch.as_tensor(np.asarray(tok_chunk, np.int32)).cuda()
    sc = torch.as_tensor(np.asarray(scores, np.float32)).cuda()
    T = tc.numel()
    pol = L.policy(M, n_s, n_w, N)
    idx = torch.full((max(min(T, M), 1),), -7, dtype=torch.int32, device="cuda")
    n = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    mask = torch.full((max(T, 1),), 9, dtype=torch.uint8, device="cuda")
    ws = L.alloc_workspace(L.deltas_select_retain_workspace_size(T))
    L.deltas_select_retain(pol, T, tc, sc, idx, n, mask, ws)
    torch.cuda.synchronize()
    st = L.deltas_get_device_status(ws)
    nn = int(n.item())
    return idx[:nn].cpu().numpy(), mask[:T].cpu().numpy(), st


def _assert_same_selection(L, M, n_s, n_w, N, tc, sc):
    ref_idx, ref_mask = oracle.select_retain(M, n_s, n_w, N, tc, sc)
    idx, mask, st = gpu_select(L, M, n_s, n_w, N, tc, sc)
    assert st == (0, 0)
    assert np.array_equal(idx, ref_idx), (M, n_s, n_w, N, len(tc))
    assert np.array_equal(mask, ref_mask)


def test_select_golden_examples(L):
    for case in json.load(open(os.path.join(GOLDEN, "select_examples.json")))["cases"]:
        idx, mask, st = gpu_select(L, case["budget_M"], case["n_sink"], case["n_window"], case["n_buckets"],
                                   case["tok_chunk"], case["chunk_scores"])
        assert st == (0, 0)
        assert idx.tolist() == case["retain"], case["name"]


def test_select_random_small(L):
    rng = np.random.default_rng(101)
    for _ in range(300):
        n_ch = int(rng.integers(1, 30))
        tc = np.repeat(np.arange(n_ch, dtype=np.int32), rng.integers(1, 25, size=n_ch))
        sc = rng.exponential(size=n_ch).astype(np.float32)
        sc[rng.integers(0, n_ch, size=3)] = sc[0]              # exact ties
        T = len(tc)
        n_s = int(rng.integers(0, 6))
        n_w = int(rng.integers(0, 40))
        M = int(rng.integers(n_s + n_w + 1, max(T, n_s + n_w + 1) + 4))
        N = int(rng.integers(0, 9))
        _assert_same_selection(L, M, n_s, n_w, N, tc, sc)


def test_select_many_runs_and_odd_orders(L):
    """Runs of length 1 (chunk ids alternate), non-monotone chunk ids, repeated chunks, special
    float scores (+inf, -0.0, +0.0, negative)."""
    rng = np.random.default_rng(102)
    for _ in range(40):
        T = int(rng.integers(50, 5000))
        n_ch = int(rng.integers(2, 200))
        tc = rng.integers(0, n_ch, size=T).astype(np.int32)
        sc = rng.standard_normal(n_ch).astype(np.float32)
        sc[rng.integers(0, n_ch, size=4)] = np.float32(np.inf)
        sc[rng.integers(0, n_ch, size=2)] = np.float32(-0.0)
        sc[rng.integers(0, n_ch, size=2)] = np.float32(0.0)
        M = int(rng.integers(3, T))
        n_s = int(rng.integers(0, 2))
        n_w = int(rng.integers(0, 2))
        _assert_same_selection(L, M, n_s, n_w, int(rng.integers(1, 33)), tc, sc)


@pytest.mark.parametrize("variant", ["a", "b"])
def test_select_kv_workload(L, variant):
    """64k-token cache of 64 chunks x 1024, Exp(1) scores with 6 exact ties at the 16th-largest
    value, budget 16k; variant a: no sink/window, one span (exactly 16 chunks); variant b: the
    paper's n_s=4, n_w=1024, N=4."""
    tc = inputs.chunked_tok_chunk(64, 1024).numpy()
    sc = inputs.chunk_scores_with_ties(64, seed=3).numpy()
    if variant == "a":
        _assert_same_selection(L, 16384, 0, 0, 1, tc, sc)
    else:
        _assert_same_selection(L, 16384, 4, 1024, 4, tc, sc)


def test_select_streaming_shape(L):
    """Streaming workload's eviction input: cache of M + 512 = 33280 tokens after earlier
    evictions (chunks partially kept), paper policy, budget 32768."""
    rng = np.random.default_rng(104)
    kept_lens = rng.integers(1, 513, size=200)
    tc = np.concatenate([np.full(n, c, np.int32) for c, n in enumerate(kept_lens)])
    assert tc.size >= 32768
    tc = np.concatenate([tc[-32768:], np.full(512, 200, np.int32)])
    sc = rng.exponential(size=201).astype(np.float32)
    _assert_same_selection(L, 32768, 4, 1024, 4, tc, sc)


@pytest.mark.parametrize("T,n_ch,run_max", [(100000, 700, 400), (150000, 20000, 6), (262144, 900, 700),
                                            (262145, 900, 700), (300000, 30000, 6)])
def test_select_large_caches(L, T, n_ch, run_max):
    """Large caches through the grid-wide run scan, the decision kernel and the grid-wide
    emission: a few hundred long runs (ranked in shared memory) and tens of thousands of short
    ones (the radix path), 256k slots and one slot more, the paper's policy and exact score ties."""
    rng = np.random.default_rng(T + n_ch)
    lens = rng.integers(1, run_max + 1, size=4 * T // (run_max + 1) + 8)
    ids = np.sort(rng.integers(0, n_ch, size=lens.size)).astype(np.int32)
    tc = np.repeat(ids, lens)[:T].astype(np.int32)
    assert tc.size == T
    sc = rng.exponential(size=n_ch).astype(np.float32)
    sc[rng.integers(0, n_ch, size=6)] = sc[3]
    _assert_same_selection(L, T // 3, 4, 1024, 4, tc, sc)
    _assert_same_selection(L, T - 1, 0, 0, 1, tc, sc)


@pytest.mark.parametrize("T,run_max,n_s,n_w", [(65536, 6, 4, 1024), (65537, 6, 4, 1024), (65536, 1, 0, 0),
                                             (4097, 3, 1023, 1025), (2048, 1024, 1024, 0)])
def test_select_scan_block_edges(L, T, run_max, n_s, n_w):
    """Runs of 1 to run_max slots cross the run scan's 1024-slot block edges; a cache of 64k
    slots and one of a slot more (a one-slot last block); sink and window ends on and next to a
    block edge; one token per chunk makes 64k runs (the radix path)."""
    rng = np.random.default_rng(T + run_max)
    lens = rng.integers(1, run_max + 1, size=T)
    tc = np.repeat(np.arange(lens.size, dtype=np.int32), lens)[:T].astype(np.int32)
    n_ch = int(tc[-1]) + 1
    sc = rng.exponential(size=n_ch).astype(np.float32)
    sc[rng.integers(0, n_ch, size=6)] = sc[1]
    _assert_same_selection(L, T // 3 + n_s + n_w, n_s, n_w, 4, tc, sc)
    _assert_same_selection(L, T - 1, 0, 0, 1, tc, sc)


def test_select_edge_cases(L):
    rng = np.random.default_rng(105)
    tc = np.repeat(np.arange(10, dtype=np.int32), 10)
    sc = rng.exponential(size=10).astype(np.float32)
    _assert_same_selection(L, 100, 0, 0, 1, tc, sc)          # T == M: keep all
    _assert_same_selection(L, 1000, 4, 8, 4, tc, sc)         # T < M
    _assert_same_selection(L, 13, 6, 6, 4, tc, sc)           # M = n_s + n_w + 1
    _assert_same_selection(L, 50, 0, 0, 32, tc, sc)          # more spans than chunks
    _assert_same_selection(L, 50, 0, 0, 0, tc, sc)           # N = 0 read as one span
    _assert_same_selection(L, 99, 0, 0, 3, tc, sc)           # evict one token
    _assert_same_selection(L, 1, 0, 0, 1, tc, sc)            # budget of one
    idx, mask, st = gpu_select(L, 5, 0, 0, 1, np.zeros(0, np.int32), np.zeros(1, np.float32))
    assert st == (0, 0) and idx.size == 0


def test_select_reports_bad_chunk_ids(L):
    tc = np.array([0, 1, 2, 7, 3], np.int32)
    idx, mask, st = gpu_select(L, 2, 0, 0, 1, tc, np.ones(4, np.float32))
    assert st == (L.DELTAS_ERR_DEVICE_INDEX, 3)
    # bad ids in later scan blocks (one on a block edge): the last bad slot is reported
    for T in (3000, 70000):
        tc = np.repeat(np.arange(T // 10, dtype=np.int32), 10)
        tc[1024] = -1
        tc[T - 500] = T // 10
        idx, mask, st = gpu_select(L, T // 2, 0, 0, 1, tc, np.ones(T // 10, np.float32))
        assert st == (L.DELTAS_ERR_DEVICE_INDEX, T - 500)


# ----------------------------------------------------------------------------- compaction

def _gpu_compact(L, kc, vc, tc, tp, keep, cache_len):
    Lf, Hkv, cap, D = kc.shape
    desc = L.kv_desc(Lf, Hkv, D, kc.dtype, cap)
    k = kc.cuda()
    v = vc.cuda()
    t1 = tc.cuda()
    t2 = tp.cuda()
    idx = torch.zeros(max(len(keep), 1), dtype=torch.int32)
    idx[: len(keep)] = torch.as_tensor(np.asarray(keep, np.int32))
    idx = idx.cuda()
    n = torch.tensor([len(keep)], dtype=torch.int32, device="cuda")
    ws = L.alloc_workspace(L.deltas_compact_kv_workspace_size(desc, cache_len))
    L.deltas_compact_kv(desc, k, v, t1, t2, idx, n, cache_len, ws)
    torch.cuda.synchronize()
    return k.cpu(), v.cpu(), t1.cpu(), t2.cpu(), L.deltas_get_device_status(ws)


def _np(t):
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.numpy()


def _check_compact(L, kc, vc, keep, cache_len):
    cap = kc.shape[2]
    tc = torch.arange(cap, dtype=torch.int32) // 7
    tp = torch.arange(cap, dtype=torch.int32) + 1000
    k2, v2, t1, t2, st = _gpu_compact(L, kc, vc, tc, tp, keep, cache_len)
    assert st == (0, 0)
    rk, rv, rtc, rtp = oracle.compact_kv(_np(kc), _np(vc), tc.numpy(), tp.numpy(), keep, cache_len)
    assert np.array_equal(_np(k2), rk) and np.array_equal(_np(v2), rv)
    assert np.array_equal(t1.numpy(), rtc) and np.array_equal(t2.numpy(), rtp)


@pytest.mark.parametrize("dtype,D", [(torch.float32, 16), (torch.bfloat16, 256), (torch.bfloat16, 64),
                                     (torch.float32, 4)])
def test_compact_random(L, dtype, D):
    rng = np.random.default_rng(D)
    cap = 3000
    kc = torch.randn(2, 2, cap, D).to(dtype)
    vc = torch.randn(2, 2, cap, D).to(dtype)
    for cache_len, n in ((2900, 1000), (2000, 1999), (500, 1), (3000, 3000), (3000, 0)):
        keep = np.sort(rng.choice(cache_len, size=n, replace=False)).astype(np.int32)
        _check_compact(L, kc, vc, keep, cache_len)


def test_compact_patterns(L):
    """Identity (nothing moves), evict the first token only (everything moves by one), evict one
    early chunk, keep only the last tokens (long-distance moves)."""
    cap = 5000
    kc = torch.randn(1, 3, cap, 128).to(torch.bfloat16)
    vc = torch.randn(1, 3, cap, 128).to(torch.bfloat16)
    T = 4800
    for keep in (np.arange(3000), np.arange(1, T), np.r_[0:100, 600:T], np.arange(T - 700, T),
                 np.r_[0:4, 2000:2100, 4000:T]):
        _check_compact(L, kc, vc, keep.astype(np.int32), T)


def test_compact_kv_workload(L):
    """Full-size KV workload: 8 layers x 2 heads x 256 bf16, 64k tokens, budget 16k chosen by the
    selector (paper policy) -> the same moves as the benchmark."""
    Lf, Hkv, D, cap = 8, 2, 256, 65536
    kc, vc = inputs.kv_cache(Lf, Hkv, cap, D, "bf16", seed=21)
    tc = inputs.chunked_tok_chunk(64, 1024).numpy()
    sc = inputs.chunk_scores_with_ties(64, seed=3).numpy()
    keep, _ = oracle.select_retain(16384, 4, 1024, 4, tc, sc)
    _check_compact(L, kc, vc, keep, cap)


def test_compact_rejects_bad_indices(L):
    cap = 256
    kc = torch.randn(1, 1, cap, 16)
    tc = torch.zeros(cap, dtype=torch.int32)
    tp = torch.arange(cap, dtype=torch.int32)
    for bad in ([0, 5, 5, 9], [3, 2], [0, 1, 300], [1, 0]):
        k2, v2, _, _, st = _gpu_compact(L, kc, kc.clone(), tc, tp, np.array(bad, np.int32), 200)
        assert st[0] == L.DELTAS_ERR_DEVICE_INDEX
        assert torch.equal(k2, kc), "nothing may move when the index list is invalid"


def test_append_kv(L):
    Lf, Hkv, D, cap = 2, 2, 64, 600
    desc = L.kv_desc(Lf, Hkv, D, torch.bfloat16, cap)
    kc = torch.zeros(Lf, Hkv, cap, D, dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros_like(kc)
    tc = torch.full((cap,), -1, dtype=torch.int32, device="cuda")
    tp = torch.full((cap,), -1, dtype=torch.int32, device="cuda")
    kn, vn = inputs.kv_chunk(Lf, Hkv, 100, D, "bf16", 5)
    L.deltas_append_kv(desc, kc, vc, tc, tp, 250, kn.cuda(), vn.cuda(), 7, 12345)
    torch.cuda.synchronize()
    assert torch.equal(kc[:, :, 250:350].cpu(), kn) and torch.equal(vc[:, :, 250:350].cpu(), vn)
    assert torch.count_nonzero(kc[:, :, :250]) == 0 and torch.count_nonzero(kc[:, :, 350:]) == 0
    assert tc[250:350].eq(7).all() and tp[250:350].cpu().tolist() == list(range(12345, 12445))
    assert tc[:250].eq(-1).all() and tc[350:].eq(-1).all()
