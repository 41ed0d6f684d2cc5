"""Per-head token signals (Sec. 4.3: key norm -||k||, value norm ||v||, ranked per KV head under the
Sec. 3.3 policy) through the C ABI on the GPU, against the CPU oracle.

Scores are float32 sums of squares on the GPU and fp64 in the oracle, so they are compared within a
relative 2e-6 (a float32 sum of 256 exact squares, a warp tree and a rounded square root stay well
inside it).  Selection and compaction are index and byte work: they must match the oracle exactly,
given identical scores (the oracle ranks with the GPU's float32 scores)."""
import numpy as np
import pytest
import torch

import oracle
from oracle.stream import run_stream_heads
from paper_2609_27470_gb300 import inputs

pytestmark = pytest.mark.gpu

SCORE_RTOL = 2e-6


@pytest.fixture(scope="module")
def L():
    from paper_2609_27470_gb300 import build
    build.build()
    from paper_2609_27470_gb300 import _lib
    return _lib


def _bits(t):
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)


def _np(t):
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.numpy()


@pytest.mark.parametrize("signal", ["key_norm", "value_norm"])
@pytest.mark.parametrize("D,dt,cache_len,n_new", [
    (256, "bf16", 1000, 512),
    (256, "bf16", 0, 131),        # first chunk, ragged length
    (16, "f32", 37, 64),
    (128, "bf16", 5, 1),
])
def test_append_heads_copies_rows_and_scores_them(L, signal, D, dt, cache_len, n_new):
    dev = torch.device("cuda")
    tdt = torch.float32 if dt == "f32" else torch.bfloat16
    Lf, Hkv, cap = 2, 3, cache_len + n_new + 7
    kv = L.kv_desc(Lf, Hkv, D, tdt, cap)
    gen = torch.Generator().manual_seed(D + cache_len + n_new)
    kc = torch.randn(Lf, Hkv, cap, D, generator=gen).to(tdt)
    vc = torch.randn(Lf, Hkv, cap, D, generator=gen).to(tdt)
    meta = [torch.randint(0, 99, (Lf, Hkv, cap), generator=gen, dtype=torch.int32) for _ in range(2)]
    ts = torch.randn(Lf, Hkv, cap, generator=gen)
    kn = torch.randn(Lf, Hkv, n_new, D, generator=gen).to(tdt)
    vn = 3.0 * torch.randn(Lf, Hkv, n_new, D, generator=gen).to(tdt)
    kn[0, 1, 0] = 0                                      # a zero row scores (-)0
    d = [t.to(dev) for t in (kc, vc, meta[0], meta[1], ts)]
    L.deltas_append_kv_heads(kv, signal, d[0], d[1], d[2], d[3], d[4], cache_len, kn.to(dev), vn.to(dev), 41, 9000)
    torch.cuda.synchronize()
    kc2, vc2, tc2, tp2, ts2 = (t.cpu() for t in d)
    sl = slice(cache_len, cache_len + n_new)
    assert torch.equal(_bits(kc2[:, :, sl]), _bits(kn)) and torch.equal(_bits(vc2[:, :, sl]), _bits(vn))
    for new, old in ((kc2, kc), (vc2, vc), (tc2, meta[0]), (tp2, meta[1]), (ts2, ts)):
        assert torch.equal(_bits(new[:, :, :cache_len]), _bits(old[:, :, :cache_len]))
        assert torch.equal(_bits(new[:, :, cache_len + n_new:]), _bits(old[:, :, cache_len + n_new:]))
    assert torch.all(tc2[:, :, sl] == 41)
    assert torch.equal(tp2[:, :, sl], (9000 + torch.arange(n_new, dtype=torch.int32)).expand(Lf, Hkv, n_new))
    rows = (kn if signal == "key_norm" else vn).float().numpy()
    ref = oracle.row_norm_scores(rows, signal)
    np.testing.assert_allclose(ts2[:, :, sl].numpy(), ref, rtol=SCORE_RTOL, atol=0)
    if signal == "key_norm":
        assert ts2[0, 1, cache_len].item() == 0.0


def _plane_inputs(rng, planes, T, n_chunks, stride):
    """Per-plane chunk ids (ascending, with the gaps repeated evictions leave) and scores with
    exact ties, signed zeros and infinities."""
    tc = np.zeros((planes, stride), np.int32)
    ts = np.zeros((planes, stride), np.float32)
    for p in range(planes):
        tc[p, :T] = np.sort(rng.integers(0, n_chunks, size=T))
        s = np.round(rng.standard_normal(T), 2).astype(np.float32)       # ties
        if T > 20:
            idx = rng.choice(T, size=8, replace=False)
            s[idx[:2]] = -0.0
            s[idx[2:4]] = 0.0
            s[idx[4]] = np.inf
            s[idx[5]] = -np.inf
        ts[p, :T] = s
    return tc, ts


SELECT_CASES = [
    # planes, T, M, n_s, n_w, N
    (4, 1000, 600, 4, 128, 4),
    (3, 777, 700, 0, 0, 1),
    (2, 3000, 2500, 2, 10, 32),
    (2, 300, 40, 4, 30, 8),            # quota 0: everything comes from the fill
    (3, 500, 600, 4, 128, 4),          # no eviction: the identity
    (5, 2049, 1024, 4, 1000, 0),       # N = 0 read as one span
    (16, 33280, 32768, 4, 1024, 4),    # streaming shape: keys in shared memory
    (16, 65536, 16384, 4, 1024, 4),    # 64k slots: a quarter per CTA, keys in shared memory
    (2, 180000, 60000, 4, 1024, 4),    # 180k slots: keys in the workspace
    (3, 9, 5, 1, 1, 2),                # fewer candidates than the cluster has CTAs per plane
    (48, 2000, 1500, 4, 128, 4),       # more planes than clusters resident at once
]


@pytest.mark.parametrize("planes,T,M,n_s,n_w,N", SELECT_CASES)
@pytest.mark.parametrize("with_mask", [True, False])
def test_select_heads_matches_oracle(L, planes, T, M, n_s, n_w, N, with_mask):
    dev = torch.device("cuda")
    rng = np.random.default_rng(T + M + N)
    stride = T + 13
    tc, ts = _plane_inputs(rng, planes, T, max(4, T // 50), stride)
    pol = L.policy(M, n_s, n_w, N)
    ws = L.alloc_workspace(L.deltas_select_retain_heads_workspace_size(planes, T), dev)
    ri = torch.full((planes, M), -1, dtype=torch.int32, device=dev)
    nr = torch.zeros(1, dtype=torch.int32, device=dev)
    mk = torch.full((planes, stride), 7, dtype=torch.uint8, device=dev) if with_mask else None
    L.deltas_select_retain_heads(pol, T, torch.from_numpy(tc).to(dev), torch.from_numpy(ts).to(dev), ri, nr, mk, ws)
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(ws) == (0, 0)
    n = min(T, M)
    assert nr.item() == n
    ri = ri.cpu().numpy()
    for p in range(planes):
        idx, mask = oracle.select_retain_tokens(M, n_s, n_w, N, tc[p, :T], ts[p, :T])
        assert np.array_equal(ri[p, :n], idx), p
        assert np.all(ri[p, n:] == -1)
        if with_mask:
            m = mk[p].cpu().numpy()
            assert np.array_equal(m[:T], mask) and np.all(m[T:] == 7)


@pytest.mark.parametrize("slot,n_s,n_w", [(50, 0, 0), (1, 4, 10), (97, 4, 10)])
def test_select_heads_reports_negative_chunk_ids(L, slot, n_s, n_w):
    """A negative chunk id among the candidates, in the sink or in the window of plane 1 (each
    checked by a different CTA of the plane's cluster) is reported; the call then recovers."""
    dev = torch.device("cuda")
    tc = torch.zeros(2, 100, dtype=torch.int32)
    tc[1, slot] = -3
    ts = torch.randn(2, 100)
    ws = L.alloc_workspace(L.deltas_select_retain_heads_workspace_size(2, 100), dev)
    L.deltas_clear_device_status(ws)
    ri = torch.zeros(2, 60, dtype=torch.int32, device=dev)
    nr = torch.zeros(1, dtype=torch.int32, device=dev)
    L.deltas_select_retain_heads(L.policy(60, n_s, n_w, 1), 100, tc.to(dev), ts.to(dev), ri, nr, None, ws)
    assert L.deltas_get_device_status(ws)[0] == L.DELTAS_ERR_DEVICE_INDEX
    L.deltas_clear_device_status(ws)
    tc[1, slot] = 0
    L.deltas_select_retain_heads(L.policy(60, n_s, n_w, 1), 100, tc.to(dev), ts.to(dev), ri, nr, None, ws)
    assert L.deltas_get_device_status(ws) == (0, 0) and nr.item() == 60


@pytest.mark.parametrize("D,dt,T,M", [
    (256, "bf16", 33280, 32768),
    (256, "bf16", 5000, 1111),
    (16, "f32", 777, 500),
    (64, "bf16", 130, 129),
])
def test_compact_heads_matches_oracle(L, D, dt, T, M):
    dev = torch.device("cuda")
    tdt = torch.float32 if dt == "f32" else torch.bfloat16
    Lf, Hkv, cap = 2, 3, T + 9
    P = Lf * Hkv
    rng = np.random.default_rng(T + D)
    lists = []
    for p in range(P):
        if p == 0:
            lists.append(np.arange(M, dtype=np.int32))                         # nothing moves
        elif p == 1:
            lists.append(np.r_[np.arange(M - 1), T - 1].astype(np.int32))      # only the last row moves
        else:
            lists.append(np.sort(rng.choice(T, size=M, replace=False)).astype(np.int32))
    kv = L.kv_desc(Lf, Hkv, D, tdt, cap)
    gen = torch.Generator().manual_seed(T)
    kc = torch.randn(Lf, Hkv, cap, D, generator=gen).to(tdt)
    vc = torch.randn(Lf, Hkv, cap, D, generator=gen).to(tdt)
    tc = torch.randint(0, 1 << 20, (Lf, Hkv, cap), generator=gen, dtype=torch.int32)
    tp = torch.randint(0, 1 << 20, (Lf, Hkv, cap), generator=gen, dtype=torch.int32)
    ts = torch.randn(Lf, Hkv, cap, generator=gen)
    ref = oracle.compact_kv_heads(_np(kc), _np(vc), tc.numpy(), tp.numpy(), ts.numpy(), lists, T)
    d = [t.to(dev) for t in (kc, vc, tc, tp, ts)]
    ri = torch.from_numpy(np.stack(lists)).to(dev)
    nr = torch.tensor([M], dtype=torch.int32, device=dev)
    ws = L.alloc_workspace(L.deltas_compact_kv_heads_workspace_size(kv, T), dev)
    L.deltas_compact_kv_heads(kv, d[0], d[1], d[2], d[3], d[4], ri, nr, T, ws)
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(ws) == (0, 0)
    for got, want in zip(d, ref):
        g = got.cpu()
        g = _np(g) if g.dtype == torch.bfloat16 else g.numpy()
        assert np.array_equal(g.view(np.int32) if g.dtype == np.float32 else g,
                              want.view(np.int32) if want.dtype == np.float32 else want)


def test_compact_heads_rejects_a_bad_list(L):
    dev = torch.device("cuda")
    kv = L.kv_desc(1, 2, 64, torch.bfloat16, 100)
    kc = torch.randn(1, 2, 100, 64, device=dev).to(torch.bfloat16)
    before = kc.clone()
    tc = torch.zeros(1, 2, 100, dtype=torch.int32, device=dev)
    ri = torch.tensor([[0, 5, 9], [0, 7, 3]], dtype=torch.int32, device=dev)   # plane 1 not ascending
    nr = torch.tensor([3], dtype=torch.int32, device=dev)
    ws = L.alloc_workspace(L.deltas_compact_kv_heads_workspace_size(kv, 50), dev)
    L.deltas_clear_device_status(ws)
    L.deltas_compact_kv_heads(kv, kc, kc.clone(), tc, tc.clone(), torch.zeros(1, 2, 100, device=dev), ri, nr, 50, ws)
    assert L.deltas_get_device_status(ws)[0] == L.DELTAS_ERR_DEVICE_INDEX
    assert torch.equal(_bits(kc), _bits(before))


STREAM_CFG = dict(L=2, Hk=2, Hv=4, d=128, Lf=2, Hkv=2, D=256, M=600, n_s=4, n_w=128, N=4,
                  lens=[118, 132, 124, 121, 129, 119, 127, 125, 130, 118, 126, 131])


@pytest.mark.parametrize("signal", ["key_norm", "value_norm"])
def test_stream_heads_matches_oracle(L, signal):
    """The stream driver with a per-head signal vs the oracle's per-head loop, given the GPU's own
    token scores; the scores themselves against the oracle's; the recurrent state still moves."""
    from paper_2609_27470_gb300.stream import DeltaSStream
    cfg = STREAM_CFG
    dev = torch.device("cuda")
    lens = cfg["lens"]
    chunks = [inputs.gdn_chunk(cfg["L"], lens[c], cfg["Hk"], cfg["Hv"], cfg["d"], "bf16", inputs.seed_for(81, c))
              for c in range(len(lens))]
    kvs = [inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], lens[c], cfg["D"], "bf16", inputs.seed_for(82, c))
           for c in range(len(lens))]
    s0 = inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 83)
    s = DeltaSStream(num_layers=cfg["L"], num_k_heads=cfg["Hk"], num_v_heads=cfg["Hv"], head_dim=cfg["d"],
                     act_dtype=torch.bfloat16, kv_layers=cfg["Lf"], kv_heads=cfg["Hkv"], kv_head_dim=cfg["D"],
                     kv_dtype=torch.bfloat16, budget_M=cfg["M"], n_sink=cfg["n_s"], n_window=cfg["n_w"],
                     n_buckets=cfg["N"], chunk_len=max(lens), max_chunks=len(lens), state0=s0.to(dev), device=dev,
                     signal=signal)
    state_before = s.state.clone()
    for c in range(len(lens)):
        x = {k: v.to(dev) for k, v in chunks[c].items()}
        s.step(x["q"], x["k"], x["v"], x["g"], x["beta"], kvs[c][0].to(dev), kvs[c][1].to(dev))
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(s.workspace) == (0, 0)
    assert not torch.equal(s.state, state_before)
    assert s.evictions > 0

    # the GPU's score of every chunk's tokens: the same append into a scratch cache
    kvd = L.kv_desc(cfg["Lf"], cfg["Hkv"], cfg["D"], torch.bfloat16, max(lens))
    shp = (cfg["Lf"], cfg["Hkv"], max(lens))
    scratch = [torch.zeros(*shp, cfg["D"], dtype=torch.bfloat16, device=dev) for _ in range(2)]
    meta = [torch.zeros(shp, dtype=torch.int32, device=dev) for _ in range(2)]
    gpu_scores = []
    for c in range(len(lens)):
        sc = torch.zeros(shp, device=dev)
        L.deltas_append_kv_heads(kvd, signal, scratch[0], scratch[1], meta[0], meta[1], sc, 0,
                                 kvs[c][0].to(dev), kvs[c][1].to(dev), c, 0)
        gpu_scores.append(sc[:, :, : lens[c]].cpu().numpy())
    policy = dict(budget_M=cfg["M"], n_sink=cfg["n_s"], n_window=cfg["n_w"], n_buckets=cfg["N"])
    ref = run_stream_heads(lambda c: (_np(kvs[c][0]), _np(kvs[c][1])), len(lens), policy, s.capacity, signal,
                           score_override=lambda c: gpu_scores[c])
    own = run_stream_heads(lambda c: (_np(kvs[c][0]), _np(kvs[c][1])), 1, dict(policy, budget_M=10 ** 6),
                           max(lens), signal)
    np.testing.assert_allclose(gpu_scores[0], own.tok_score[:, :, : lens[0]], rtol=SCORE_RTOL, atol=0)
    n = s.cache_len
    assert n == ref.cache_len and s.evictions == len(ref.evictions)
    assert np.array_equal(_np(s.k_cache.cpu())[:, :, :n], ref.k_cache[:, :, :n])
    assert np.array_equal(_np(s.v_cache.cpu())[:, :, :n], ref.v_cache[:, :, :n])
    for name in ("tok_chunk", "tok_pos"):
        assert np.array_equal(getattr(s, name).cpu().numpy()[:, :, :n], getattr(ref, name)[:, :, :n]), name
    assert np.array_equal(s.tok_score.cpu().numpy()[:, :, :n].view(np.int32), ref.tok_score[:, :, :n].view(np.int32))
    # heads really differ in what they keep
    tp = s.tok_pos.cpu().numpy()
    assert not np.array_equal(tp[0, 0, :n], tp[0, 1, :n])


def test_copy_stream_state_heads_is_exact(L):
    """deltas_copy_stream_state_heads: every plane's first cache_len metadata entries and token
    scores, the cache rows and the state are copied bit for bit; nothing past cache_len moves."""
    dev = torch.device("cuda")
    gdn = L.gdn_desc(2, 2, 4, 128, torch.bfloat16)
    kv = L.kv_desc(2, 3, 256, torch.bfloat16, 1004)
    gen = torch.Generator().manual_seed(91)

    def rand_set():
        shp = (2, 3, 1004)
        return {"state": torch.randn(2, 4, 128, 128, generator=gen).to(dev),
                "chunk_scores": torch.rand(40, generator=gen).to(dev),
                "k_cache": torch.randn(*shp, 256, generator=gen).to(torch.bfloat16).to(dev),
                "v_cache": torch.randn(*shp, 256, generator=gen).to(torch.bfloat16).to(dev),
                "tok_chunk": torch.randint(0, 999, shp, generator=gen, dtype=torch.int32).to(dev),
                "tok_pos": torch.randint(0, 1 << 20, shp, generator=gen, dtype=torch.int32).to(dev),
                "tok_score": torch.randn(shp, generator=gen).to(dev)}
    src, dst = rand_set(), rand_set()
    before = {n: t.clone() for n, t in dst.items()}
    n = 777
    L.deltas_copy_stream_state(gdn, kv, n, 40, src, dst, per_head=True)
    torch.cuda.synchronize()
    assert torch.equal(dst["state"].view(torch.int32), src["state"].view(torch.int32))
    for name in ("k_cache", "v_cache", "tok_chunk", "tok_pos", "tok_score"):
        assert torch.equal(_bits(dst[name][:, :, :n]), _bits(src[name][:, :, :n])), name
        assert torch.equal(_bits(dst[name][:, :, n:]), _bits(before[name][:, :, n:])), name


@pytest.mark.parametrize("signal", ["key_norm", "value_norm"])
def test_question_turn_in_a_head_stream_leaves_it_unchanged(L, signal):
    """Sec. 3.3 question handling with a per-head signal: snapshot, a question chunk that updates
    the state and evicts per plane, restore; the stream then equals a run without the question."""
    from paper_2609_27470_gb300.stream import DeltaSStream
    cfg = STREAM_CFG
    dev = torch.device("cuda")
    lens = cfg["lens"]
    chunks = [inputs.gdn_chunk(cfg["L"], lens[c], cfg["Hk"], cfg["Hv"], cfg["d"], "bf16", inputs.seed_for(85, c))
              for c in range(len(lens))]
    kvs = [inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], lens[c], cfg["D"], "bf16", inputs.seed_for(86, c))
           for c in range(len(lens))]
    qx = inputs.gdn_chunk(cfg["L"], 127, cfg["Hk"], cfg["Hv"], cfg["d"], "bf16", inputs.seed_for(87, 0))
    qkv = inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], 127, cfg["D"], "bf16", inputs.seed_for(88, 0))
    s0 = inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 89)

    def make():
        return DeltaSStream(num_layers=cfg["L"], num_k_heads=cfg["Hk"], num_v_heads=cfg["Hv"], head_dim=cfg["d"],
                            act_dtype=torch.bfloat16, kv_layers=cfg["Lf"], kv_heads=cfg["Hkv"], kv_head_dim=cfg["D"],
                            kv_dtype=torch.bfloat16, budget_M=cfg["M"], n_sink=cfg["n_s"], n_window=cfg["n_w"],
                            n_buckets=cfg["N"], chunk_len=max(lens), max_chunks=len(lens) + 1, state0=s0.to(dev),
                            device=dev, signal=signal)

    def feed(s, x, kv):
        x = {k: v.to(dev) for k, v in x.items()}
        s.step(x["q"], x["k"], x["v"], x["g"], x["beta"], kv[0].to(dev), kv[1].to(dev))
    plain, asked = make(), make()
    for c in range(len(lens)):
        feed(plain, chunks[c], kvs[c])
        if c == 7:
            snap = asked.snapshot()
            ev = asked.evictions
            feed(asked, qx, qkv)
            torch.cuda.synchronize()
            assert asked.evictions == ev + 1
            asked.restore(snap)
        feed(asked, chunks[c], kvs[c])
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(asked.workspace) == (0, 0)
    assert (asked.cache_len, asked.position, asked.chunk, asked.evictions) == \
        (plain.cache_len, plain.position, plain.chunk, plain.evictions)
    n = asked.cache_len
    assert torch.equal(asked.state.view(torch.int32), plain.state.view(torch.int32))
    for name in ("k_cache", "v_cache", "tok_chunk", "tok_pos", "tok_score"):
        assert torch.equal(_bits(getattr(asked, name)[:, :, :n]), _bits(getattr(plain, name)[:, :, :n])), name


@pytest.mark.parametrize("signal", ["value_norm", "key_norm"])
def test_paper_stream_per_head_full_size(L, signal):
    """The paper-shaped stream ranked per KV head at full size, driven through the C ABI as the
    benchmark drives it (8 full-attention layers x 4 KV heads x D = 256 bf16, chunks of 118-132
    tokens cycling, budget 8192, sink 4, window 1024, 4 spans): filled past the budget, then every
    chunk evicts.  Every eviction's 32 retain lists are checked bit for bit against the oracle's
    selection on the chunk ids and scores read back right before it; after the last chunk every
    plane keeps its sinks and window in stream order, sampled kept rows equal the rows they were
    appended from, and every kept token's stored score is its signal recomputed from its row."""
    from paper_2609_27470_gb300 import configs
    from paper_2609_27470_gb300.stream import DeltaSStream
    cfg = configs.PAPER
    dev = torch.device("cuda")
    Lf, Hkv, D, M = cfg["Lf"], cfg["Hkv"], cfg["D"], cfg["budget_M"]
    n_s, n_w, N = cfg["n_sink"], cfg["n_window"], cfg["n_buckets"]
    lens = [cfg["chunk_lens"][c % len(cfg["chunk_lens"])] for c in range(80)]       # about 66 fill, 14 evict
    P = Lf * Hkv
    s = DeltaSStream(num_layers=1, num_k_heads=1, num_v_heads=2, head_dim=128, act_dtype=torch.bfloat16,
                     kv_layers=Lf, kv_heads=Hkv, kv_head_dim=D, kv_dtype=torch.bfloat16, budget_M=M, n_sink=n_s,
                     n_window=n_w, n_buckets=N, chunk_len=max(lens), max_chunks=len(lens), device=dev,
                     signal=signal)
    kvs = [inputs.kv_chunk(Lf, Hkv, lens[c], D, "bf16", inputs.seed_for(95, c), device=dev) for c in range(len(lens))]
    T, pos, evictions = 0, 0, 0
    for c in range(len(lens)):
        L.deltas_append_kv_heads(s.kv, signal, s.k_cache, s.v_cache, s.tok_chunk, s.tok_pos, s.tok_score, T,
                                 kvs[c][0], kvs[c][1], c, pos)
        T += lens[c]
        pos += lens[c]
        if T <= M:
            continue
        L.deltas_select_retain_heads(s.policy, T, s.tok_chunk.view(P, -1), s.tok_score.view(P, -1), s.retain_idx,
                                     s.n_retained, None, s.workspace)
        torch.cuda.synchronize()
        tc_in = s.tok_chunk.view(P, -1)[:, :T].cpu().numpy()
        ts_in = s.tok_score.view(P, -1)[:, :T].cpu().numpy()
        ri = s.retain_idx.cpu().numpy()
        assert s.n_retained.item() == M
        for p in range(P):
            idx, _ = oracle.select_retain_tokens(M, n_s, n_w, N, tc_in[p], ts_in[p])
            assert np.array_equal(ri[p], idx), (c, p)
        L.deltas_compact_kv_heads(s.kv, s.k_cache, s.v_cache, s.tok_chunk, s.tok_pos, s.tok_score, s.retain_idx,
                                  s.n_retained, T, s.workspace)
        T = M
        evictions += 1
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(s.workspace) == (0, 0)
    assert evictions >= 10
    n = T
    tc = s.tok_chunk.view(P, -1)[:, :n].cpu().numpy()
    tp = s.tok_pos.view(P, -1)[:, :n].cpu().numpy()
    ts = s.tok_score.view(P, -1)[:, :n].cpu().numpy()
    kc = s.k_cache.view(P, -1, D)[:, :n].cpu().view(torch.int16).numpy()
    vc = s.v_cache.view(P, -1, D)[:, :n].cpu().view(torch.int16).numpy()
    starts = np.cumsum([0] + lens)
    for p in range(P):
        assert np.all(np.diff(tp[p]) > 0) and tp[p][:n_s].tolist() == list(range(n_s))
        assert tp[p][-n_w:].tolist() == list(range(starts[-1] - n_w, starts[-1]))
        assert np.array_equal(tc[p], np.searchsorted(starts, tp[p], side="right") - 1)
    rng = np.random.default_rng(97)
    for p in [0, P - 1] + [int(x) for x in rng.integers(0, P, size=2)]:
        l, h = divmod(p, Hkv)
        for j in rng.integers(0, n, size=64):
            c = int(tc[p, j])
            r = int(tp[p, j] - starts[c])
            assert np.array_equal(kc[p, j], kvs[c][0][l, h, r].cpu().view(torch.int16).numpy())
            assert np.array_equal(vc[p, j], kvs[c][1][l, h, r].cpu().view(torch.int16).numpy())
        src = (kc if signal == "key_norm" else vc)[p]
        ref = oracle.row_norm_scores((src.astype(np.int32) << 16).view(np.float32), signal)
        np.testing.assert_allclose(ts[p], ref, rtol=SCORE_RTOL, atol=0)
