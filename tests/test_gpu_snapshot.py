"""Question-time snapshot / restore (Sec. 3.3, "Question answering") through the C ABI.

deltas_copy_stream_state is a copy: its result must equal the source bit for bit on the copied
ranges and leave everything else of the destination alone.  Driven by the stream, a question
between snapshot() and restore() (here a chunk of other tokens, which moves the state, scores a
slot and evicts) must leave the stream exactly as a run without the question, and that run must
match the CPU oracle's Alg. 1 loop with the question undone in the same way."""
import numpy as np
import pytest
import torch

from oracle.stream import run_stream
from paper_2609_27470_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    from paper_2609_27470_gb300 import build
    build.build()
    from paper_2609_27470_gb300 import _lib
    return _lib


def _bits(t):
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)


def _rand_set(gdn, kv, dev, gen, tdt):
    shp = (gdn.num_layers, gdn.num_v_heads, gdn.value_dim, gdn.key_dim)
    s = {"state": torch.randn(shp, generator=gen).to(dev), "chunk_scores": torch.rand(37, generator=gen).to(dev)}
    if kv is not None:
        cshp = (kv.num_layers, kv.num_kv_heads, kv.capacity, kv.head_dim)
        s["k_cache"] = torch.randn(cshp, generator=gen).to(tdt).to(dev)
        s["v_cache"] = torch.randn(cshp, generator=gen).to(tdt).to(dev)
        s["tok_chunk"] = torch.randint(0, 1000, (kv.capacity,), generator=gen, dtype=torch.int32).to(dev)
        s["tok_pos"] = torch.randint(0, 1 << 20, (kv.capacity,), generator=gen, dtype=torch.int32).to(dev)
    return s


@pytest.mark.parametrize("D,dt,cache_len,n_chunks", [
    (16, "f32", 257, 7),          # ragged: row bytes not a multiple of 16 for the 4-byte arrays
    (256, "bf16", 300, 37),       # the whole cache, every score
    (256, "bf16", 0, 0),          # nothing but the state
    (128, "f32", 1, 1),
])
@pytest.mark.parametrize("full", [True, False])
def test_copy_stream_state_exact(L, D, dt, cache_len, n_chunks, full):
    dev = torch.device("cuda")
    tdt = torch.float32 if dt == "f32" else torch.bfloat16
    gen = torch.Generator().manual_seed(D + cache_len + n_chunks)
    gdn = L.gdn_desc(2, 2, 4, 128, torch.bfloat16)
    kv = L.kv_desc(3, 2, D, tdt, 300)
    src = _rand_set(gdn, kv if full else None, dev, gen, tdt)
    dst = _rand_set(gdn, kv, dev, gen, tdt)
    before = {n: t.clone() for n, t in dst.items()}
    L.deltas_copy_stream_state(gdn, kv if full else None, cache_len, n_chunks, src,
                               dst if full else {n: dst[n] for n in ("state", "chunk_scores")})
    torch.cuda.synchronize()
    assert torch.equal(dst["state"].view(torch.int32), src["state"].view(torch.int32))
    assert torch.equal(dst["chunk_scores"][:n_chunks].view(torch.int32), src["chunk_scores"][:n_chunks].view(torch.int32))
    assert torch.equal(dst["chunk_scores"][n_chunks:], before["chunk_scores"][n_chunks:])
    for n in ("k_cache", "v_cache"):
        if full:
            assert torch.equal(_bits(dst[n][:, :, :cache_len]), _bits(src[n][:, :, :cache_len]))
        else:
            assert torch.equal(_bits(dst[n][:, :, :cache_len]), _bits(before[n][:, :, :cache_len]))
        assert torch.equal(_bits(dst[n][:, :, cache_len:]), _bits(before[n][:, :, cache_len:]))
    for n in ("tok_chunk", "tok_pos"):
        ref = src[n] if full else before[n]
        assert torch.equal(dst[n][:cache_len], ref[:cache_len])
        assert torch.equal(dst[n][cache_len:], before[n][cache_len:])


def _np(t):
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.numpy()


CFG = dict(L=2, Hk=2, Hv=4, d=128, lens=[118, 132, 124, 121, 129, 119, 127, 125, 130, 118], Lf=2, Hkv=4, D=256,
           M=500, n_s=4, n_w=128, N=4)


def _make(cfg, dev, s0):
    from paper_2609_27470_gb300.stream import DeltaSStream
    return DeltaSStream(num_layers=cfg["L"], num_k_heads=cfg["Hk"], num_v_heads=cfg["Hv"], head_dim=cfg["d"],
                        act_dtype=torch.bfloat16, kv_layers=cfg["Lf"], kv_heads=cfg["Hkv"], kv_head_dim=cfg["D"],
                        kv_dtype=torch.bfloat16, budget_M=cfg["M"], n_sink=cfg["n_s"], n_window=cfg["n_w"],
                        n_buckets=cfg["N"], chunk_len=max(cfg["lens"]), max_chunks=len(cfg["lens"]) + 1,
                        state0=s0.to(dev), device=dev)


def _feed(s, x, kv, dev):
    x = {k: v.to(dev) for k, v in x.items()}
    s.step(x["q"], x["k"], x["v"], x["g"], x["beta"], kv[0].to(dev), kv[1].to(dev))


def _same_stream(a, b):
    assert (a.cache_len, a.position, a.chunk) == (b.cache_len, b.position, b.chunk)
    n = a.cache_len
    assert torch.equal(a.state.view(torch.int32), b.state.view(torch.int32))
    assert torch.equal(a.chunk_scores[: a.chunk].view(torch.int32), b.chunk_scores[: b.chunk].view(torch.int32))
    for name in ("k_cache", "v_cache"):
        assert torch.equal(_bits(getattr(a, name)[:, :, :n]), _bits(getattr(b, name)[:, :, :n]))
    for name in ("tok_chunk", "tok_pos"):
        assert torch.equal(getattr(a, name)[:n], getattr(b, name)[:n])


@pytest.mark.parametrize("at", [3, 7])
def test_question_turn_leaves_stream_unchanged(L, at):
    """Full snapshot: the question is a chunk of other tokens run through step() (state update,
    a score written at the next chunk slot, an append and, with the cache at its budget, an
    eviction), then restore().  The stream then continues; every buffer and counter must equal a
    run without the question, bit for bit, and the oracle loop with the question undone."""
    cfg = CFG
    dev = torch.device("cuda")
    lens = cfg["lens"]
    chunks = [inputs.gdn_chunk(cfg["L"], lens[c], cfg["Hk"], cfg["Hv"], cfg["d"], "bf16", inputs.seed_for(60, c))
              for c in range(len(lens))]
    kvs = [inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], lens[c], cfg["D"], "bf16", inputs.seed_for(61, c))
           for c in range(len(lens))]
    q_len = 127                     # with the cache at 374 or 500 tokens the question always evicts
    qx = inputs.gdn_chunk(cfg["L"], q_len, cfg["Hk"], cfg["Hv"], cfg["d"], "bf16", inputs.seed_for(62, at))
    qkv = inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], q_len, cfg["D"], "bf16", inputs.seed_for(63, at))
    s0 = inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 64)
    plain, asked = _make(cfg, dev, s0), _make(cfg, dev, s0)
    for c in range(len(lens)):
        _feed(plain, chunks[c], kvs[c], dev)
        if c == at:
            snap = asked.snapshot()
            ev = asked.evictions
            _feed(asked, qx, qkv, dev)
            torch.cuda.synchronize()
            assert asked.evictions == ev + 1                       # the question did evict
            assert not torch.equal(asked.state, snap.buffers["state"])
            asked.restore(snap)
        _feed(asked, chunks[c], kvs[c], dev)
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(asked.workspace) == (0, 0)
    _same_stream(asked, plain)

    f = lambda t: t.float().numpy()
    ref = run_stream(lambda c: tuple(f(chunks[c][k]) for k in ("q", "k", "v", "g", "beta")),
                     lambda c: (_np(kvs[c][0]), _np(kvs[c][1])), s0.double().numpy(), len(lens),
                     dict(budget_M=cfg["M"], n_sink=cfg["n_s"], n_window=cfg["n_w"], n_buckets=cfg["N"]),
                     capacity=asked.capacity, score_override=asked.chunk_scores[: len(lens)].cpu().numpy(),
                     questions={at: lambda: (tuple(f(qx[k]) for k in ("q", "k", "v", "g", "beta")),
                                             (_np(qkv[0]), _np(qkv[1])))})
    S = asked.state.double().cpu().numpy()
    rel = np.sqrt(((S - ref.state) ** 2).sum(axis=(2, 3)) / (ref.state ** 2).sum(axis=(2, 3)))
    assert rel.max() <= 2e-3
    np.testing.assert_allclose(asked.chunk_scores[: len(lens)].cpu().numpy(), ref.chunk_scores, rtol=1e-3)
    n = asked.cache_len
    assert n == ref.cache_len
    assert np.array_equal(asked.tok_chunk[:n].cpu().numpy(), ref.tok_chunk[:n])
    assert np.array_equal(asked.tok_pos[:n].cpu().numpy(), ref.tok_pos[:n])
    assert np.array_equal(_np(asked.k_cache[:, :, :n].cpu()), ref.k_cache[:, :, :n])


def test_light_snapshot_question_appends_only(L):
    """full=False saves the state and the scores only: a question that updates the state and
    appends to the caches without evicting is undone by restoring them and the host's cache
    length; a question that evicts cannot be (restore refuses)."""
    cfg = CFG
    dev = torch.device("cuda")
    lens = cfg["lens"][:6]
    chunks = [inputs.gdn_chunk(cfg["L"], lens[c], cfg["Hk"], cfg["Hv"], cfg["d"], "bf16", inputs.seed_for(65, c))
              for c in range(len(lens))]
    kvs = [inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], lens[c], cfg["D"], "bf16", inputs.seed_for(66, c))
           for c in range(len(lens))]
    qx = inputs.gdn_chunk(cfg["L"], 40, cfg["Hk"], cfg["Hv"], cfg["d"], "bf16", inputs.seed_for(67, 0))
    qkv = inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], 40, cfg["D"], "bf16", inputs.seed_for(68, 0))
    s0 = inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 69)
    plain, asked = _make(cfg, dev, s0), _make(cfg, dev, s0)
    for c in range(len(lens)):
        _feed(plain, chunks[c], kvs[c], dev)
        if c == 4:
            # the question's own pieces: update (writes drift partials), score at the next slot,
            # append past the cache (capacity = M + the longest chunk leaves room), no selection
            snap = asked.snapshot(full=False)
            x = {k: v.to(dev) for k, v in qx.items()}
            L.deltas_gdn_chunk_update(asked.gdn, 40, None, x["k"], x["v"], x["g"], x["beta"], asked.state, None,
                                      asked.partials, asked.workspace)
            L.deltas_score_chunks(cfg["L"], cfg["Hv"], asked.partials, asked.chunk, asked.chunk_scores)
            L.deltas_append_kv(asked.kv, asked.k_cache, asked.v_cache, asked.tok_chunk, asked.tok_pos,
                               asked.cache_len, qkv[0].to(dev), qkv[1].to(dev), asked.chunk, asked.position)
            asked.cache_len += 40
            asked.position += 40
            asked.restore(snap)
        _feed(asked, chunks[c], kvs[c], dev)
    torch.cuda.synchronize()
    _same_stream(asked, plain)
    snap = asked.snapshot(full=False)
    _feed(asked, qx, qkv, dev)                       # a step at the budget evicts
    with pytest.raises(ValueError):
        asked.restore(snap)
