"""End-to-end Alg. 1 through the C ABI on the GPU vs the CPU oracle's Alg. 1 loop.

Selection is compared given identical scores (the oracle ranks with the GPU's own float32 chunk
scores), so a near-tie in drift cannot flip an eviction; the scores themselves are compared
within the drift tolerance (1e-3 relative, +inf == +inf)."""
import numpy as np
import pytest
import torch

from oracle.stream import run_stream
from paper_2609_27470_gb300 import inputs

pytestmark = pytest.mark.gpu


def _np(t):
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.numpy()


@pytest.mark.parametrize("cfg", [
    # tiny workload, both policies: (a) pure top chunks, (b) sink + window + 2 spans
    dict(L=1, Hk=2, Hv=2, d=16, dt="f32", C=64, n_ch=8, Lf=1, Hkv=2, D=16, M=256, n_s=0, n_w=0, N=1, zero=True),
    dict(L=1, Hk=2, Hv=2, d=16, dt="f32", C=64, n_ch=8, Lf=1, Hkv=2, D=16, M=256, n_s=4, n_w=64, N=2, zero=True),
    # wider heads, bf16, ragged chunk length, paper-like policy
    dict(L=2, Hk=2, Hv=4, d=128, dt="bf16", C=120, n_ch=12, Lf=2, Hkv=2, D=256, M=600, n_s=4, n_w=128, N=4,
         zero=False),
    # the paper's stream shape: chunk lengths varying over 118-132 tokens, 4 KV heads, sink, window
    # and spans (Sec. 4.1), budget a few chunks so that most chunks evict
    dict(L=2, Hk=2, Hv=4, d=128, dt="bf16", Cs=[118, 132, 124, 121, 129, 119, 127, 125, 130, 118, 126, 131, 122, 128],
         Lf=2, Hkv=4, D=256, M=500, n_s=4, n_w=128, N=4, zero=False),
    # the same stream scored by the comparison signal of Sec. 4.3 (write sizes) instead of drift
    dict(L=2, Hk=2, Hv=4, d=128, dt="bf16", Cs=[118, 132, 124, 121, 129, 119, 127, 125, 130, 118, 126, 131, 122, 128],
         Lf=2, Hkv=4, D=256, M=500, n_s=4, n_w=128, N=4, zero=False, signal="write_norm"),
    dict(L=1, Hk=2, Hv=2, d=16, dt="f32", C=64, n_ch=8, Lf=1, Hkv=2, D=16, M=256, n_s=4, n_w=64, N=2, zero=True,
         signal="write_norm"),
])
def test_stream_matches_oracle(cfg):
    from paper_2609_27470_gb300.stream import DeltaSStream
    dev = torch.device("cuda")
    tdt = torch.float32 if cfg["dt"] == "f32" else torch.bfloat16
    lens = cfg["Cs"] if "Cs" in cfg else [cfg["C"]] * cfg["n_ch"]
    cfg = dict(cfg, n_ch=len(lens), C=max(lens))
    chunks = [inputs.gdn_chunk(cfg["L"], lens[c], cfg["Hk"], cfg["Hv"], cfg["d"], cfg["dt"], inputs.seed_for(3, c))
              for c in range(cfg["n_ch"])]
    kvs = [inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], lens[c], cfg["D"], cfg["dt"], inputs.seed_for(4, c))
           for c in range(cfg["n_ch"])]
    s0 = (torch.zeros(cfg["L"], cfg["Hv"], cfg["d"], cfg["d"]) if cfg["zero"]
          else inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 5))
    s = DeltaSStream(num_layers=cfg["L"], num_k_heads=cfg["Hk"], num_v_heads=cfg["Hv"], head_dim=cfg["d"],
                     act_dtype=tdt, kv_layers=cfg["Lf"], kv_heads=cfg["Hkv"], kv_head_dim=cfg["D"], kv_dtype=tdt,
                     budget_M=cfg["M"], n_sink=cfg["n_s"], n_window=cfg["n_w"], n_buckets=cfg["N"],
                     chunk_len=cfg["C"], max_chunks=cfg["n_ch"], state0=s0.to(dev), device=dev,
                     signal=cfg.get("signal", "drift"))
    for c in range(cfg["n_ch"]):
        x = {k: v.to(dev) for k, v in chunks[c].items()}
        s.step(x["q"], x["k"], x["v"], x["g"], x["beta"], kvs[c][0].to(dev), kvs[c][1].to(dev))
    torch.cuda.synchronize()
    from paper_2609_27470_gb300 import _lib as L
    assert L.deltas_get_device_status(s.workspace) == (0, 0)
    gpu_scores = s.chunk_scores.cpu().numpy()
    f = lambda t: t.float().numpy()
    ref = run_stream(lambda c: tuple(f(chunks[c][k]) for k in ("q", "k", "v", "g", "beta")),
                     lambda c: (_np(kvs[c][0]), _np(kvs[c][1])), s0.double().numpy(), cfg["n_ch"],
                     dict(budget_M=cfg["M"], n_sink=cfg["n_s"], n_window=cfg["n_w"], n_buckets=cfg["N"]),
                     capacity=s.capacity, score_override=gpu_scores, signal=cfg.get("signal", "drift"))
    fin = np.isfinite(ref.chunk_scores)
    assert np.array_equal(np.isfinite(gpu_scores), fin)
    np.testing.assert_allclose(gpu_scores[fin], ref.chunk_scores[fin], rtol=1e-3)
    st = s.state.cpu().double().numpy()
    rel = np.sqrt(((st - ref.state) ** 2).sum(axis=(2, 3)) / (ref.state ** 2).sum(axis=(2, 3)))
    assert rel.max() <= 2e-3
    n = s.cache_len
    assert n == ref.cache_len and s.evictions == len(ref.evictions)
    assert np.array_equal(_np(s.k_cache[:, :, :n].cpu()), ref.k_cache[:, :, :n])
    assert np.array_equal(_np(s.v_cache[:, :, :n].cpu()), ref.v_cache[:, :, :n])
    assert np.array_equal(s.tok_chunk[:n].cpu().numpy(), ref.tok_chunk[:n])
    assert np.array_equal(s.tok_pos[:n].cpu().numpy(), ref.tok_pos[:n])


def test_stream_read_out_paper_shape():
    """Alg. 1 Prefill with the layer output: the paper's chunk lengths (118-132 tokens, every
    chunk a ragged tail, blocks of 128 read-out tokens cut at different places) through a stream
    built with read_out=True (d = 128 bf16: the tensor-core update and read-out kernels), with
    evictions running in between; every chunk's outputs against the oracle replayed from the
    stream's own state before the chunk, and a stream without read_out refuses an output buffer."""
    import oracle
    from paper_2609_27470_gb300.stream import DeltaSStream
    dev = torch.device("cuda")
    Lg, Hk, Hv, d = 2, 2, 4, 128
    lens = [118, 132, 124, 121, 129, 119, 127, 125]
    qs = 128 ** -0.5
    mk = lambda ro: DeltaSStream(num_layers=Lg, num_k_heads=Hk, num_v_heads=Hv, head_dim=d, act_dtype=torch.bfloat16,
                                 kv_layers=1, kv_heads=2, kv_head_dim=128, kv_dtype=torch.bfloat16, budget_M=300,
                                 n_sink=4, n_window=64, n_buckets=2, chunk_len=max(lens), max_chunks=len(lens),
                                 state0=inputs.initial_state(Lg, Hv, d, 7).to(dev), device=dev, q_scale=qs,
                                 read_out=ro)
    s = mk(True)
    f64 = lambda t: t.float().cpu().double().numpy()       # noqa: E731
    for c, T in enumerate(lens):
        x = {k: v.to(dev) for k, v in inputs.gdn_chunk(Lg, T, Hk, Hv, d, "bf16", inputs.seed_for(8, c)).items()}
        kn, vn = inputs.kv_chunk(1, 2, T, 128, "bf16", inputs.seed_for(9, c))
        s_before = s.state.clone()
        out = torch.empty(Lg, T, Hv, d, dtype=torch.bfloat16, device=dev)
        s.step(x["q"], x["k"], x["v"], x["g"], x["beta"], kn.to(dev), vn.to(dev), out=out)
        torch.cuda.synchronize()
        _, o_ref = oracle.gdn_recurrence(f64(x["q"]), f64(x["k"]), f64(x["v"]), f64(x["g"]), f64(x["beta"]),
                                         f64(s_before), q_scale=qs, want_out=True)
        o = f64(out)
        rel = np.sqrt(((o - o_ref) ** 2).sum(axis=(1, 3)) / (o_ref ** 2).sum(axis=(1, 3)))
        assert rel.max() <= 2e-3 + 2.0 ** -8, (c, rel.max())
    from paper_2609_27470_gb300 import _lib as L
    assert L.deltas_get_device_status(s.workspace) == (0, 0) and s.evictions > 0
    plain = mk(False)
    x = {k: v.to(dev) for k, v in inputs.gdn_chunk(Lg, lens[0], Hk, Hv, d, "bf16", 1).items()}
    kn, vn = inputs.kv_chunk(1, 2, lens[0], 128, "bf16", 2)
    with pytest.raises(ValueError):
        plain.step(x["q"], x["k"], x["v"], x["g"], x["beta"], kn.to(dev), vn.to(dev),
                   out=torch.empty(Lg, lens[0], Hv, d, dtype=torch.bfloat16, device=dev))
