"""The streaming workload at full size (24 gated-delta layers x 32 value heads x 128 x 128 state,
512-token chunks, 8 full-attention layers x 2 KV heads x D = 256, budget 32,768 with sink 4,
window 1024 and 4 spans), driven through the C ABI exactly as the benchmark drives it: the cache is
filled to the budget, then every chunk evicts.  Checked against the CPU oracle where the oracle
can follow (Alg. 1, Sec. 3.2-3.3):

* the recurrent state of sampled (layer, head) pairs over the whole stream (oracle token loop);
* the drift partials of sampled heads for the last chunk, replayed from the GPU's own S_before;
* every eviction's retain list, bit-exact against the oracle's selection given the GPU's scores
  and the cache's chunk ids, and the compacted chunk ids / positions;
* sampled rows of the final K / V caches against the keys and values they were appended from
  (a property of in-place compaction that holds at any size).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_27470_gb300 import configs, inputs

pytestmark = pytest.mark.gpu

STATE_TOL = 2e-3


def _f64(t):
    return t.detach().float().cpu().double().numpy()


def test_streaming_full_size_against_oracle():
    from paper_2609_27470_gb300 import _lib as L
    from paper_2609_27470_gb300.stream import DeltaSStream
    cfg = configs.STREAMING
    dev = torch.device("cuda")
    Lg, Hk, Hv, d, C = cfg["L"], cfg["Hk"], cfg["Hv"], cfg["d"], cfg["chunk_len"]
    Lf, Hkv, D, M = cfg["Lf"], cfg["Hkv"], cfg["D"], cfg["budget_M"]
    n_s, n_w, N = cfg["n_sink"], cfg["n_window"], cfg["n_buckets"]
    n_fill = M // C
    n_chunks = n_fill + 6                                     # six eviction events
    gdn = lambda c: inputs.gdn_chunk(Lg, C, Hk, Hv, d, "bf16", inputs.seed_for(60, c), device=dev)
    kvn = lambda c: inputs.kv_chunk(Lf, Hkv, C, D, "bf16", inputs.seed_for(61, c), device=dev)
    state0 = inputs.initial_state(Lg, Hv, d, 62, device=dev)
    s = DeltaSStream(num_layers=Lg, num_k_heads=Hk, num_v_heads=Hv, head_dim=d, act_dtype=torch.bfloat16,
                     kv_layers=Lf, kv_heads=Hkv, kv_head_dim=D, kv_dtype=torch.bfloat16, budget_M=M,
                     n_sink=n_s, n_window=n_w, n_buckets=N, chunk_len=C, max_chunks=n_chunks,
                     state0=state0, device=dev)
    rng = np.random.default_rng(63)
    heads = [(0, 0), (Lg - 1, Hv - 1), (int(rng.integers(Lg)), int(rng.integers(Hv)))]
    ref_states = {lh: _f64(state0[lh[0], lh[1]])[None, None] for lh in heads}
    s_before_last = None
    n_evictions = 0
    for c in range(n_chunks):
        x = gdn(c)
        k_new, v_new = kvn(c)
        if c == n_chunks - 1:
            s_before_last = s.state.clone()
        prev_ids = s.tok_chunk[: s.cache_len].clone()
        s.step(None, x["k"], x["v"], x["g"], x["beta"], k_new, v_new)
        torch.cuda.synchronize()
        # oracle recurrence of the sampled heads over this chunk
        for (l, h) in heads:
            kh = h * Hk // Hv
            ref_states[(l, h)], _ = oracle.gdn_recurrence(
                None, _f64(x["k"][l:l + 1, :, kh:kh + 1]), _f64(x["v"][l:l + 1, :, h:h + 1]),
                _f64(x["g"][l:l + 1, :, h:h + 1]), _f64(x["beta"][l:l + 1, :, h:h + 1]), ref_states[(l, h)])
        if s.evictions > n_evictions:                          # this chunk evicted
            n_evictions = s.evictions
            ids = np.concatenate([prev_ids.cpu().numpy(), np.full(C, c, np.int32)])
            scores = s.chunk_scores[: c + 1].cpu().numpy()
            ref_idx, _ = oracle.select_retain(M, n_s, n_w, N, ids, scores)
            nn = int(s.n_retained.item())
            assert nn == M
            assert np.array_equal(s.retain_idx[:nn].cpu().numpy(), ref_idx), f"chunk {c}"
            assert np.array_equal(s.tok_chunk[:nn].cpu().numpy(), ids[ref_idx])
        if c == n_chunks - 1:
            last_x = x
    assert n_evictions == n_chunks - n_fill
    assert L.deltas_get_device_status(s.workspace) == (0, 0)

    # state trajectory of the sampled heads
    st = s.state
    for (l, h), ref in ref_states.items():
        got = _f64(st[l, h])
        rel = np.linalg.norm(got - ref[0, 0]) / np.linalg.norm(ref[0, 0])
        assert rel <= STATE_TOL, ((l, h), rel)

    # drift partials of the last chunk, replayed from the GPU's S_before
    for (l, h) in heads:
        kh = h * Hk // Hv
        sb = _f64(s_before_last[l:l + 1, h:h + 1])
        sa, _ = oracle.gdn_recurrence(None, _f64(last_x["k"][l:l + 1, :, kh:kh + 1]),
                                      _f64(last_x["v"][l:l + 1, :, h:h + 1]), _f64(last_x["g"][l:l + 1, :, h:h + 1]),
                                      _f64(last_x["beta"][l:l + 1, :, h:h + 1]), sb)
        p_ref = oracle.drift_partials(sb, sa)[0, 0]
        np.testing.assert_allclose(_f64(s.partials[l, h]), p_ref, rtol=1e-3)

    # sampled rows of the final caches equal the rows they were appended from
    n = s.cache_len
    tc = s.tok_chunk[:n].cpu().numpy()
    tp = s.tok_pos[:n].cpu().numpy()
    assert np.all(np.diff(tp) > 0)                            # stream order, positions kept
    slots = np.sort(rng.choice(n, size=512, replace=False))
    for c in np.unique(tc[slots]):
        sel = slots[tc[slots] == c]
        k_new, v_new = kvn(int(c))
        rows = torch.as_tensor(tp[sel] - int(c) * C, device=dev, dtype=torch.long)
        js = torch.as_tensor(sel, device=dev, dtype=torch.long)
        assert torch.equal(s.k_cache[:, :, js], k_new[:, :, rows])
        assert torch.equal(s.v_cache[:, :, js], v_new[:, :, rows])
