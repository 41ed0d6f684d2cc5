"""Alg. 1 of the paper (DeltaS: state-guided KV eviction) run end to end on the CPU oracle.

Test infrastructure only.  One iteration per arriving chunk c:

1. ``S_before <- S``;
2. ``Prefill(c)``: the gated delta rule (Eq. 2) updates S over the chunk's tokens, and the
   chunk's keys/values are appended to every full-attention cache;
3. ``Delta S`` of Eq. 3 from S_before and S, stored (in float32, as the paper computes all scores
   in float32) as the score of every token of c (or, with ``signal="write_norm"``, the comparison
   signal of Sec. 4.3: the tokens' write sizes beta_t ||v_t - alpha_t S_{t-1} k_t|| averaged over
   heads, layers and the chunk's tokens);
4. if the cache holds more than M tokens: sink / window / spans / quota + fill (Sec. 3.3), then
   the in-stream-order gather of every cache, keeping original positions.

Scores of earlier chunks are reused at later evictions (Sec. 3.3).

:func:`run_stream_heads` runs the same loop with a cache-internal token signal of Sec. 4.3 (key
norm or value norm) in place of the chunk score: every KV head ranks its own tokens, so every
(layer, KV head) plane keeps its own M tokens, with its own chunk ids, positions and scores.

A question (Sec. 3.3, "Question answering") arriving before chunk c saves the whole stream state
(recurrent state, caches with chunk ids and positions, scores, counters), runs the question's
tokens through the same loop body, and then puts the saved state back: question turns change
nothing that later chunks see.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

from . import (compact_kv, compact_kv_heads, gdn_recurrence, row_norm_scores, select_retain,
               select_retain_tokens, state_drift, write_norm_score)


@dataclass
class StreamResult:
    state: np.ndarray                 # final S [L,Hv,dv,dk] fp64
    chunk_scores: np.ndarray          # [n_chunks] float32
    k_cache: np.ndarray               # [Lf,Hkv,capacity,D]
    v_cache: np.ndarray
    tok_chunk: np.ndarray             # [capacity] int32
    tok_pos: np.ndarray               # [capacity] int32
    cache_len: int
    states_after_chunk: list = field(default_factory=list)
    evictions: list = field(default_factory=list)   # (chunk, retain_idx) per eviction event
    question_states: list = field(default_factory=list)   # S right after each question, before the restore


def run_stream(chunk_inputs, kv_inputs, state0, n_chunks: int, policy: dict, capacity: int,
               q_scale: float | None = None, score_override=None, keep_states: bool = False,
               questions: dict | None = None, signal: str = "drift"):
    """Run Alg. 1 over ``n_chunks`` chunks.

    ``chunk_inputs(c)`` -> (q, k, v, g, beta) numpy arrays in the oracle layouts;
    ``kv_inputs(c)`` -> (k_new, v_new) of shape [Lf,Hkv,C,D];
    ``policy`` = dict(budget_M, n_sink, n_window, n_buckets);
    ``score_override`` (optional) [n_chunks] float32: scores to rank with instead of the oracle's
    own (so that selection can be compared given identical scores);
    ``questions`` (optional) {c: () -> ((q, k, v, g, beta), (k_new, v_new))}: a question arriving
    before chunk c, run as a loop body and then undone.
    """
    S = np.array(state0, dtype=np.float64, copy=True)
    scores = np.zeros(n_chunks, dtype=np.float32)
    kc = vc = None
    tok_chunk = np.zeros(capacity, dtype=np.int32)
    tok_pos = np.zeros(capacity, dtype=np.int32)
    T = 0
    pos = 0
    res = StreamResult(S, scores, None, None, tok_chunk, tok_pos, 0)

    def body(c, gdn_in, kv_in, rank_scores_of):
        nonlocal S, kc, vc, tok_chunk, tok_pos, T, pos
        q, k, v, g, beta = gdn_in
        s_before = S.copy()
        if signal == "write_norm":
            S, _, wn = gdn_recurrence(None, k, v, g, beta, S, q_scale=q_scale, want_write_norms=True)
        else:
            S, _ = gdn_recurrence(None, k, v, g, beta, S, q_scale=q_scale)
        k_new, v_new = kv_in
        Lf, Hkv, C, D = k_new.shape
        if kc is None:
            kc = np.zeros((Lf, Hkv, capacity, D), dtype=k_new.dtype)
            vc = np.zeros_like(kc)
        if T + C > capacity:
            raise ValueError("cache capacity too small for the stream")
        kc[:, :, T:T + C] = k_new
        vc[:, :, T:T + C] = v_new
        tok_chunk[T:T + C] = c
        tok_pos[T:T + C] = np.arange(pos, pos + C, dtype=np.int32)
        T += C
        pos += C
        if signal == "write_norm":
            scores[c] = np.float32(write_norm_score(wn, k.shape[1]))
        else:
            scores[c] = np.float32(state_drift(s_before, S))
        if T > policy["budget_M"]:
            idx, _ = select_retain(policy["budget_M"], policy["n_sink"], policy["n_window"],
                                   policy["n_buckets"], tok_chunk[:T], rank_scores_of()[: c + 1])
            kc, vc, tok_chunk, tok_pos = compact_kv(kc, vc, tok_chunk, tok_pos, idx, T)
            T = int(idx.shape[0])
            return idx
        return None

    for c in range(n_chunks):
        if questions and c in questions:
            saved = (S.copy(), scores.copy(), None if kc is None else kc.copy(), None if vc is None else vc.copy(),
                     tok_chunk.copy(), tok_pos.copy(), T, pos)
            gdn_q, kv_q = questions[c]()
            body(c, gdn_q, kv_q, lambda: scores)
            res.question_states.append(S.copy())
            S, scores, kc, vc, tok_chunk, tok_pos, T, pos = saved
        idx = body(c, chunk_inputs(c), kv_inputs(c),
                   lambda: scores if score_override is None else np.asarray(score_override, np.float32))
        if keep_states:
            res.states_after_chunk.append(S.copy())
        if idx is not None:
            res.evictions.append((c, idx))
    res.state = S
    res.chunk_scores = scores
    res.k_cache, res.v_cache = kc, vc
    res.tok_chunk, res.tok_pos = tok_chunk, tok_pos
    res.cache_len = T
    return res


@dataclass
class HeadStreamResult:
    k_cache: np.ndarray               # [Lf,Hkv,capacity,D]
    v_cache: np.ndarray
    tok_chunk: np.ndarray             # [Lf,Hkv,capacity] int32
    tok_pos: np.ndarray               # [Lf,Hkv,capacity] int32
    tok_score: np.ndarray             # [Lf,Hkv,capacity] float32
    cache_len: int
    evictions: list = field(default_factory=list)   # (chunk, [retain list per plane])


def run_stream_heads(kv_inputs, n_chunks: int, policy: dict, capacity: int, signal: str,
                     score_override=None):
    """Alg. 1's append / select / gather loop with a token signal of Sec. 4.3 ranked per KV head.

    ``kv_inputs(c)`` -> (k_new, v_new) [Lf,Hkv,C,D]; ``signal`` is ``key_norm`` (-||k||) or
    ``value_norm`` (||v||); each appended token gets its score once, from its own row (the score
    depends on nothing else, so it equals a score recomputed from the cache at eviction time).
    ``score_override(c)`` (optional) -> [Lf,Hkv,C] float32 scores to rank chunk c's tokens with
    instead of the oracle's own (selection compared given identical scores).  The recurrent state
    is not involved: run :func:`run_stream` or the recurrence for it."""
    kc = vc = None
    T = pos = 0
    res = HeadStreamResult(None, None, None, None, None, 0)
    for c in range(n_chunks):
        k_new, v_new = kv_inputs(c)
        Lf, Hkv, C, D = k_new.shape
        if kc is None:
            kc = np.zeros((Lf, Hkv, capacity, D), dtype=k_new.dtype)
            vc = np.zeros_like(kc)
            tok_chunk = np.zeros((Lf, Hkv, capacity), np.int32)
            tok_pos = np.zeros((Lf, Hkv, capacity), np.int32)
            tok_score = np.zeros((Lf, Hkv, capacity), np.float32)
        if T + C > capacity:
            raise ValueError("cache capacity too small for the stream")
        kc[:, :, T:T + C] = k_new
        vc[:, :, T:T + C] = v_new
        tok_chunk[:, :, T:T + C] = c
        tok_pos[:, :, T:T + C] = np.arange(pos, pos + C, dtype=np.int32)
        if score_override is not None:
            tok_score[:, :, T:T + C] = np.asarray(score_override(c), np.float32)
        else:
            rows = k_new if signal == "key_norm" else v_new
            if rows.dtype == np.int16:                       # bf16 bit patterns -> float32, exactly
                rows = (rows.astype(np.int32) << 16).view(np.float32)
            tok_score[:, :, T:T + C] = row_norm_scores(rows, signal)
        T += C
        pos += C
        if T > policy["budget_M"]:
            lists = [select_retain_tokens(policy["budget_M"], policy["n_sink"], policy["n_window"],
                                          policy["n_buckets"], tok_chunk[l, h, :T], tok_score[l, h, :T])[0]
                     for l in range(Lf) for h in range(Hkv)]
            kc, vc, tok_chunk, tok_pos, tok_score = compact_kv_heads(kc, vc, tok_chunk, tok_pos, tok_score,
                                                                     lists, T)
            T = int(lists[0].shape[0])
            res.evictions.append((c, lists))
    res.k_cache, res.v_cache = kc, vc
    res.tok_chunk, res.tok_pos, res.tok_score = tok_chunk, tok_pos, tok_score
    res.cache_len = T
    return res
