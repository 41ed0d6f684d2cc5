"""Alg. 1 (DeltaS: state-guided KV eviction) driven through the C ABI on one GPU.

Per arriving chunk c, all on one CUDA stream and with no host synchronisation:

1. ``deltas_gdn_chunk_update`` — Prefill(c) of every gated-delta layer: the state S goes from
   S_before to S_after (Eq. 1) and the per-(layer, head) drift partials come out of the same
   kernel (the pre-chunk state is never stored separately);
2. ``deltas_score_chunks`` — Delta S of Eq. 3, stored as score[c] (shared by c's tokens); with
   ``signal="write_norm"`` the chunk is scored instead by the comparison signal of Sec. 4.3, the
   tokens' write sizes beta_t ||v_t - alpha_t S_{t-1} k_t|| averaged over heads, layers and
   tokens (``deltas_gdn_chunk_update_write_norms`` + ``deltas_score_write_norms``);
3. ``deltas_append_kv`` — c's keys/values enter every full-attention cache, with their arrival
   chunk and stream position;
4. if the cache holds more than M tokens: ``deltas_select_retain`` then ``deltas_compact_kv``.

The host tracks the cache length without reading the device: after an eviction it is exactly M
(the selection keeps min(T, M) tokens).

With ``signal="key_norm"`` or ``"value_norm"`` the stream ranks tokens by a cache-internal signal
of Sec. 4.3 instead (-||k|| or ||v||, per KV head and per token): step 2 is dropped (the update
runs without drift partials), step 3 is ``deltas_append_kv_heads`` (which also scores the new
tokens) and step 4 is ``deltas_select_retain_heads`` + ``deltas_compact_kv_heads``: every
(layer, KV head) plane keeps its own M tokens, so ``tok_chunk``, ``tok_pos`` and ``tok_score``
are [Lf, Hkv, capacity] and ``retain_idx`` is [Lf * Hkv, M].

Questions (Sec. 3.3): ``snapshot()`` saves the stream state before a question and ``restore()``
puts it back after the answer (``deltas_copy_stream_state``: the recurrent state, the chunk
scores, and unless ``full=False`` the live cache rows with their chunk ids and positions; the host
counters travel with it), so whatever the question ran on the stream in between, appends,
updates or evictions, leaves no trace in the subsequent stream.
"""
from __future__ import annotations

import torch

from . import _lib as L


class StreamSnapshot:
    """A saved stream state: device copies of the buffers ``deltas_copy_stream_state`` moves and
    the host counters.  ``full=False`` keeps the recurrent state and the scores only (enough when
    the question appends to the caches but evicts nothing)."""

    def __init__(self, s: "DeltaSStream", full: bool = True):
        self.full = full
        self.buffers = {"state": torch.empty_like(s.state), "chunk_scores": torch.empty_like(s.chunk_scores)}
        if full:
            for n in ("k_cache", "v_cache", "tok_chunk", "tok_pos") + (("tok_score",) if s.per_head else ()):
                self.buffers[n] = torch.empty_like(getattr(s, n))
        self.cache_len = self.position = self.chunk = self.evictions = 0


class DeltaSStream:
    def __init__(self, *, num_layers, num_k_heads, num_v_heads, head_dim, act_dtype: torch.dtype,
                 kv_layers, kv_heads, kv_head_dim, kv_dtype: torch.dtype, budget_M, n_sink=0,
                 n_window=0, n_buckets=1, chunk_len, max_chunks, q_scale=None, state0=None,
                 device="cuda", signal: str = "drift", read_out: bool = False):
        if signal not in ("drift", "write_norm") + tuple(L.SIGNALS):
            raise ValueError(f"unknown signal {signal!r}")
        self.signal = signal
        self.per_head = signal in L.SIGNALS
        self.gdn = L.gdn_desc(num_layers, num_k_heads, num_v_heads, head_dim, act_dtype, q_scale)
        self.policy = L.policy(budget_M, n_sink, n_window, n_buckets)
        self.capacity = budget_M + chunk_len
        if signal in L.SIGNALS:          # per-plane metadata rows start on 16-byte boundaries
            self.capacity = (self.capacity + 3) // 4 * 4
        self.kv = L.kv_desc(kv_layers, kv_heads, kv_head_dim, kv_dtype, self.capacity)
        self.chunk_len = chunk_len
        self.max_chunks = max_chunks
        dev = torch.device(device)
        self.state = (state0.clone() if state0 is not None else
                      torch.zeros(num_layers, num_v_heads, head_dim, head_dim, device=dev))
        self.partials = None if self.per_head else torch.zeros(num_layers, num_v_heads, 2, device=dev)
        self.write_norms = torch.zeros(num_layers, num_v_heads, device=dev) if signal == "write_norm" else None
        self.chunk_scores = torch.zeros(max_chunks, device=dev)
        self.k_cache = torch.zeros(kv_layers, kv_heads, self.capacity, kv_head_dim, dtype=kv_dtype, device=dev)
        self.v_cache = torch.zeros_like(self.k_cache)
        meta = (kv_layers, kv_heads, self.capacity) if self.per_head else (self.capacity,)
        self.tok_chunk = torch.zeros(meta, dtype=torch.int32, device=dev)
        self.tok_pos = torch.zeros(meta, dtype=torch.int32, device=dev)
        self.tok_score = torch.zeros(meta, device=dev) if self.per_head else None
        lists = (kv_layers * kv_heads, budget_M) if self.per_head else (budget_M,)
        self.retain_idx = torch.zeros(lists, dtype=torch.int32, device=dev)
        self.n_retained = torch.zeros(1, dtype=torch.int32, device=dev)
        # read_out: step() may be given ``out`` (the layer output o_t); the update's workspace then
        # also holds each token's write and the block states (d = 128 bf16)
        gdn_ws = (L.deltas_gdn_chunk_update_readout_workspace_size if read_out else
                  L.deltas_gdn_chunk_update_workspace_size)(self.gdn, chunk_len)
        self.read_out = read_out
        if self.per_head:
            ws = max(gdn_ws,
                     L.deltas_select_retain_heads_workspace_size(kv_layers * kv_heads, self.capacity),
                     L.deltas_compact_kv_heads_workspace_size(self.kv, self.capacity))
        else:
            ws = max(gdn_ws,
                     L.deltas_select_retain_workspace_size(self.capacity),
                     L.deltas_compact_kv_workspace_size(self.kv, self.capacity))
        self.workspace = L.alloc_workspace(ws, dev)
        self.cache_len = 0
        self.position = 0
        self.chunk = 0
        self.evictions = 0

    def step(self, q, k, v, g, beta, k_new, v_new, out=None, stream=None):
        """Process one chunk (Alg. 1 loop body).  Returns True if an eviction ran."""
        c = self.chunk
        if c >= self.max_chunks:
            raise ValueError("stream longer than max_chunks")
        T = int(k.shape[1])
        if out is not None and not self.read_out:
            raise ValueError("step(out=...) needs a stream built with read_out=True")
        L.deltas_gdn_chunk_update(self.gdn, T, q, k, v, g, beta, self.state, out, self.partials,
                                  self.workspace, stream, write_norms=self.write_norms)
        if self.per_head:
            return self._step_heads(k_new, v_new, stream)
        if self.signal == "write_norm":
            L.deltas_score_write_norms(self.gdn.num_layers, self.gdn.num_v_heads, self.write_norms, T, c,
                                       self.chunk_scores, stream)
        else:
            L.deltas_score_chunks(self.gdn.num_layers, self.gdn.num_v_heads, self.partials, c,
                                  self.chunk_scores, stream)
        n_new = int(k_new.shape[2])
        L.deltas_append_kv(self.kv, self.k_cache, self.v_cache, self.tok_chunk, self.tok_pos,
                           self.cache_len, k_new, v_new, c, self.position, stream)
        self.cache_len += n_new
        self.position += n_new
        self.chunk += 1
        if self.cache_len > self.policy.budget_M:
            L.deltas_select_retain(self.policy, self.cache_len, self.tok_chunk,
                                   self.chunk_scores[: c + 1], self.retain_idx, self.n_retained,
                                   None, self.workspace, stream)
            L.deltas_compact_kv(self.kv, self.k_cache, self.v_cache, self.tok_chunk, self.tok_pos,
                                self.retain_idx, self.n_retained, self.cache_len, self.workspace,
                                stream)
            self.cache_len = self.policy.budget_M
            self.evictions += 1
            return True
        return False

    def _step_heads(self, k_new, v_new, stream):
        c = self.chunk
        n_new = int(k_new.shape[2])
        L.deltas_append_kv_heads(self.kv, self.signal, self.k_cache, self.v_cache, self.tok_chunk, self.tok_pos,
                                 self.tok_score, self.cache_len, k_new, v_new, c, self.position, stream)
        self.cache_len += n_new
        self.position += n_new
        self.chunk += 1
        if self.cache_len > self.policy.budget_M:
            P = self.kv.num_layers * self.kv.num_kv_heads
            L.deltas_select_retain_heads(self.policy, self.cache_len, self.tok_chunk.view(P, -1),
                                         self.tok_score.view(P, -1), self.retain_idx, self.n_retained, None,
                                         self.workspace, stream)
            L.deltas_compact_kv_heads(self.kv, self.k_cache, self.v_cache, self.tok_chunk, self.tok_pos,
                                      self.tok_score, self.retain_idx, self.n_retained, self.cache_len,
                                      self.workspace, stream)
            self.cache_len = self.policy.budget_M
            self.evictions += 1
            return True
        return False

    def _buffers(self, full: bool) -> dict:
        b = {"state": self.state, "chunk_scores": self.chunk_scores}
        if full:
            b.update(k_cache=self.k_cache, v_cache=self.v_cache, tok_chunk=self.tok_chunk, tok_pos=self.tok_pos)
            if self.per_head:
                b["tok_score"] = self.tok_score
        return b

    def snapshot(self, full: bool = True, into: StreamSnapshot | None = None, stream=None) -> StreamSnapshot:
        """Save the stream state before a question (Sec. 3.3); ``into`` reuses a snapshot's buffers."""
        snap = into if into is not None else StreamSnapshot(self, full)
        if snap.full != full:
            raise ValueError("the snapshot's buffers were made for the other kind of snapshot")
        L.deltas_copy_stream_state(self.gdn, self.kv if full else None, self.cache_len, self.chunk,
                                   self._buffers(full), snap.buffers, stream, per_head=self.per_head and full)
        snap.cache_len, snap.position, snap.chunk, snap.evictions = (self.cache_len, self.position, self.chunk,
                                                                     self.evictions)
        return snap

    def restore(self, snap: StreamSnapshot, stream=None):
        """Put the stream back to ``snap`` after the answer: nothing the question ran remains."""
        if not snap.full and self.evictions != snap.evictions:
            raise ValueError("the question evicted from the cache: only a full snapshot can restore it")
        L.deltas_copy_stream_state(self.gdn, self.kv if snap.full else None, snap.cache_len, snap.chunk,
                                   snap.buffers, self._buffers(snap.full), stream, per_head=self.per_head and snap.full)
        self.cache_len, self.position, self.chunk, self.evictions = (snap.cache_len, snap.position, snap.chunk,
                                                                     snap.evictions)
