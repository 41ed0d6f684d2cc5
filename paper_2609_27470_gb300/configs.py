"""The synthetic workloads, shaped like the paper's hybrid backbone (Sec. 4.1, App. A).

* ``tiny``      — 1 gated-delta layer, 2 heads, d=16, fp32, 8 chunks x 64 tokens, zero start
                  state, 1 full-attention layer (2 KV heads, D=16, fp32 KV), budget 4 chunks.
* ``layer``     — 1 layer at the backbone's width: 16 key heads, 32 value heads, d=128, bf16
                  activations, fp32 state, 16 chunks x 1024 tokens.
* ``stack``     — 24 gated-delta layers x 32 value heads x 128 x 128 fp32 state (48 MiB,
                  Sec. 3.1), 256 chunks x 1024 tokens, states carried across chunks.
* ``kv``        — 8 full-attention layers, 2 KV heads, D=256 bf16, a 64k-token cache of
                  64 chunks x 1024 tokens, Exp(1) chunk scores with exact ties, budget 16k.
* ``streaming`` — ``stack`` with 512-token chunks plus ``kv`` caches, 4096 chunks, budget 32k,
                  the paper's policy (n_s=4, n_w=1024, N=4; Sec. 4.1).
* ``paper_key_norm``, ``paper_value_norm`` — ``paper`` ranked per KV head by the key norm or the
                  value norm (Sec. 4.3), each plane keeping its own M tokens.
* ``paper``     — the paper's own stream shape (Sec. 4.1, App. A): chunks of two frames, 118-132
                  tokens each (a cycle of eight lengths), 8 full-attention layers x 4 KV heads x
                  D = 256, budget 8192, the paper's policy; gated-delta stack as ``stack``.
"""
from __future__ import annotations

PAPER_POLICY = {"n_sink": 4, "n_window": 1024, "n_buckets": 4}   # Sec. 4.1

TINY = dict(name="tiny", L=1, Hk=2, Hv=2, d=16, dtype="f32", chunk_len=64, n_chunks=8,
            Lf=1, Hkv=2, D=16, kv_dtype="f32", budget_M=256, zero_state=True)

LAYER = dict(name="layer", L=1, Hk=16, Hv=32, d=128, dtype="bf16", chunk_len=1024, n_chunks=16)
# the same with the layer output o_t = q_scale S_t q_t (Alg. 1 Prefill) asked for
LAYER_OUT = dict(LAYER, name="layer_out", with_out=True)

STACK = dict(name="stack", L=24, Hk=16, Hv=32, d=128, dtype="bf16", chunk_len=1024, n_chunks=256,
             ring=8)
# the same with the layer output of every layer
STACK_OUT = dict(STACK, name="stack_out", with_out=True)

# the standalone drift (Eq. 3) of the full stack's states: S_before and S_after of 24 layers x 32
# value heads x 128 x 128 fp32 (48 MiB each), a ring of 4 pairs (384 MiB, beyond L2)
DRIFT = dict(name="drift", L=24, Hk=16, Hv=32, d=128, chunk_len=512, n_chunks=4096, ring=4)

KV = dict(name="kv", Lf=8, Hkv=2, D=256, kv_dtype="bf16", chunk_len=1024, n_chunks=64,
          budget_M=16384)

STREAMING = dict(name="streaming", L=24, Hk=16, Hv=32, d=128, dtype="bf16", chunk_len=512,
                 n_chunks=4096, ring=8, Lf=8, Hkv=2, D=256, kv_dtype="bf16", budget_M=32768,
                 **PAPER_POLICY)

# chunk lengths cycle through these (118-132 tokens: two frames plus timestamps, Sec. 4.1)
PAPER_CHUNK_LENS = (118, 132, 124, 121, 129, 119, 127, 125)

PAPER = dict(name="paper", L=24, Hk=16, Hv=32, d=128, dtype="bf16", chunk_len=max(PAPER_CHUNK_LENS),
             chunk_lens=PAPER_CHUNK_LENS, n_chunks=4096, ring=8, Lf=8, Hkv=4, D=256, kv_dtype="bf16",
             budget_M=8192, **PAPER_POLICY)

# the paper stream scored by the comparison signal of Sec. 4.3 (write sizes) instead of drift
PAPER_WRITE_NORM = dict(PAPER, name="paper_write_norm", signal="write_norm")

# the paper stream ranked by a cache-internal token signal of Sec. 4.3, per KV head and token:
# the key norm (-||k||) or the value norm (||v||)
PAPER_KEY_NORM = dict(PAPER, name="paper_key_norm", signal="key_norm")
PAPER_VALUE_NORM = dict(PAPER, name="paper_value_norm", signal="value_norm")

ALL = {c["name"]: c for c in (TINY, LAYER, STACK, KV, STREAMING, PAPER, PAPER_WRITE_NORM, PAPER_KEY_NORM,
                              PAPER_VALUE_NORM)}
