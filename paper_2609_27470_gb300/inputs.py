"""Seeded synthetic inputs shaped like the paper's workloads.

This module holds input generation only — none of the method's arithmetic — so both the CUDA
path's tests/benchmark and the CPU oracle can be fed the same bytes.

Distributions (the paper's backbone is not available, so activations are synthetic):
* q, k ~ N(0, 1), then L2-normalised per token and head (the paper's keys are L2-normalised,
  Sec. 3.2); rounded once to the activation dtype (bf16 round-to-nearest-even when bf16).
* v ~ N(0, 1).
* log-decay g = -0.1 * softplus(N(0, 1))  (alpha = exp(g) in (0, 1)).
* write strength beta = sigmoid(N(0, 1)).
* full-attention K, V ~ N(0, 1).
* chunk scores ~ Exp(1) with injected exact ties.

Layouts match the library: q,k [L,T,Hk,d]; v [L,T,Hv,d]; g,beta [L,T,Hv]; new K/V of a chunk
[Lf,Hkv,C,D].
"""
from __future__ import annotations

import torch

_DT = {"bf16": torch.bfloat16, "f32": torch.float32}


def seed_for(base: int, *parts: int) -> int:
    """Deterministic 63-bit seed from a base seed and integer coordinates (config, layer, chunk)."""
    s = (base * 0x9E3779B97F4A7C15 + 0x632BE59BD9B4E019) & ((1 << 64) - 1)
    for p in parts:
        s ^= (p + 0x9E3779B97F4A7C15 + (s << 6) + (s >> 2)) & ((1 << 64) - 1)
        s = (s * 0xBF58476D1CE4E5B9) & ((1 << 64) - 1)
    return s & ((1 << 63) - 1)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _softplus(x: torch.Tensor) -> torch.Tensor:
    # log(1 + e^x), written so that large x does not overflow
    return torch.clamp(x, min=0) + torch.log1p(torch.exp(-torch.abs(x)))


def _sigmoid(x: torch.Tensor) -> torch.Tensor:
    return 1.0 / (1.0 + torch.exp(-x))


def gdn_chunk(L: int, T: int, Hk: int, Hv: int, d: int, dtype: str, seed: int, device="cpu",
              decay_scale: float = 0.1):
    """One chunk of gated-delta-rule inputs: returns dict(q, k, v, g, beta)."""
    gen = _gen(seed, device)
    f32 = torch.float32
    q = torch.randn(L, T, Hk, d, generator=gen, device=device, dtype=f32)
    k = torch.randn(L, T, Hk, d, generator=gen, device=device, dtype=f32)
    v = torch.randn(L, T, Hv, d, generator=gen, device=device, dtype=f32)
    g = -decay_scale * _softplus(torch.randn(L, T, Hv, generator=gen, device=device, dtype=f32))
    beta = _sigmoid(torch.randn(L, T, Hv, generator=gen, device=device, dtype=f32))
    q = q / torch.linalg.vector_norm(q, dim=-1, keepdim=True)
    k = k / torch.linalg.vector_norm(k, dim=-1, keepdim=True)
    dt = _DT[dtype]
    return {"q": q.to(dt).contiguous(), "k": k.to(dt).contiguous(), "v": v.to(dt).contiguous(),
            "g": g.contiguous(), "beta": beta.contiguous()}


def initial_state(L: int, Hv: int, d: int, seed: int, device="cpu", scale: float = 1.0):
    """A nonzero starting state [L,Hv,d,d] fp32 (so that the drift denominator is positive)."""
    gen = _gen(seed, device)
    return (scale * torch.randn(L, Hv, d, d, generator=gen, device=device, dtype=torch.float32)
            / (d ** 0.5)).contiguous()


def kv_chunk(Lf: int, Hkv: int, C: int, D: int, dtype: str, seed: int, device="cpu"):
    """New keys and values of one chunk for every full-attention layer: [Lf,Hkv,C,D] each."""
    gen = _gen(seed, device)
    k = torch.randn(Lf, Hkv, C, D, generator=gen, device=device, dtype=torch.float32)
    v = torch.randn(Lf, Hkv, C, D, generator=gen, device=device, dtype=torch.float32)
    dt = _DT[dtype]
    return k.to(dt).contiguous(), v.to(dt).contiguous()


def kv_cache(Lf: int, Hkv: int, capacity: int, D: int, dtype: str, seed: int, device="cpu"):
    """A full cache [Lf,Hkv,capacity,D] of K and V ~ N(0,1)."""
    gen = _gen(seed, device)
    dt = _DT[dtype]
    k = torch.empty(Lf, Hkv, capacity, D, device=device, dtype=dt)
    v = torch.empty(Lf, Hkv, capacity, D, device=device, dtype=dt)
    for a in (k, v):
        for layer in range(Lf):   # per layer keeps the fp32 temporary small
            a[layer].copy_(torch.randn(Hkv, capacity, D, generator=gen, device=device,
                                       dtype=torch.float32).to(dt))
    return k, v


def chunk_scores_with_ties(n_chunks: int, seed: int, tie_rank: int = 16, n_ties: int = 6):
    """Exp(1) chunk scores; ``n_ties`` other chunks are set to exactly the ``tie_rank``-th largest
    value, so that a top-``tie_rank`` cut falls inside a group of equal scores."""
    gen = _gen(seed, "cpu")
    s = torch.empty(n_chunks, dtype=torch.float32).exponential_(1.0, generator=gen)
    if 0 < tie_rank <= n_chunks and n_ties > 0:
        order = torch.argsort(s, descending=True)
        tv = s[order[tie_rank - 1]].clone()
        others = order[tie_rank:]
        pick = others[torch.randperm(others.numel(), generator=gen)[:n_ties]]
        s[pick] = tv
    return s


def chunked_tok_chunk(n_chunks: int, chunk_len: int):
    """Per-slot arrival chunk of a cache filled with whole chunks in stream order."""
    return torch.arange(n_chunks, dtype=torch.int32).repeat_interleave(chunk_len)
