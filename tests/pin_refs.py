"""Independent formulations used to pin the CPU oracle (not the oracle, not the CUDA path).

* :func:`gdn_chunked_wy` — the chunkwise (WY / UT-transform) form of the gated delta rule: over a
  tile of C tokens with cumulative log-decay G, the tile's writes U solve
  (I + A) U = diag(beta) (V - diag(e^G) K S0^T), A strictly lower with
  A[t,i] = beta_t e^(G_t - G_i) k_t.k_i, and S_C = e^(G_C) S0 + U^T diag(e^(G_C - G)) K.
  It is an algebraic rearrangement of Eq. 1/2 (Sec. 3.2), so it must agree with the token loop
  to rounding at every tile size.
* :func:`select_by_global_sort` — a second implementation of the Sec. 3.3 retention: one global
  ranking, a single pass that fills each span up to its quota, a second pass that fills the rest.
* :func:`select_by_max_weight` — exhaustive search: among all candidate subsets of size
  M - n_s - n_w that give every span at least min(quota, |span|) members, the one with the largest
  sum of 2^rank (rank in the score order).  Quota-then-fill is the greedy algorithm on this
  (matroid) constraint family, so with strictly ordered keys the two coincide.

Both selection references take ``per_slot=True`` for the token signals of Sec. 4.3: ``scores``
then holds one score per slot instead of one per chunk.
"""
from __future__ import annotations

import itertools

import numpy as np


def gdn_chunked_wy(q, k, v, g, beta, S0, C: int, q_scale: float, want_out: bool):
    k = np.asarray(k, np.float64)
    v = np.asarray(v, np.float64)
    g = np.asarray(g, np.float64)
    beta = np.asarray(beta, np.float64)
    L, T, Hk, dk = k.shape
    Hv, dv = v.shape[2], v.shape[3]
    S_all = np.array(S0, dtype=np.float64, copy=True)
    out = np.zeros((L, T, Hv, dv)) if want_out else None
    qq = np.asarray(q, np.float64) if want_out else None
    for l in range(L):
        for h in range(Hv):
            kh = (h * Hk) // Hv
            S = S_all[l, h]
            for t0 in range(0, T, C):
                t1 = min(t0 + C, T)
                K = k[l, t0:t1, kh]
                V = v[l, t0:t1, h]
                b = beta[l, t0:t1, h]
                G = np.cumsum(g[l, t0:t1, h])
                n = t1 - t0
                decay = np.exp(G[:, None] - G[None, :])
                A = np.tril(b[:, None] * decay * (K @ K.T), k=-1)
                U = np.linalg.solve(np.eye(n) + A, b[:, None] * (V - np.exp(G)[:, None] * (K @ S.T)))
                if want_out:
                    Q = qq[l, t0:t1, kh]
                    P = np.tril(decay * (Q @ K.T))
                    out[l, t0:t1, h] = q_scale * (np.exp(G)[:, None] * (Q @ S.T) + P @ U)
                S = np.exp(G[-1]) * S + U.T @ (np.exp(G[-1] - G)[:, None] * K)
            S_all[l, h] = S
    return S_all, out


def _score_key(s: float) -> int:
    b = int(np.array([s], dtype=np.float32).view(np.uint32)[0])
    return (~b) & 0xFFFFFFFF if b & 0x80000000 else b | 0x80000000


def _spans(tok_chunk, lo, hi, N):
    a = np.asarray(tok_chunk[lo:hi], np.int64)
    c_lo, c_hi = int(a.min()), int(a.max())
    return ((a - c_lo) * N) // (c_hi - c_lo + 1)


def _slot_score(tok_chunk, scores, per_slot):
    return (lambda i: scores[i]) if per_slot else (lambda i: scores[tok_chunk[i]])


def select_by_global_sort(M, n_s, n_w, N, tok_chunk, scores, per_slot=False):
    tok_chunk = np.asarray(tok_chunk)
    score_of = _slot_score(tok_chunk, scores, per_slot)
    T = len(tok_chunk)
    if T <= M:
        return list(range(T))
    N = max(N, 1)
    lo, hi = n_s, T - n_w
    R = M - n_s - n_w
    quota = R // N
    spans = _spans(tok_chunk, lo, hi, N)
    order = sorted(range(lo, hi), key=lambda i: (-_score_key(score_of(i)), i))
    keep = set(range(n_s)) | set(range(hi, T))
    used = [0] * N
    for i in order:
        j = spans[i - lo]
        if used[j] < quota:
            used[j] += 1
            keep.add(i)
    left = R - sum(used)
    for i in order:
        if left == 0:
            break
        if i not in keep:
            keep.add(i)
            left -= 1
    return sorted(keep)


def select_by_max_weight(M, n_s, n_w, N, tok_chunk, scores, per_slot=False):
    tok_chunk = np.asarray(tok_chunk)
    score_of = _slot_score(tok_chunk, scores, per_slot)
    T = len(tok_chunk)
    if T <= M:
        return list(range(T))
    N = max(N, 1)
    lo, hi = n_s, T - n_w
    R = M - n_s - n_w
    quota = R // N
    spans = _spans(tok_chunk, lo, hi, N)
    cand = list(range(lo, hi))
    order = sorted(cand, key=lambda i: (_score_key(score_of(i)), -i))  # worst first
    weight = {i: 1 << r for r, i in enumerate(order)}
    need = [min(quota, int(np.sum(spans == j))) for j in range(N)]
    best, best_w = None, -1
    for sub in itertools.combinations(cand, R):
        cnt = [0] * N
        for i in sub:
            cnt[spans[i - lo]] += 1
        if any(cnt[j] < need[j] for j in range(N)):
            continue
        w = sum(weight[i] for i in sub)
        if w > best_w:
            best, best_w = sub, w
    return sorted(set(range(n_s)) | set(best) | set(range(hi, T)))
