"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU needed).

Each test names the passage it checks.  None of them re-types the oracle's own loop: they use
hand-worked values, exact high-precision arithmetic, a second formulation (Eq. 1 vs Eq. 2, the
chunkwise WY form), closed forms, invariants and exhaustive search.
"""
import json
import os

import numpy as np
import pytest

import oracle
from oracle.stream import run_stream, run_stream_heads
from pin_refs import gdn_chunked_wy, select_by_global_sort, select_by_max_weight

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rand_inputs(rng, L, T, Hk, Hv, d, decay=0.1):
    q = rng.standard_normal((L, T, Hk, d))
    k = rng.standard_normal((L, T, Hk, d))
    q /= np.linalg.norm(q, axis=-1, keepdims=True)
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    v = rng.standard_normal((L, T, Hv, d))
    g = -decay * np.log1p(np.exp(rng.standard_normal((L, T, Hv))))
    beta = 1.0 / (1.0 + np.exp(-rng.standard_normal((L, T, Hv))))
    f = lambda a: a.astype(np.float32)
    return f(q), f(k), f(v), f(g), f(beta)


def _rel(a, b):
    return float(np.linalg.norm(np.asarray(a) - np.asarray(b)) / max(np.linalg.norm(b), 1e-300))


# ---------------------------------------------------------------- recurrence (Eq. 1 / Eq. 2)

def test_recurrence_hand_worked_d2():
    """Sec. 3.2 Eq. 1/2: hand-worked 2x2 example (tests/golden/recurrence_d2.json)."""
    gold = json.load(open(os.path.join(GOLDEN, "recurrence_d2.json")))
    toks = gold["tokens"]
    T = len(toks)
    k = np.array([t["k"] for t in toks], np.float32).reshape(1, T, 1, 2)
    q = np.array([t["q"] for t in toks], np.float32).reshape(1, T, 1, 2)
    v = np.array([t["v"] for t in toks], np.float32).reshape(1, T, 1, 2)
    g = np.log(np.array([t["alpha"] for t in toks])).astype(np.float32).reshape(1, T, 1)
    beta = np.array([t["beta"] for t in toks], np.float32).reshape(1, T, 1)
    S0 = np.array(gold["S0"]).reshape(1, 1, 2, 2)
    for n in range(1, T + 1):
        S, out = oracle.gdn_recurrence(q[:, :n], k[:, :n], v[:, :n], g[:, :n], beta[:, :n], S0,
                                       q_scale=1.0, want_out=True)
        np.testing.assert_allclose(S[0, 0], gold["S_after_each"][n - 1], rtol=1e-6, atol=1e-6)
        np.testing.assert_allclose(out[0, :, 0], gold["o"][:n], rtol=1e-6, atol=1e-6)


def test_recurrence_exact_arithmetic_brute_force():
    """Eq. 1 evaluated in 60-digit arithmetic (mpmath) on tiny random inputs matches the oracle."""
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 60
    rng = np.random.default_rng(11)
    for d, T in ((2, 5), (3, 4), (4, 3)):
        q, k, v, g, beta = _rand_inputs(rng, 1, T, 1, 1, d, decay=0.3)
        S0 = rng.standard_normal((1, 1, d, d))
        S = mpmath.matrix([[mpmath.mpf(float(S0[0, 0, i, j])) for j in range(d)] for i in range(d)])
        for t in range(T):
            kt = mpmath.matrix([mpmath.mpf(float(x)) for x in k[0, t, 0]])
            vt = mpmath.matrix([mpmath.mpf(float(x)) for x in v[0, t, 0]])
            a = mpmath.exp(mpmath.mpf(float(g[0, t, 0])))
            b = mpmath.mpf(float(beta[0, t, 0]))
            S = S * (a * (mpmath.eye(d) - b * kt * kt.T)) + b * vt * kt.T
        exact = np.array([[float(S[i, j]) for j in range(d)] for i in range(d)])
        got, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
        np.testing.assert_allclose(got[0, 0], exact, rtol=1e-12, atol=1e-13)


def test_product_form_equals_residual_form():
    """Eq. 1 (product) and Eq. 2 (residual) are the same recurrence (Sec. 3.2)."""
    rng = np.random.default_rng(3)
    q, k, v, g, beta = _rand_inputs(rng, 2, 40, 2, 4, 8)
    S0 = rng.standard_normal((2, 4, 8, 8))
    a, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
    b = oracle.gdn_recurrence_product_form(k, v, g, beta, S0)
    assert _rel(a, b) < 1e-13


@pytest.mark.parametrize("C", [1, 4, 16, 64])
def test_sequential_equals_chunked_wy(C):
    """Token loop == chunkwise WY form at every tile size, ragged tail included (T = 150)."""
    rng = np.random.default_rng(C)
    q, k, v, g, beta = _rand_inputs(rng, 1, 150, 2, 4, 16)
    S0 = rng.standard_normal((1, 4, 16, 16)) * 0.5
    S_seq, o_seq = oracle.gdn_recurrence(q, k, v, g, beta, S0, q_scale=0.25, want_out=True)
    S_wy, o_wy = gdn_chunked_wy(q, k, v, g, beta, S0, C, 0.25, True)
    assert _rel(S_seq, S_wy) < 1e-11
    assert _rel(o_seq, o_wy) < 1e-11


def test_beta_zero_is_pure_decay():
    """beta = 0 leaves only the decay: S_T = exp(sum g) S_0 (Eq. 2 with the write removed)."""
    rng = np.random.default_rng(5)
    q, k, v, g, beta = _rand_inputs(rng, 1, 30, 1, 3, 8)
    beta[:] = 0
    S0 = rng.standard_normal((1, 3, 8, 8))
    S, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
    gamma = np.exp(np.sum(g.astype(np.float64), axis=1))[0]          # per head
    np.testing.assert_allclose(S[0], gamma[:, None, None] * S0[0], rtol=1e-13)


def test_beta_one_writes_value_exactly():
    """beta = 1: the delta rule replaces what k_t retrieves, S_t k_t = v_t for a unit key.  The
    float32 key is unit only to rounding, so the exact identity checked is
    S_t k = |k|^2 v + alpha (1 - |k|^2) S_{t-1} k."""
    rng = np.random.default_rng(6)
    for t in range(8):
        q, k, v, g, beta = _rand_inputs(rng, 1, 1, 1, 2, 8)
        beta[:] = 1
        S0 = rng.standard_normal((1, 2, 8, 8))
        S, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
        kk = k[0, 0, 0].astype(np.float64)
        n2 = kk @ kk
        assert abs(n2 - 1) < 1e-6
        for h in range(2):
            alpha = np.exp(np.float64(g[0, 0, h]))
            expect = n2 * v[0, 0, h].astype(np.float64) + alpha * (1 - n2) * (S0[0, h] @ kk)
            np.testing.assert_allclose(S[0, h] @ kk, expect, rtol=1e-12, atol=1e-13)


def test_orthonormal_keys_rebuild_value_matrix():
    """alpha = 1, beta = 1, keys e_1..e_d: the state becomes sum_i v_i e_i^T whatever S_0 was."""
    d = 6
    rng = np.random.default_rng(7)
    k = np.eye(d, dtype=np.float32).reshape(1, d, 1, d)
    v = rng.standard_normal((1, d, 1, d)).astype(np.float32)
    g = np.zeros((1, d, 1), np.float32)
    beta = np.ones((1, d, 1), np.float32)
    S0 = rng.standard_normal((1, 1, d, d))
    S, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
    np.testing.assert_allclose(S[0, 0], v[0, :, 0].T.astype(np.float64), rtol=0, atol=1e-15)


def test_write_norm_first_token_and_repeated_key():
    """The write size beta_t ||v_t - alpha_t S_{t-1} k_t|| (Sec. 4.3 comparison signal), by hand:
    from S_0 = 0 the first token writes beta_1 v_1; with alpha = beta = 1 a second token on the
    same unit key writes v_2 - v_1 (the state already returns v_1 for that key)."""
    d = 4
    k = np.zeros((1, 2, 1, d), np.float32)
    k[0, :, 0, 1] = 1.0                                              # e_2 twice
    v = np.array([[[[1, 2, 3, 4]], [[2, 0, 3, 8]]]], np.float32)
    g = np.zeros((1, 2, 1), np.float32)
    beta = np.array([[[0.5], [1.0]]], np.float32)
    S0 = np.zeros((1, 1, d, d))
    _, _, wn = oracle.gdn_recurrence(None, k[:, :1], v[:, :1], g[:, :1], beta[:, :1], S0, want_write_norms=True)
    assert wn[0, 0] == pytest.approx(0.5 * np.sqrt(30.0), rel=1e-15)
    beta[:] = 1.0
    _, _, wn = oracle.gdn_recurrence(None, k, v, g, beta, S0, want_write_norms=True)
    assert wn[0, 0] == pytest.approx(np.sqrt(30.0) + np.sqrt(1 + 4 + 0 + 16), rel=1e-15)


def test_write_norm_equals_state_step_change():
    """For a unit key the write u_t k_t^T has Frobenius norm ||u_t||: the sum of write sizes equals
    the sum over tokens of ||S_t - alpha_t S_{t-1}||_F, with the states taken one token at a time
    from the product form of Eq. 1 (a second formulation), for several heads and grouped keys."""
    rng = np.random.default_rng(15)
    L, T, Hk, Hv, d = 2, 9, 1, 2, 6
    q, k, v, g, beta = _rand_inputs(rng, L, T, Hk, Hv, d)
    k = (k.astype(np.float64) / np.linalg.norm(k.astype(np.float64), axis=-1, keepdims=True)).astype(np.float32)
    S0 = rng.standard_normal((L, Hv, d, d))
    _, _, wn = oracle.gdn_recurrence(None, k, v, g, beta, S0, want_write_norms=True)
    S = S0.copy()
    ref = np.zeros((L, Hv))
    for t in range(T):
        sl = slice(t, t + 1)
        S1 = oracle.gdn_recurrence_product_form(k[:, sl], v[:, sl], g[:, sl], beta[:, sl], S)
        alpha = np.exp(g[:, t].astype(np.float64))                  # [L, Hv]
        kk = k[:, t, 0].astype(np.float64)
        n2 = np.sum(kk * kk, axis=-1)                                 # |k|^2 = 1 up to float32 rounding
        ref += np.linalg.norm(S1 - alpha[:, :, None, None] * S, axis=(2, 3)) / np.sqrt(n2)[:, None]
        S = S1
    np.testing.assert_allclose(wn, ref, rtol=1e-10)


def test_write_norm_score_is_the_mean_over_heads_layers_tokens():
    """The chunk score averages the write sizes over heads, layers and the chunk's tokens."""
    wn = np.array([[1.0, 2.0, 3.0], [4.0, 5.0, 6.5]])
    assert oracle.write_norm_score(wn, 7) == pytest.approx(21.5 / (2 * 3 * 7), rel=1e-15)
    assert oracle.write_norm_score(wn, 0) == 0.0


def test_write_norm_zero_without_write():
    """beta = 0: nothing is written, every write size is 0 whatever the state and values."""
    rng = np.random.default_rng(16)
    q, k, v, g, beta = _rand_inputs(rng, 1, 12, 1, 2, 8)
    beta[:] = 0
    _, _, wn = oracle.gdn_recurrence(None, k, v, g, beta, rng.standard_normal((1, 2, 8, 8)), want_write_norms=True)
    assert np.all(wn == 0.0)


def test_contraction_bound():
    """||I - beta k k^T||_2 <= 1 for beta in [0,1], ||k|| = 1, so
    ||S_t||_F <= alpha_t ||S_{t-1}||_F + beta_t ||v_t|| (Eq. 1)."""
    rng = np.random.default_rng(8)
    q, k, v, g, beta = _rand_inputs(rng, 1, 60, 1, 1, 8)
    S = rng.standard_normal((1, 1, 8, 8)) * 3
    for t in range(60):
        Sn, _ = oracle.gdn_recurrence(None, k[:, t:t + 1], v[:, t:t + 1], g[:, t:t + 1], beta[:, t:t + 1], S)
        bound = np.exp(float(g[0, t, 0])) * np.linalg.norm(S) + float(beta[0, t, 0]) * np.linalg.norm(v[0, t, 0])
        assert np.linalg.norm(Sn) <= bound * (1 + 1e-12)
        S = Sn


def test_grouped_keys_mapping():
    """Value head h reads key head floor(h*Hk/Hv): running 4 value heads over 2 key heads equals
    running each value head alone with its key head."""
    rng = np.random.default_rng(9)
    q, k, v, g, beta = _rand_inputs(rng, 1, 20, 2, 4, 8)
    S0 = rng.standard_normal((1, 4, 8, 8))
    S, o = oracle.gdn_recurrence(q, k, v, g, beta, S0, q_scale=0.5, want_out=True)
    for h in range(4):
        kh = h // 2
        Sh, oh = oracle.gdn_recurrence(q[:, :, kh:kh + 1], k[:, :, kh:kh + 1], v[:, :, h:h + 1],
                                       g[:, :, h:h + 1], beta[:, :, h:h + 1], S0[:, h:h + 1],
                                       q_scale=0.5, want_out=True)
        np.testing.assert_array_equal(S[:, h:h + 1], Sh)
        np.testing.assert_array_equal(o[:, :, h:h + 1], oh)


def test_output_reads_the_updated_state():
    """o_t = q_scale * S_t q_t with S_t the state after token t (prefix runs give S_t)."""
    rng = np.random.default_rng(10)
    q, k, v, g, beta = _rand_inputs(rng, 1, 12, 1, 1, 8)
    S0 = rng.standard_normal((1, 1, 8, 8))
    _, o = oracle.gdn_recurrence(q, k, v, g, beta, S0, q_scale=0.3, want_out=True)
    for t in range(12):
        St, _ = oracle.gdn_recurrence(None, k[:, :t + 1], v[:, :t + 1], g[:, :t + 1], beta[:, :t + 1], S0)
        np.testing.assert_allclose(o[0, t, 0], 0.3 * St[0, 0] @ q[0, t, 0].astype(np.float64), rtol=1e-13, atol=1e-14)


@pytest.mark.parametrize("blk", [1, 5, 8, 13])
def test_block_readout_identity(blk):
    """The algebra the GPU read-out uses, checked against the oracle's token loop: unrolling Eq. 1
    from the state S_b before a block, S_t = exp(G_t) S_b + sum_{i <= t} exp(G_t - G_i) u_i k_i^T
    (G the inclusive cumulative log-decay inside the block, u_i = beta_i (v_i - alpha_i S_{i-1} k_i)
    the write of token i), so a block's outputs are q_scale ((Q K^T o D) U + diag(exp(G)) Q S_b^T).
    Blocks of several lengths (one token, and lengths that do not divide T) over 30 tokens."""
    rng = np.random.default_rng(20 + blk)
    T, d, qs = 30, 6, 0.4
    q, k, v, g, beta = _rand_inputs(rng, 1, T, 1, 1, d, decay=0.5)
    S0 = rng.standard_normal((1, 1, d, d))
    _, o_ref = oracle.gdn_recurrence(q, k, v, g, beta, S0, q_scale=qs, want_out=True)
    q, k, v = (x[0, :, 0].astype(np.float64) for x in (q, k, v))
    g, beta = (x[0, :, 0].astype(np.float64) for x in (g, beta))
    S = S0[0, 0].copy()
    u = np.zeros((T, d))
    for t in range(T):                     # the writes u_t of the token loop (plain numpy)
        a = np.exp(g[t])
        u[t] = beta[t] * (v[t] - a * S @ k[t])
        S = a * S + np.outer(u[t], k[t])
    S = S0[0, 0].copy()
    o = np.zeros((T, d))
    for b0 in range(0, T, blk):
        b1 = min(T, b0 + blk)
        G = np.cumsum(g[b0:b1])
        D = np.tril(np.exp(G[:, None] - G[None, :]))
        Q, K, U = q[b0:b1], k[b0:b1], u[b0:b1]
        o[b0:b1] = qs * (((Q @ K.T) * D) @ U + np.exp(G)[:, None] * (Q @ S.T))
        S = np.exp(G[-1]) * S + (np.exp(G[-1] - G)[:, None] * U).T @ K     # the state after the block
    np.testing.assert_allclose(o, o_ref[0, :, 0], rtol=1e-11, atol=1e-12)


# ---------------------------------------------------------------- drift (Eq. 3)

def test_drift_hand_worked_two_layers():
    """Eq. 3: per-layer norms over all heads, mean over layers (tests/golden/drift_two_layers.json)."""
    gold = json.load(open(os.path.join(GOLDEN, "drift_two_layers.json")))
    sb = np.array(gold["S_before"], np.float64)
    sa = np.array(gold["S_after"], np.float64)
    p = oracle.drift_partials(sb, sa)
    np.testing.assert_array_equal(p, np.array(gold["partials"], np.float64))
    assert oracle.chunk_score(p) == pytest.approx(gold["delta_s"], rel=1e-15)


def test_drift_closed_form_pure_decay():
    """beta = 0 and a constant per-head decay gamma_h over the chunk: S_after,h = gamma_h S_0,h, so
    ||S_after - S_before||^2 = sum_h (1 - gamma_h)^2 ||S_0,h||^2 (exact closed form)."""
    rng = np.random.default_rng(12)
    L, Hv, d, T = 3, 4, 8, 25
    q, k, v, g, beta = _rand_inputs(rng, L, T, 2, Hv, d)
    beta[:] = 0
    per_head = -rng.uniform(0.01, 0.2, size=(L, Hv)).astype(np.float32)
    g[:] = per_head[:, None, :]
    S0 = rng.standard_normal((L, Hv, d, d))
    S1, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
    gam = np.exp(T * per_head.astype(np.float64))                      # [L,Hv]
    n0 = np.sum(S0 ** 2, axis=(2, 3))
    expected = np.mean(np.sqrt(np.sum((1 - gam) ** 2 * n0, axis=1)) / np.sqrt(np.sum(n0, axis=1)))
    assert oracle.state_drift(S0, S1) == pytest.approx(expected, rel=1e-11)
    # equal decay everywhere: Delta S = 1 - gamma
    g[:] = np.float32(-0.05)
    S1, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
    gamma = np.exp(T * np.float64(np.float32(-0.05)))
    assert oracle.state_drift(S0, S1) == pytest.approx(1 - gamma, rel=1e-11)


def test_drift_zero_without_decay_or_write():
    """alpha = 1 and beta = 0: the state does not move, Delta S = 0 exactly."""
    rng = np.random.default_rng(13)
    q, k, v, g, beta = _rand_inputs(rng, 2, 30, 1, 2, 8)
    g[:] = 0
    beta[:] = 0
    S0 = rng.standard_normal((2, 2, 8, 8))
    S1, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
    assert oracle.state_drift(S0, S1) == 0.0


def test_drift_scale_invariance():
    """S_0 -> lam S_0 and v -> lam v scales every state by lam, so the normalised drift is unchanged."""
    rng = np.random.default_rng(14)
    q, k, v, g, beta = _rand_inputs(rng, 2, 40, 1, 2, 8)
    S0 = rng.standard_normal((2, 2, 8, 8))
    S1, _ = oracle.gdn_recurrence(None, k, v, g, beta, S0)
    lam = np.float32(4.0)   # a power of two keeps the scaled float32 inputs exact
    S1b, _ = oracle.gdn_recurrence(None, k, v * lam, g, beta, S0 * lam)
    assert oracle.state_drift(S0 * lam, S1b) == pytest.approx(oracle.state_drift(S0, S1), rel=1e-13)


def test_drift_zero_state_reading():
    """The paper leaves ||S_before|| = 0 open: a zero state that receives writes scores +inf; a
    zero state that stays zero scores 0."""
    z = np.zeros((1, 2, 4, 4))
    s = np.zeros((1, 2, 4, 4))
    s[0, 1, 2, 3] = 1e-3
    assert oracle.state_drift(z, s) == np.inf
    assert oracle.state_drift(z, z) == 0.0


# ---------------------------------------------------------------- selection (Sec. 3.3, Alg. 1)

def _select(case):
    idx, mask = oracle.select_retain(case["budget_M"], case["n_sink"], case["n_window"],
                                     case["n_buckets"], case["tok_chunk"], case["chunk_scores"])
    return idx, mask


def test_select_hand_worked_examples():
    gold = json.load(open(os.path.join(GOLDEN, "select_examples.json")))
    for case in gold["cases"]:
        idx, mask = _select(case)
        assert idx.tolist() == case["retain"], case["name"]
        assert mask.tolist() == [1 if i in case["retain"] else 0 for i in range(len(case["tok_chunk"]))]


def _random_case(rng, T_max, ties=True):
    n_ch = int(rng.integers(1, 9))
    lens = rng.integers(1, 5, size=n_ch)
    tok_chunk = np.repeat(np.arange(n_ch, dtype=np.int32), lens)[:T_max]
    T = len(tok_chunk)
    scores = rng.exponential(size=n_ch).astype(np.float32)
    if ties and n_ch > 2:
        scores[rng.integers(0, n_ch, size=2)] = scores[0]
    n_s = int(rng.integers(0, 3))
    n_w = int(rng.integers(0, 3))
    M = int(rng.integers(n_s + n_w + 1, max(n_s + n_w + 2, T + 2)))
    N = int(rng.integers(0, 5))
    return M, n_s, n_w, N, tok_chunk, scores


def test_select_matches_exhaustive_max_weight():
    """Quota-then-fill == the max-weight subset under the span lower bounds (exhaustive, T <= 12)."""
    rng = np.random.default_rng(21)
    n = 0
    while n < 300:
        M, n_s, n_w, N, tc, sc = _random_case(rng, 12)
        if len(tc) <= M:
            continue
        idx, _ = oracle.select_retain(M, n_s, n_w, N, tc, sc)
        assert idx.tolist() == select_by_max_weight(M, n_s, n_w, N, tc, sc)
        n += 1


def test_select_matches_global_sort_implementation():
    """A second implementation (one global ranking, quota pass then fill pass) on larger cases."""
    rng = np.random.default_rng(22)
    for _ in range(200):
        n_ch = int(rng.integers(2, 60))
        lens = rng.integers(1, 40, size=n_ch)
        tc = np.repeat(np.arange(n_ch, dtype=np.int32), lens)
        sc = rng.exponential(size=n_ch).astype(np.float32)
        sc[rng.integers(0, n_ch, size=5)] = sc[1]
        T = len(tc)
        n_s = int(rng.integers(0, 5))
        n_w = int(rng.integers(0, 50))
        M = int(rng.integers(n_s + n_w + 1, max(T, n_s + n_w + 1) + 5))
        N = int(rng.integers(0, 9))
        idx, _ = oracle.select_retain(M, n_s, n_w, N, tc, sc)
        assert idx.tolist() == select_by_global_sort(M, n_s, n_w, N, tc, sc)


def test_select_single_span_is_stable_top_m():
    """N = 1, no sink or window: plain top-M by score with earlier slots first on ties."""
    rng = np.random.default_rng(23)
    for _ in range(50):
        n_ch = int(rng.integers(2, 30))
        tc = np.repeat(np.arange(n_ch, dtype=np.int32), rng.integers(1, 20, size=n_ch))
        sc = np.round(rng.exponential(size=n_ch), 1).astype(np.float32)   # many ties
        M = int(rng.integers(1, len(tc) + 3))
        idx, _ = oracle.select_retain(M, 0, 0, 1, tc, sc)
        order = sorted(range(len(tc)), key=lambda i: -float(sc[tc[i]]))   # Python's sort is stable
        assert idx.tolist() == sorted(order[:M])


def test_select_invariants():
    """Budget never exceeded, sink and window kept, stream order, per-span minimum met, and no
    dropped candidate outranks a kept one of the same span beyond the quota."""
    rng = np.random.default_rng(24)
    for _ in range(200):
        n_ch = int(rng.integers(2, 40))
        tc = np.repeat(np.arange(n_ch, dtype=np.int32), rng.integers(1, 30, size=n_ch))
        sc = rng.exponential(size=n_ch).astype(np.float32)
        T = len(tc)
        n_s = int(rng.integers(0, 6))
        n_w = int(rng.integers(0, 40))
        M = int(rng.integers(n_s + n_w + 1, max(T, n_s + n_w + 1) + 5))
        N = int(rng.integers(1, 7))
        idx, mask = oracle.select_retain(M, n_s, n_w, N, tc, sc)
        assert len(idx) == min(T, M)
        assert np.all(np.diff(idx) > 0)
        assert mask.sum() == len(idx) and np.all(mask[idx] == 1)
        if T <= M:
            continue
        assert np.all(mask[:n_s] == 1) and np.all(mask[T - n_w:] == 1)
        lo, hi = n_s, T - n_w
        a = tc[lo:hi].astype(np.int64)
        span = ((a - a.min()) * N) // (a.max() - a.min() + 1)
        q = (M - n_s - n_w) // N
        for j in range(N):
            members = np.nonzero(span == j)[0] + lo
            assert mask[members].sum() >= min(q, len(members))


def test_select_spans_follow_arrival_time_not_slots():
    """Spans split arrival time, not cache slots (Sec. 3.3): after an eviction has removed most of
    the early chunks, the remaining few early tokens still form their own span."""
    tok_chunk = np.array([0, 5, 10, 11, 12, 13, 14, 15, 16, 17, 18, 19], np.int32)
    scores = np.zeros(20, np.float32)
    scores[10:] = 1.0      # later chunks score higher
    idx, _ = oracle.select_retain(4, 0, 0, 2, tok_chunk, scores)
    # span 0 = chunks 0..9 (slots 0,1), span 1 = chunks 10..19; quota 2 each
    assert idx.tolist() == [0, 1, 2, 3]


def test_select_rejects_bad_arguments():
    with pytest.raises(ValueError):
        oracle.select_retain(4, 2, 2, 1, [0, 0, 0, 0, 0, 0], [1.0])       # M < n_s + n_w + 1
    with pytest.raises(ValueError):
        oracle.select_retain(2, 0, 0, 1, [0, 1, 5], [1.0, 2.0])           # chunk id out of range


# ---------------------------------------------------------------- compaction (Alg. 1, Sec. 3.3)

def test_compaction_is_index_gather():
    """out[j] = in[retain[j]] for j < n, rows past n untouched (numpy.take as the reference)."""
    rng = np.random.default_rng(31)
    planes = rng.standard_normal((6, 50, 7)).astype(np.float32)
    keep = np.sort(rng.choice(40, size=23, replace=False)).astype(np.int32)
    out = oracle.compact_rows(planes, keep, 40)
    np.testing.assert_array_equal(out[:, :23], np.take(planes, keep, axis=1))
    np.testing.assert_array_equal(out[:, 23:], planes[:, 23:])


def test_compaction_keeps_original_positions():
    """Survivors keep their original position ids (Sec. 3.3: no re-numbering, no re-rotation)."""
    cap = 16
    kc = np.arange(2 * 1 * cap * 4, dtype=np.float32).reshape(2, 1, cap, 4)
    tc = np.arange(cap, dtype=np.int32) // 4
    tp = np.arange(100, 100 + cap, dtype=np.int32)
    keep = np.array([0, 1, 6, 7, 12], np.int32)
    k2, v2, tc2, tp2 = oracle.compact_kv(kc, kc.copy(), tc, tp, keep, 14)
    assert tp2[:5].tolist() == [100, 101, 106, 107, 112]
    assert tc2[:5].tolist() == [0, 0, 1, 1, 3]
    np.testing.assert_array_equal(k2[:, :, :5], kc[:, :, keep])


# ---------------------------------------------------------------- Alg. 1 loop

def test_stream_loop_invariants_tiny():
    """Alg. 1 on the tiny workload: first chunk from a zero state scores +inf, the cache never
    exceeds M after an eviction, positions stay in stream order, sink slots survive."""
    rng = np.random.default_rng(41)
    L, Hk, Hv, d, C, n_ch = 1, 2, 2, 16, 64, 8
    chunks = [_rand_inputs(rng, L, C, Hk, Hv, d) for _ in range(n_ch)]
    kvs = [(rng.standard_normal((1, 2, C, 16)).astype(np.float32),
            rng.standard_normal((1, 2, C, 16)).astype(np.float32)) for _ in range(n_ch)]
    policy = dict(budget_M=256, n_sink=4, n_window=64, n_buckets=2)
    res = run_stream(lambda c: chunks[c], lambda c: kvs[c], np.zeros((L, Hv, d, d)), n_ch, policy,
                     capacity=256 + C)
    assert np.isinf(res.chunk_scores[0]) and np.all(np.isfinite(res.chunk_scores[1:]))
    assert res.cache_len == 256 and len(res.evictions) == n_ch - 4
    pos = res.tok_pos[: res.cache_len]
    assert np.all(np.diff(pos) > 0) and pos[:4].tolist() == [0, 1, 2, 3]
    assert pos[-64:].tolist() == list(range(n_ch * C - 64, n_ch * C))


def test_question_turn_leaves_stream_unchanged():
    """Sec. 3.3: a question saved-and-restored around changes nothing later chunks see.  The
    question (one chunk of other tokens) does run: it moves the state and, with the cache at its
    budget, forces an eviction; after the restore the stream equals a run without it, exactly."""
    rng = np.random.default_rng(43)
    L, Hk, Hv, d, C, n_ch = 1, 2, 2, 16, 64, 8
    chunks = [_rand_inputs(rng, L, C, Hk, Hv, d) for _ in range(n_ch)]
    kvs = [(rng.standard_normal((1, 2, C, 16)).astype(np.float32),
            rng.standard_normal((1, 2, C, 16)).astype(np.float32)) for _ in range(n_ch)]
    qin = _rand_inputs(rng, L, C, Hk, Hv, d)
    qkv = (rng.standard_normal((1, 2, C, 16)).astype(np.float32),
           rng.standard_normal((1, 2, C, 16)).astype(np.float32))
    policy = dict(budget_M=256, n_sink=4, n_window=64, n_buckets=2)
    s0 = np.zeros((L, Hv, d, d))
    plain = run_stream(lambda c: chunks[c], lambda c: kvs[c], s0, n_ch, policy, capacity=256 + C,
                       keep_states=True)
    asked = run_stream(lambda c: chunks[c], lambda c: kvs[c], s0, n_ch, policy, capacity=256 + C,
                       questions={5: lambda: (qin, qkv)})
    assert len(asked.question_states) == 1
    assert not np.allclose(asked.question_states[0], plain.states_after_chunk[4])
    assert len(asked.evictions) == len(plain.evictions)
    np.testing.assert_array_equal(asked.state, plain.state)
    np.testing.assert_array_equal(asked.chunk_scores, plain.chunk_scores)
    assert asked.cache_len == plain.cache_len
    for name in ("k_cache", "v_cache", "tok_chunk", "tok_pos"):
        np.testing.assert_array_equal(getattr(asked, name), getattr(plain, name))
    for (c1, i1), (c2, i2) in zip(asked.evictions, plain.evictions):
        assert c1 == c2
        np.testing.assert_array_equal(i1, i2)



# ---------------------------------------------------------------- token signals (Sec. 4.3)

def test_row_norm_scores_are_signed_l2_norms():
    """Key norm scores -||k||_2, value norm ||v||_2 (the appendix's table of signals): equal to
    numpy.linalg.norm on random rows (bf16-rounded values included), sqrt(D) for a row of ones,
    |x| for a one-hot row, and |lambda| times the score for a scaled row."""
    rng = np.random.default_rng(71)
    rows = rng.standard_normal((3, 5, 256)).astype(np.float32)
    bf = ((rows.view(np.uint32) + 0x8000) & 0xFFFF0000).view(np.float32)      # bf16 values
    for r in (rows, bf):
        ref = np.linalg.norm(r.astype(np.float64), axis=-1)
        np.testing.assert_allclose(oracle.row_norm_scores(r, "value_norm"), ref, rtol=1e-7)
        np.testing.assert_allclose(oracle.row_norm_scores(r, "key_norm"), -ref, rtol=1e-7)
    assert oracle.row_norm_scores(np.ones((1, 256), np.float32), "value_norm")[0] == 16.0
    hot = np.zeros((1, 16), np.float32)
    hot[0, 5] = -3.5
    assert oracle.row_norm_scores(hot, "key_norm")[0] == -3.5
    assert oracle.row_norm_scores(hot, "value_norm")[0] == 3.5
    np.testing.assert_allclose(oracle.row_norm_scores(4.0 * rows, "value_norm"),
                               4.0 * oracle.row_norm_scores(rows, "value_norm"), rtol=1e-7)
    with pytest.raises(ValueError):
        oracle.row_norm_scores(rows, "attention")


def _random_token_case(rng, T_max, ties=True):
    M, n_s, n_w, N, tc, _ = _random_case(rng, T_max, ties=False)
    sc = rng.standard_normal(len(tc)).astype(np.float32)
    if ties and len(tc) > 3:
        sc[rng.integers(0, len(tc), size=3)] = sc[0]
    return M, n_s, n_w, N, tc, sc


def test_select_tokens_equals_chunk_selection_on_shared_scores():
    """With every token carrying its chunk's score, the token-level selection is the Sec. 3.3
    chunk selection (pinned above)."""
    rng = np.random.default_rng(72)
    for _ in range(300):
        n_ch = int(rng.integers(2, 40))
        tc = np.repeat(np.arange(n_ch, dtype=np.int32), rng.integers(1, 25, size=n_ch))
        sc = rng.exponential(size=n_ch).astype(np.float32)
        sc[rng.integers(0, n_ch, size=4)] = sc[0]
        T = len(tc)
        n_s, n_w = int(rng.integers(0, 5)), int(rng.integers(0, 30))
        M = int(rng.integers(n_s + n_w + 1, max(T, n_s + n_w + 1) + 5))
        N = int(rng.integers(0, 7))
        a = oracle.select_retain(M, n_s, n_w, N, tc, sc)
        b = oracle.select_retain_tokens(M, n_s, n_w, N, tc, sc[tc])
        np.testing.assert_array_equal(a[0], b[0])
        np.testing.assert_array_equal(a[1], b[1])


def test_select_tokens_matches_exhaustive_max_weight():
    """Per-token scores: quota-then-fill == the max-weight subset under the span lower bounds
    (exhaustive over all subsets, T <= 12)."""
    rng = np.random.default_rng(73)
    n = 0
    while n < 300:
        M, n_s, n_w, N, tc, sc = _random_token_case(rng, 12)
        if len(tc) <= M:
            continue
        idx, _ = oracle.select_retain_tokens(M, n_s, n_w, N, tc, sc)
        assert idx.tolist() == select_by_max_weight(M, n_s, n_w, N, tc, sc, per_slot=True)
        n += 1


def test_select_tokens_matches_global_sort_implementation():
    rng = np.random.default_rng(74)
    for _ in range(200):
        n_ch = int(rng.integers(2, 60))
        tc = np.repeat(np.arange(n_ch, dtype=np.int32), rng.integers(1, 40, size=n_ch))
        T = len(tc)
        sc = np.round(rng.standard_normal(T), 2).astype(np.float32)             # many exact ties
        sc[rng.integers(0, T, size=3)] = -0.0
        n_s, n_w = int(rng.integers(0, 5)), int(rng.integers(0, 50))
        M = int(rng.integers(n_s + n_w + 1, max(T, n_s + n_w + 1) + 5))
        N = int(rng.integers(0, 9))
        idx, _ = oracle.select_retain_tokens(M, n_s, n_w, N, tc, sc)
        assert idx.tolist() == select_by_global_sort(M, n_s, n_w, N, tc, sc, per_slot=True)


def test_select_tokens_single_span_is_stable_top_m():
    """N = 1, no sink or window: the M best tokens by score, earlier slot first on ties
    (numpy's stable argsort as the reference)."""
    rng = np.random.default_rng(75)
    for _ in range(50):
        T = int(rng.integers(2, 300))
        tc = np.sort(rng.integers(0, 20, size=T)).astype(np.int32)
        sc = np.round(rng.standard_normal(T), 1).astype(np.float32)
        M = int(rng.integers(1, T + 3))
        idx, _ = oracle.select_retain_tokens(M, 0, 0, 1, tc, sc)
        order = np.argsort(-sc.astype(np.float64), kind="stable")
        assert idx.tolist() == sorted(order[:M].tolist())


def test_select_tokens_invariants():
    """Budget, sink and window, stream order, per-span minimum, and inside every span the kept
    candidates are the best ones of that span (quota and fill both take from the top)."""
    rng = np.random.default_rng(76)
    for _ in range(200):
        n_ch = int(rng.integers(2, 40))
        tc = np.repeat(np.arange(n_ch, dtype=np.int32), rng.integers(1, 30, size=n_ch))
        T = len(tc)
        sc = rng.standard_normal(T).astype(np.float32)
        n_s, n_w = int(rng.integers(0, 6)), int(rng.integers(0, 40))
        M = int(rng.integers(n_s + n_w + 1, max(T, n_s + n_w + 1) + 5))
        N = int(rng.integers(1, 7))
        idx, mask = oracle.select_retain_tokens(M, n_s, n_w, N, tc, sc)
        assert len(idx) == min(T, M) and np.all(np.diff(idx) > 0)
        if T <= M:
            continue
        assert np.all(mask[:n_s] == 1) and np.all(mask[T - n_w:] == 1)
        lo, hi = n_s, T - n_w
        a = tc[lo:hi].astype(np.int64)
        span = ((a - a.min()) * N) // (a.max() - a.min() + 1)
        q = (M - n_s - n_w) // N
        for j in range(N):
            members = np.nonzero(span == j)[0] + lo
            kept = members[mask[members] == 1]
            dropped = members[mask[members] == 0]
            assert len(kept) >= min(q, len(members))
            if len(kept) and len(dropped):
                assert sc[kept].min() >= sc[dropped].max()


def test_compact_heads_gathers_each_plane_by_its_own_list():
    """Per-head gather: plane p of K, V and of the per-head metadata equals numpy.take by list p;
    rows past the kept length are untouched."""
    rng = np.random.default_rng(77)
    Lf, Hkv, cap, D, T, n = 2, 3, 40, 8, 33, 20
    kc = rng.standard_normal((Lf, Hkv, cap, D)).astype(np.float32)
    vc = rng.standard_normal((Lf, Hkv, cap, D)).astype(np.float32)
    tc = rng.integers(0, 9, size=(Lf, Hkv, cap)).astype(np.int32)
    tp = rng.integers(0, 999, size=(Lf, Hkv, cap)).astype(np.int32)
    ts = rng.standard_normal((Lf, Hkv, cap)).astype(np.float32)
    lists = [np.sort(rng.choice(T, size=n, replace=False)).astype(np.int32) for _ in range(Lf * Hkv)]
    out = oracle.compact_kv_heads(kc, vc, tc, tp, ts, lists, T)
    for arr, o in zip((kc, vc, tc, tp, ts), out):
        for p in range(Lf * Hkv):
            l, h = divmod(p, Hkv)
            np.testing.assert_array_equal(o[l, h, :n], np.take(arr[l, h], lists[p], axis=0))
            np.testing.assert_array_equal(o[l, h, n:], arr[l, h, n:])


@pytest.mark.parametrize("signal", ["key_norm", "value_norm"])
def test_stream_heads_invariants_tiny(signal):
    """The per-head loop: every plane keeps M tokens with sinks and window, in stream order; the
    stored score of every kept token equals its signal recomputed from the cache row it now sits
    in (the score is a function of the row alone); planes disagree on what they keep."""
    rng = np.random.default_rng(78)
    Lf, Hkv, C, D, n_ch = 1, 2, 64, 16, 8
    kvs = [(rng.standard_normal((Lf, Hkv, C, D)).astype(np.float32),
            rng.standard_normal((Lf, Hkv, C, D)).astype(np.float32)) for _ in range(n_ch)]
    policy = dict(budget_M=256, n_sink=4, n_window=64, n_buckets=2)
    res = run_stream_heads(lambda c: kvs[c], n_ch, policy, capacity=256 + C, signal=signal)
    n = res.cache_len
    assert n == 256 and len(res.evictions) == n_ch - 4
    rows = res.k_cache if signal == "key_norm" else res.v_cache
    np.testing.assert_array_equal(res.tok_score[:, :, :n], oracle.row_norm_scores(rows[:, :, :n], signal))
    for h in range(Hkv):
        pos = res.tok_pos[0, h, :n]
        assert np.all(np.diff(pos) > 0) and pos[:4].tolist() == [0, 1, 2, 3]
        assert pos[-64:].tolist() == list(range(n_ch * C - 64, n_ch * C))
        np.testing.assert_array_equal(res.tok_chunk[0, h, :n], pos // C)
    assert not np.array_equal(res.tok_pos[0, 0, :n], res.tok_pos[0, 1, :n])
