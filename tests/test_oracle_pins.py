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
from oracle.stream import run_stream
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
