"""GPU parity of the gated-delta chunk update + fused drift partials (Sec. 3.2, Eq. 1-3) and of
the standalone drift / score kernels, against the fp64 CPU oracle on the same seeded inputs.

Tolerances (floating point):
* state: relative Frobenius error <= 2e-3 per (layer, head) at every chunk boundary;
* drift partials: relative error <= 1e-3 on sum (S_after - S_before)^2 and sum S_before^2;
* read-out o: relative Frobenius error per (layer, head) <= 2e-3 (+ bfloat16 output rounding,
  2^-8 relative, when the activations are bfloat16);
* chunk score: |Delta| / |ref| <= 1e-3, and +inf must match +inf.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_27470_gb300 import inputs

pytestmark = pytest.mark.gpu

STATE_TOL = 2e-3


@pytest.fixture(scope="module")
def L():
    from paper_2609_27470_gb300 import _lib
    return _lib


def _f64(t):
    return t.detach().float().cpu().double().numpy()


def _per_head_rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    axes = tuple(range(2, a.ndim))
    num = np.sqrt(np.sum((a - b) ** 2, axis=axes))
    den = np.sqrt(np.sum(b ** 2, axis=axes))
    return num / np.maximum(den, 1e-30)


def _run_gpu(L, x, state, want_out, dtype, q_scale):
    Lg, T, Hk, d = x["k"].shape
    Hv = x["v"].shape[2]
    desc = L.gdn_desc(Lg, Hk, Hv, d, dtype, q_scale)
    dev = torch.device("cuda")
    xs = {k: v.to(dev) for k, v in x.items()}
    st = state.to(dev).clone()
    out = torch.empty(Lg, T, Hv, d, dtype=dtype, device=dev) if want_out else None
    part = torch.full((Lg, Hv, 2), -1.0, device=dev)
    size = (L.deltas_gdn_chunk_update_readout_workspace_size if want_out else
            L.deltas_gdn_chunk_update_workspace_size)(desc, T)
    ws = L.alloc_workspace(size, dev)
    L.deltas_gdn_chunk_update(desc, T, xs["q"] if want_out else None, xs["k"], xs["v"], xs["g"], xs["beta"],
                              st, out, part, ws)
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(ws) == (0, 0)
    return st, out, part


def _check_chunk(L, x, state0, want_out, dtype, q_scale):
    st, out, part = _run_gpu(L, x, state0, want_out, dtype, q_scale)
    S_ref, o_ref = oracle.gdn_recurrence(_f64(x["q"]), _f64(x["k"]), _f64(x["v"]), _f64(x["g"]), _f64(x["beta"]),
                                         _f64(state0), q_scale=q_scale, want_out=want_out)
    rel = _per_head_rel(_f64(st), S_ref)
    assert rel.max() <= STATE_TOL, f"state rel err {rel.max():.3e}"
    p_ref = oracle.drift_partials(_f64(state0), S_ref)
    p = _f64(part)
    np.testing.assert_allclose(p[..., 1], p_ref[..., 1], rtol=1e-5, atol=0)
    np.testing.assert_allclose(p[..., 0], p_ref[..., 0], rtol=1e-3, atol=1e-30)
    if want_out:
        tol = STATE_TOL + (2.0 ** -8 if dtype == torch.bfloat16 else 0.0)
        o = _f64(out).transpose(0, 2, 1, 3)            # [L,Hv,T,d] per (layer, head)
        orl = _per_head_rel(o, o_ref.transpose(0, 2, 1, 3))
        assert orl.max() <= tol, f"out rel err {orl.max():.3e}"
    return st, rel.max()


@pytest.mark.parametrize("d", [16, 32, 64, 128])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("T", [1, 63, 64, 100, 257])
@pytest.mark.parametrize("want_out", [True, False])
def test_gdn_update_shapes(L, d, dtype, T, want_out):
    """Every head size, both activation dtypes, ragged token counts (one token, a tile minus one,
    exactly one tile, several tiles with a ragged tail), grouped keys (Hk=2, Hv=4), two layers,
    with and without the read-out (d = 128 bf16 runs on the tensor cores, the read-out there in a
    third kernel over 128-token blocks: T = 100 and 257 end inside a block's second tile)."""
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    x = inputs.gdn_chunk(2, T, 2, 4, d, dtype, inputs.seed_for(1, d, T))
    s0 = inputs.initial_state(2, 4, d, inputs.seed_for(2, d, T))
    _check_chunk(L, x, s0, want_out, tdt, d ** -0.5)


def test_gdn_update_tiny_stream_from_zero(L):
    """Tiny workload: 8 chunks x 64 tokens, d = 16, fp32, zero start state; every chunk boundary
    is compared against the oracle replaying that chunk from the GPU's own S_before, and the
    final state against the oracle's own trajectory."""
    Lg, Hk, Hv, d, C = 1, 2, 2, 16, 64
    state = torch.zeros(Lg, Hv, d, d)
    ref = np.zeros((Lg, Hv, d, d))
    for c in range(8):
        x = inputs.gdn_chunk(Lg, C, Hk, Hv, d, "f32", inputs.seed_for(0, 0, c))
        st, _ = _check_chunk(L, x, state, False, torch.float32, 0.25)
        ref, _ = oracle.gdn_recurrence(None, _f64(x["k"]), _f64(x["v"]), _f64(x["g"]), _f64(x["beta"]), ref)
        state = st.cpu()
    assert _per_head_rel(state.double().numpy(), ref).max() <= STATE_TOL


def test_gdn_update_zero_tokens(L):
    """n_tokens = 0: the state is unchanged, partials are (0, ||S_before||^2)."""
    s0 = inputs.initial_state(1, 4, 64, 5)
    x = inputs.gdn_chunk(1, 0, 2, 4, 64, "bf16", 6)
    st, _, part = _run_gpu(L, x, s0, False, torch.bfloat16, 0.125)
    assert torch.equal(st.cpu(), s0)
    p = part.cpu().double().numpy()
    assert np.all(p[..., 0] == 0)
    np.testing.assert_allclose(p[..., 1], np.sum(s0.double().numpy() ** 2, axis=(2, 3)), rtol=1e-5)


@pytest.mark.parametrize("want_out", [True, False])
def test_gdn_update_layer_width_chunk(L, want_out):
    """The single-layer workload's shape: 16 key heads, 32 value heads, d = 128, bf16, one chunk
    of 1024 tokens (spans many tiles), with and without read-out."""
    x = inputs.gdn_chunk(1, 1024, 16, 32, 128, "bf16", inputs.seed_for(7, 1, 0))
    s0 = inputs.initial_state(1, 32, 128, 8)
    _check_chunk(L, x, s0, want_out, torch.bfloat16, 128 ** -0.5)


@pytest.mark.parametrize("T,want_out", [(1, False), (130, False), (500, False), (130, True), (500, True)])
def test_gdn_update_more_heads_than_sms(L, T, want_out):
    """160 (layer, head) pairs (5 layers x 32 value heads, d = 128, bf16): more heads than SMs, so
    the tensor-core kernel's persistent CTAs take equal runs of tiles and most heads are split
    between two neighbouring CTAs (the state handed over at the cut); every head's state and drift
    partials are compared with the oracle (one tile, and three tiles with a ragged tail), and with
    the read-out every output (a cut may fall inside a 128-token read-out block, whose starting
    state and writes then come from two CTAs)."""
    x = inputs.gdn_chunk(5, T, 16, 32, 128, "bf16", inputs.seed_for(12, T))
    s0 = inputs.initial_state(5, 32, 128, inputs.seed_for(13, T))
    _check_chunk(L, x, s0, want_out, torch.bfloat16, 128 ** -0.5)


@pytest.mark.parametrize("want_out", [False, True])
def test_gdn_update_stack_width_sampled(L, want_out):
    """The full stack's width (24 layers x 32 value heads, d = 128, bf16, one 1024-token chunk)
    in the launch configuration the benchmark times, with and without the read-out; the oracle
    checks a sample of 12 (layer, head) pairs, each replayed from the same S_before."""
    Lg, Hk, Hv, d, T = 24, 16, 32, 128, 1024
    qs = 128 ** -0.5
    x = inputs.gdn_chunk(Lg, T, Hk, Hv, d, "bf16", inputs.seed_for(8, 2, 0))
    s0 = inputs.initial_state(Lg, Hv, d, 10)
    st, out, part = _run_gpu(L, x, s0, want_out, torch.bfloat16, qs)
    rng = np.random.default_rng(3)
    pairs = [(0, 0), (Lg - 1, Hv - 1)] + [(int(rng.integers(Lg)), int(rng.integers(Hv))) for _ in range(10)]
    for (l, h) in pairs:
        kh = h * Hk // Hv
        sub = {k: x[k][l:l + 1] for k in ("q", "k", "v", "g", "beta")}
        S_ref, o_ref = oracle.gdn_recurrence(_f64(sub["q"][:, :, kh:kh + 1]), _f64(sub["k"][:, :, kh:kh + 1]),
                                             _f64(sub["v"][:, :, h:h + 1]), _f64(sub["g"][:, :, h:h + 1]),
                                             _f64(sub["beta"][:, :, h:h + 1]), _f64(s0[l:l + 1, h:h + 1]),
                                             q_scale=qs, want_out=want_out)
        rel = _per_head_rel(_f64(st[l:l + 1, h:h + 1]), S_ref).max()
        assert rel <= STATE_TOL, (l, h, rel)
        if want_out:
            o = _f64(out[l:l + 1, :, h:h + 1]).transpose(0, 2, 1, 3)
            orl = _per_head_rel(o, o_ref.transpose(0, 2, 1, 3)).max()
            assert orl <= STATE_TOL + 2.0 ** -8, (l, h, orl)
        p_ref = oracle.drift_partials(_f64(s0[l:l + 1, h:h + 1]), S_ref)[0, 0]
        np.testing.assert_allclose(_f64(part[l, h]), p_ref, rtol=1e-3)
    # every head moved and no head was left untouched or non-finite
    assert torch.isfinite(st).all() and (part[..., 0] > 0).all()


def test_gdn_update_slow_decay_four_chunks(L):
    """Heads with long memory (alpha close to 1) keep errors from decaying away: 4 chunks of 1024
    tokens, compared at every chunk boundary with the oracle's own trajectory."""
    Lg, Hk, Hv, d = 1, 2, 4, 128
    state = inputs.initial_state(Lg, Hv, d, 9)
    ref = state.double().numpy()
    for c in range(4):
        x = inputs.gdn_chunk(Lg, 1024, Hk, Hv, d, "bf16", inputs.seed_for(9, c), decay_scale=0.002)
        st, _, _ = _run_gpu(L, x, state, False, torch.bfloat16, None)
        ref, _ = oracle.gdn_recurrence(None, _f64(x["k"]), _f64(x["v"]), _f64(x["g"]), _f64(x["beta"]), ref)
        rel = _per_head_rel(_f64(st), ref)
        assert rel.max() <= STATE_TOL, f"chunk {c}: {rel.max():.3e}"
        state = st.cpu()


@pytest.mark.parametrize("Hk,Hv", [(2, 6), (4, 4)])
def test_gdn_update_other_head_groupings(L, Hk, Hv):
    """Key heads serving three value heads and one value head each (the other cases share a key
    head between two): the key-head index of every value head, several tiles and a ragged tail,
    two layers."""
    x = inputs.gdn_chunk(2, 257, Hk, Hv, 128, "bf16", inputs.seed_for(15, Hk, Hv))
    state0 = inputs.initial_state(2, Hv, 128, 16)
    _check_chunk(L, x, state0, False, torch.bfloat16, None)
    _check_chunk(L, x, state0, True, torch.bfloat16, 0.3)


@pytest.mark.parametrize("decay_scale", [0.0, 4.0])
def test_gdn_update_decay_extremes(L, decay_scale):
    """No decay (g = 0: alpha = 1, the deferred decay never moves) and very strong decay (a tile's
    cumulative log-decay spans more than 250 powers of two, so the factors take the per-entry
    exponential, and gamma_C underflows, so every tile rescales the state): state and partials
    against the oracle over four tiles and a ragged tail."""
    Lg, Hk, Hv, d = 1, 2, 4, 128
    x = inputs.gdn_chunk(Lg, 300, Hk, Hv, d, "bf16", inputs.seed_for(13, int(decay_scale)), decay_scale=decay_scale)
    g = x["g"].double()
    if decay_scale > 0:                                 # the regimes this case is meant to reach
        span = (g[:, 64:128].sum(dim=1) / np.log(2)).abs()
        assert (span > 250).any()
    else:
        assert (g == 0).all()
    state0 = inputs.initial_state(Lg, Hv, d, 14)
    _check_chunk(L, x, state0, False, torch.bfloat16, None)
    # the read-out: a block's outputs weigh each earlier write of the block by exp(G_t - G_i) and
    # its starting state by exp(G_t), both far below the fp32 range here for most pairs
    _check_chunk(L, x, state0, True, torch.bfloat16, 0.2)


def test_state_drift_kernel(L):
    """deltas_state_drift partials == oracle (Eq. 3 numerator/denominator per layer and head)."""
    sb = inputs.initial_state(3, 4, 128, 11)
    sa = sb * 0.9 + 0.05 * inputs.initial_state(3, 4, 128, 12)
    desc = L.gdn_desc(3, 4, 4, 128, torch.bfloat16)
    part = torch.zeros(3, 4, 2, device="cuda")
    ws = L.alloc_workspace(L.deltas_state_drift_workspace_size(desc))
    L.deltas_state_drift(desc, sb.cuda(), sa.cuda(), part, ws)
    p_ref = oracle.drift_partials(sb.double().numpy(), sa.double().numpy())
    np.testing.assert_allclose(part.cpu().double().numpy(), p_ref, rtol=1e-5)


def test_score_kernel(L):
    """deltas_score_chunks == oracle Eq. 3 on the same float32 partials, incl. the zero-norm
    reading (0/0 -> 0, x/0 -> inf)."""
    rng = np.random.default_rng(13)
    scores = torch.zeros(8, device="cuda")
    for cid, (Lg, Hv) in enumerate([(1, 1), (3, 4), (24, 32), (5, 100)]):
        p = rng.exponential(size=(Lg, Hv, 2)).astype(np.float32)
        L.deltas_score_chunks(Lg, Hv, torch.from_numpy(p).cuda(), cid, scores)
        ref = oracle.chunk_score(p.astype(np.float64))
        assert abs(scores[cid].item() - ref) <= 1e-6 * abs(ref)
    z = np.zeros((2, 3, 2), np.float32)
    L.deltas_score_chunks(2, 3, torch.from_numpy(z).cuda(), 5, scores)
    assert scores[5].item() == 0.0
    z[1, 2, 0] = 1e-3
    L.deltas_score_chunks(2, 3, torch.from_numpy(z).cuda(), 6, scores)
    assert scores[6].item() == float("inf") and oracle.chunk_score(z.astype(np.float64)) == float("inf")


# ---------------------------------------------------------------- write sizes (Sec. 4.3 comparison signal)

@pytest.mark.parametrize("d,dtype,T,Hk,Hv,decay", [
    (128, "bf16", 257, 2, 4, 1.0),      # tensor cores: several tiles, ragged tail, grouped keys
    (128, "bf16", 64, 1, 3, 1.0),       # one full tile, three value heads per key head
    (128, "bf16", 300, 2, 4, 4.0),      # strong decay: the deferred decay restarts every tile
    (128, "bf16", 300, 16, 80, 1.0),    # 160 heads on fewer SMs: heads split between CTAs
    (64, "f32", 100, 2, 4, 1.0),        # CUDA-core kernel
    (16, "bf16", 33, 1, 2, 1.0),
    (128, "f32", 1, 2, 2, 1.0),
])
def test_write_norms_match_oracle(L, d, dtype, T, Hk, Hv, decay):
    """Per (layer, head) sums over the chunk of beta_t ||v_t - alpha_t S_{t-1} k_t|| against the
    oracle's token loop (relative 1e-3, the drift tolerance); asking for them changes neither the
    state nor the drift partials, bit for bit."""
    x = inputs.gdn_chunk(2, T, Hk, Hv, d, dtype, inputs.seed_for(70, d, T))
    if decay != 1.0:
        x["g"] = x["g"] * decay
    s0 = inputs.initial_state(2, Hv, d, inputs.seed_for(71, d, T))
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    dev = torch.device("cuda")
    desc = L.gdn_desc(2, Hk, Hv, d, tdt, None)
    xs = {k: v.to(dev) for k, v in x.items()}
    ws = L.alloc_workspace(L.deltas_gdn_chunk_update_workspace_size(desc, T), dev)
    runs = []
    for want in (False, True):
        st = s0.to(dev).clone()
        part = torch.full((2, Hv, 2), -1.0, device=dev)
        wn = torch.full((2, Hv), -1.0, device=dev) if want else None
        L.deltas_gdn_chunk_update(desc, T, None, xs["k"], xs["v"], xs["g"], xs["beta"], st, None, part, ws,
                                  write_norms=wn)
        torch.cuda.synchronize()
        assert L.deltas_get_device_status(ws) == (0, 0)
        runs.append((st, part, wn))
    assert torch.equal(runs[0][0].view(torch.int32), runs[1][0].view(torch.int32))
    assert torch.equal(runs[0][1].view(torch.int32), runs[1][1].view(torch.int32))
    _, _, wn_ref = oracle.gdn_recurrence(None, _f64(x["k"]), _f64(x["v"]), _f64(x["g"]), _f64(x["beta"]), _f64(s0),
                                         want_write_norms=True)
    assert np.all(wn_ref > 0)
    np.testing.assert_allclose(_f64(runs[1][2]), wn_ref, rtol=1e-3, atol=0)


def test_write_norms_zero_tokens(L):
    dev = torch.device("cuda")
    desc = L.gdn_desc(1, 2, 2, 128, torch.bfloat16, None)
    st = torch.ones(1, 2, 128, 128, device=dev)
    wn = torch.full((1, 2), -1.0, device=dev)
    ws = L.alloc_workspace(L.deltas_gdn_chunk_update_workspace_size(desc, 0), dev)
    L.deltas_gdn_chunk_update(desc, 0, None, None, None, None, None, st, None, None, ws, write_norms=wn)
    torch.cuda.synchronize()
    assert torch.all(wn == 0)


def test_write_norm_score(L):
    """Chunk score of the comparison signal: the mean over heads, layers and tokens, as the oracle
    computes it from the same float32 sums."""
    dev = torch.device("cuda")
    rng = np.random.default_rng(72)
    wn = rng.exponential(size=(24, 32)).astype(np.float32)
    scores = torch.full((10,), -1.0, device=dev)
    L.deltas_score_write_norms(24, 32, torch.from_numpy(wn).to(dev), 125, 7, scores)
    L.deltas_score_write_norms(24, 32, torch.from_numpy(wn).to(dev), 0, 8, scores)
    torch.cuda.synchronize()
    sc = scores.cpu().numpy()
    assert sc[7] == pytest.approx(oracle.write_norm_score(wn.astype(np.float64), 125), rel=1e-6)
    assert sc[8] == 0.0 and sc[6] == -1.0


# ---------------------------------------------------------------- read-out on the tensor cores

def test_readout_needs_its_workspace(L):
    """A d = 128 bfloat16 call with out != NULL runs the read-out kernel, which keeps each token's
    write and the block states in the workspace: the plain workspace size is refused (WORKSPACE),
    the read-out size is accepted, and the outputs match the oracle."""
    Lg, Hk, Hv, d, T = 1, 2, 4, 128, 200
    dev = torch.device("cuda")
    desc = L.gdn_desc(Lg, Hk, Hv, d, torch.bfloat16, 0.25)
    small = L.deltas_gdn_chunk_update_workspace_size(desc, T)
    big = L.deltas_gdn_chunk_update_readout_workspace_size(desc, T)
    assert big > small
    x = inputs.gdn_chunk(Lg, T, Hk, Hv, d, "bf16", inputs.seed_for(80, T))
    xs = {k: v.to(dev) for k, v in x.items()}
    st = torch.zeros(Lg, Hv, d, d, device=dev)
    out = torch.empty(Lg, T, Hv, d, dtype=torch.bfloat16, device=dev)
    with pytest.raises(L.DeltasError) as e:
        L.deltas_gdn_chunk_update(desc, T, xs["q"], xs["k"], xs["v"], xs["g"], xs["beta"], st, out, None,
                                  L.alloc_workspace(small, dev))
    assert e.value.status == L.DELTAS_ERR_WORKSPACE
    s0 = inputs.initial_state(Lg, Hv, d, 81)
    _check_chunk(L, x, s0, True, torch.bfloat16, 0.25)


@pytest.mark.parametrize("decay", [1.0, 4.0])
def test_readout_with_write_norms(L, decay):
    """The read-out and the write sizes in one call: outputs, state, drift partials and write
    sizes against the oracle (the read-out path applies each tile's row decays in the state
    chain instead of the factor records, so its state is checked on its own, not against the
    path without read-out)."""
    Lg, Hk, Hv, d, T = 2, 2, 4, 128, 300
    x = inputs.gdn_chunk(Lg, T, Hk, Hv, d, "bf16", inputs.seed_for(82, int(decay)))
    x["g"] = x["g"] * decay
    s0 = inputs.initial_state(Lg, Hv, d, 83)
    dev = torch.device("cuda")
    desc = L.gdn_desc(Lg, Hk, Hv, d, torch.bfloat16, 0.125)
    xs = {k: v.to(dev) for k, v in x.items()}
    st = s0.to(dev).clone()
    out = torch.empty(Lg, T, Hv, d, dtype=torch.bfloat16, device=dev)
    part = torch.full((Lg, Hv, 2), -1.0, device=dev)
    wn = torch.full((Lg, Hv), -1.0, device=dev)
    ws = L.alloc_workspace(L.deltas_gdn_chunk_update_readout_workspace_size(desc, T), dev)
    L.deltas_gdn_chunk_update(desc, T, xs["q"], xs["k"], xs["v"], xs["g"], xs["beta"], st, out, part, ws,
                              write_norms=wn)
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(ws) == (0, 0)
    S_ref, o_ref, wn_ref = oracle.gdn_recurrence(_f64(x["q"]), _f64(x["k"]), _f64(x["v"]), _f64(x["g"]),
                                                 _f64(x["beta"]), _f64(s0), q_scale=0.125, want_out=True,
                                                 want_write_norms=True)
    assert _per_head_rel(_f64(st), S_ref).max() <= STATE_TOL
    o = _f64(out).transpose(0, 2, 1, 3)
    assert _per_head_rel(o, o_ref.transpose(0, 2, 1, 3)).max() <= STATE_TOL + 2.0 ** -8
    p_ref = oracle.drift_partials(_f64(s0), S_ref)
    np.testing.assert_allclose(_f64(part)[..., 0], p_ref[..., 0], rtol=1e-3)
    np.testing.assert_allclose(_f64(part)[..., 1], p_ref[..., 1], rtol=1e-5)
    np.testing.assert_allclose(_f64(wn), wn_ref, rtol=1e-3, atol=0)


@pytest.mark.parametrize("T", [128, 129, 191, 192, 256])
def test_readout_block_boundaries(L, T):
    """Token counts at and around the read-out's 128-token blocks: a block that ends the chunk
    exactly, one token into the next block, a last block of one tile (its second half absent and
    zero-filled) and of two."""
    x = inputs.gdn_chunk(1, T, 2, 4, 128, "bf16", inputs.seed_for(84, T))
    s0 = inputs.initial_state(1, 4, 128, inputs.seed_for(85, T))
    _check_chunk(L, x, s0, True, torch.bfloat16, 128 ** -0.5)


def test_readout_zero_tokens(L):
    """n_tokens = 0 with an output buffer: nothing is written, the state is unchanged."""
    dev = torch.device("cuda")
    desc = L.gdn_desc(1, 2, 4, 128, torch.bfloat16, 0.25)
    s0 = inputs.initial_state(1, 4, 128, 86)
    st = s0.to(dev).clone()
    big = torch.full((1, 1, 4, 128), 7.0, dtype=torch.bfloat16, device=dev)   # zero-token views of it
    q = torch.zeros(1, 1, 2, 128, dtype=torch.bfloat16, device=dev)
    ws = L.alloc_workspace(L.deltas_gdn_chunk_update_readout_workspace_size(desc, 0), dev)
    L.deltas_gdn_chunk_update(desc, 0, q[:, :0], None, None, None, None, st, big[:, :0], None, ws)
    torch.cuda.synchronize()
    assert L.deltas_get_device_status(ws) == (0, 0)
    assert torch.equal(st.cpu(), s0) and bool((big == 7.0).all())


@pytest.mark.parametrize("Lg,Hk,Hv,T,decay", [
    (1, 2, 4, 1024, 0.1),     # 4 heads: two segments of 8 tiles (3 CTAs per head)
    (1, 4, 8, 1000, 0.1),     # 8 heads, a ragged last tile in the second segment
    (1, 1, 2, 512, 4.0),      # strong decay: the runs from I and from 0 restart their deferred decay
    (1, 1, 2, 1024, 0.0),     # no decay: the affine maps keep their full range
    (1, 16, 32, 512, 0.1),    # the single layer's heads, 8 tiles: two segments of 4
    (1, 16, 32, 449, 0.1),    # 8 tiles, the second segment ending in a one-token tile
    (2, 8, 16, 640, 0.1),     # two layers (the CTA groups span layers), 10 tiles
    (1, 25, 50, 512, 0.1),    # 50 heads: 150 CTAs, the most that fit on 152 SMs
    (1, 4, 4, 512, 0.1),      # one value head per key head
])
def test_gdn_update_segments(L, Lg, Hk, Hv, T, decay):
    """Few heads (at most a third of the SMs) and at least 8 tiles: the state chain runs each head's
    tiles as two segments, the second once from S = I with v = 0 and once from S = 0, and the
    combine forms S_after = S_0 A_1 + B_1 and the drift partials; state and partials against the
    oracle."""
    x = inputs.gdn_chunk(Lg, T, Hk, Hv, 128, "bf16", inputs.seed_for(89, T, Hv), decay_scale=decay)
    s0 = inputs.initial_state(Lg, Hv, 128, inputs.seed_for(90, T, Hv))
    _check_chunk(L, x, s0, False, torch.bfloat16, None)
