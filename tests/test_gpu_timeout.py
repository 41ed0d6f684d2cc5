"""The bounded-wait path on the GPU: a wait that runs out records DELTAS_ERR_TIMEOUT in the
workspace's status word, the call returns, and the next call with the default budget is correct
(the compaction's waits, and the first wait of each of the update's kernels, after which every
other role of the kernel stops on the abort flag and drains).

No wait here is left without a limit and nothing faults: the test only shortens the budget of
the waits (deltas_set_wait_budget) so that they give up at their first check.  A compaction unit
whose staged rows have not landed by then gives up and raises the abort flag, so the call ends
with part of the cache moved (which units finished first is timing-dependent): after a device
error the caches' contents are unspecified, and the test restores them before the next call.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_27470_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    from paper_2609_27470_gb300 import _lib
    return _lib


def _np(t):
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.numpy()


def test_compact_wait_runs_out_then_recovers(L):
    Lf, Hkv, D, cap = 2, 2, 256, 8192
    kc, vc = inputs.kv_cache(Lf, Hkv, cap, D, "bf16", seed=31)
    tc = inputs.chunked_tok_chunk(8, 1024).numpy()
    sc = inputs.chunk_scores_with_ties(8, seed=5, tie_rank=3, n_ties=2).numpy()
    keep, _ = oracle.select_retain(4096, 4, 1024, 2, tc, sc)
    tp = np.arange(cap, dtype=np.int32) + 77
    desc = L.kv_desc(Lf, Hkv, D, torch.bfloat16, cap)
    dev = torch.device("cuda")
    k, v = kc.to(dev), vc.to(dev)
    t1, t2 = torch.from_numpy(tc.copy()).to(dev), torch.from_numpy(tp).to(dev)
    idx = torch.from_numpy(np.asarray(keep, np.int32)).to(dev)
    n = torch.tensor([len(keep)], dtype=torch.int32, device=dev)
    ws = L.alloc_workspace(L.deltas_compact_kv_workspace_size(desc, cap), dev)

    # 1 ns: every wait gives up at its first check; the call returns with the timeout recorded
    L.deltas_set_wait_budget(ws, 1)
    L.deltas_compact_kv(desc, k, v, t1, t2, idx, n, cap, ws)
    status, unit = L.deltas_get_device_status(ws)
    assert status == L.DELTAS_ERR_TIMEOUT and unit >= 0

    # clearing the status word also restores the default budget: the same call on the restored
    # inputs is correct
    L.deltas_clear_device_status(ws)
    k.copy_(kc); v.copy_(vc)
    t1.copy_(torch.from_numpy(tc)); t2.copy_(torch.from_numpy(tp))
    L.deltas_compact_kv(desc, k, v, t1, t2, idx, n, cap, ws)
    assert L.deltas_get_device_status(ws) == (0, 0)
    rk, rv, rtc, rtp = oracle.compact_kv(_np(kc), _np(vc), tc, tp, keep, cap)
    assert np.array_equal(_np(k.cpu()), rk) and np.array_equal(_np(v.cpu()), rv)
    assert np.array_equal(t1.cpu().numpy(), rtc) and np.array_equal(t2.cpu().numpy(), rtp)


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.max(np.sqrt(np.sum((a - b) ** 2, axis=(-2, -1)) / np.sum(b ** 2, axis=(-2, -1)))))


@pytest.mark.parametrize("want_out,T", [(False, 200), (True, 200), (False, 1024)])
def test_update_wait_runs_out_then_recovers(L, want_out, T):
    """The tensor-core update (d = 128 bf16: factor kernel, state chain and, with the read-out,
    the read-out kernel) with a 1 ns wait budget, which bounds each kernel's first wait: those
    waits give up, the other roles stop at their next wait (they see the abort flag), drain the
    copies and products they issued and free TMEM; the call ends with DELTAS_ERR_TIMEOUT
    recorded.  The same call with the default budget, from the restored state, then matches the
    oracle.  With 1024 tokens (16 tiles, 4 heads) the heads run as two segments on three CTAs, and
    the first-segment CTA's bounded waits for its siblings and for the combine product also stop
    on the abort."""
    Lg, Hk, Hv, d = 1, 2, 4, 128
    x = inputs.gdn_chunk(Lg, T, Hk, Hv, d, "bf16", inputs.seed_for(90, int(want_out)))
    s0 = inputs.initial_state(Lg, Hv, d, 91)
    dev = torch.device("cuda")
    desc = L.gdn_desc(Lg, Hk, Hv, d, torch.bfloat16, 0.25)
    size = (L.deltas_gdn_chunk_update_readout_workspace_size if want_out else
            L.deltas_gdn_chunk_update_workspace_size)(desc, T)
    ws = L.alloc_workspace(size, dev)
    xs = {k: v.to(dev) for k, v in x.items()}
    st = s0.to(dev).clone()
    out = torch.empty(Lg, T, Hv, d, dtype=torch.bfloat16, device=dev) if want_out else None
    part = torch.zeros(Lg, Hv, 2, device=dev)
    q = xs["q"] if want_out else None

    L.deltas_set_wait_budget(ws, 1)
    L.deltas_gdn_chunk_update(desc, T, q, xs["k"], xs["v"], xs["g"], xs["beta"], st, out, part, ws)
    status, where = L.deltas_get_device_status(ws)
    assert status == L.DELTAS_ERR_TIMEOUT and where > 0

    L.deltas_clear_device_status(ws)
    st.copy_(s0.to(dev))
    L.deltas_gdn_chunk_update(desc, T, q, xs["k"], xs["v"], xs["g"], xs["beta"], st, out, part, ws)
    assert L.deltas_get_device_status(ws) == (0, 0)
    f64 = lambda t: t.float().cpu().double().numpy()       # noqa: E731
    S_ref, o_ref = oracle.gdn_recurrence(f64(x["q"]), f64(x["k"]), f64(x["v"]), f64(x["g"]), f64(x["beta"]),
                                         f64(s0), q_scale=0.25, want_out=want_out)
    assert _rel(f64(st), S_ref) <= 2e-3
    if want_out:
        o = f64(out).transpose(0, 2, 1, 3)
        assert _rel(o, o_ref.transpose(0, 2, 1, 3)) <= 2e-3 + 2.0 ** -8
