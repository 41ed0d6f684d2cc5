"""The bounded-wait path on the GPU: a wait that runs out records DELTAS_ERR_TIMEOUT in the
workspace's status word, the call returns, and the next call with the default budget is correct.

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
