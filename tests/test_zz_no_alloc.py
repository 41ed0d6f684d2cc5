"""deltas_select_retain_static: retain selection with the library's own fixed scratch, for callers
that may not allocate device memory.  Its results must equal those of deltas_select_retain (the
workspace entry point) bit for bit, on consecutive calls that share the scratch.

This file is named so that pytest collects it last: it must pass after every other test has run
in the same process, as well as alone in a fresh one.
"""
import ctypes

import numpy as np
import pytest
import torch

FAKE = 1 << 20      # a non-null host address that the argument checks never dereference


@pytest.fixture(scope="module")
def L():
    from paper_2609_27470_gb300 import build
    build.build()
    from paper_2609_27470_gb300 import _lib
    return _lib


def test_static_select_argument_checks(L):
    """Host checks only (no device is touched): the scratch limit and the workspace entry point's
    argument rules; each rejected call enqueues nothing."""
    raw = L.raw()

    def call(pol, T=100, nch=10):
        return raw.deltas_select_retain_static(ctypes.byref(pol) if pol else None, T, nch, FAKE, FAKE, FAKE,
                                               FAKE, None, None)
    assert L.SELECT_STATIC_MAX_CACHE_LEN == 65536
    assert call(L.Policy(10, 0, 0, 1), T=L.SELECT_STATIC_MAX_CACHE_LEN + 1) == L.DELTAS_ERR_UNSUPPORTED
    assert call(L.Policy(10, 0, 0, 1), T=1 << 30) == L.DELTAS_ERR_UNSUPPORTED
    assert call(None) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert call(L.Policy(10, 5, 5, 1)) == L.DELTAS_ERR_INVALID_ARGUMENT
    assert call(L.Policy(10, 0, 0, 33)) == L.DELTAS_ERR_UNSUPPORTED
    assert call(L.Policy(10, 0, 0, 1), T=-1) == L.DELTAS_ERR_INVALID_ARGUMENT


def _case(seed, T, n_ch, run_len_max):
    """A stream-ordered cache with many short runs (so that the run count exceeds what the kernel
    keeps in shared memory and the scratch arrays are used) and a few exact score ties."""
    rng = np.random.default_rng(seed)
    lens = rng.integers(1, run_len_max + 1, size=4 * T // (run_len_max + 1) + 8)
    ids = rng.integers(0, n_ch, size=lens.size)
    tc = np.repeat(ids, lens)[:T].astype(np.int32)
    assert tc.size == T
    sc = rng.exponential(size=n_ch).astype(np.float32)
    sc[rng.integers(0, n_ch, size=8)] = sc[1]
    return tc, sc


def _select_both(L, pol, tc, sc):
    T = tc.size
    dev = torch.device("cuda")
    tct = torch.from_numpy(tc).to(dev)
    sct = torch.from_numpy(sc).to(dev)
    outs = []
    for static in (False, True):
        idx = torch.full((max(min(T, pol.budget_M), 1),), -7, dtype=torch.int32, device=dev)
        n = torch.full((1,), -7, dtype=torch.int32, device=dev)
        mask = torch.full((max(T, 1),), 9, dtype=torch.uint8, device=dev)
        if static:
            L.deltas_select_retain_static(pol, T, tct, sct, idx, n, mask)
        else:
            ws = L.alloc_workspace(L.deltas_select_retain_workspace_size(T), dev)
            L.deltas_select_retain(pol, T, tct, sct, idx, n, mask, ws)
            torch.cuda.synchronize()
            assert L.deltas_get_device_status(ws) == (0, 0)
        torch.cuda.synchronize()
        nn = int(n.item())
        outs.append((nn, idx[:nn].cpu().numpy(), mask[:T].cpu().numpy()))
    return outs


@pytest.mark.gpu
def test_static_select_matches_workspace_select_twice(L):
    """Two calls in a row on different inputs (the second finds the first one's leftovers in the
    shared scratch), each equal to the workspace entry point's result: bit-exact, as every
    selection test is."""
    rng = np.random.default_rng(4)
    stream_tc = np.repeat(np.arange(40, dtype=np.int32), 512)        # 40 runs of one chunk each
    stream_sc = rng.exponential(size=40).astype(np.float32)
    stream_sc[[7, 21]] = stream_sc[3]
    keep_tc = np.repeat(np.arange(10, dtype=np.int32), 500)          # 5000 slots under the budget
    cases = [
        (L.policy(20000, 4, 1024, 4), *_case(1, 60000, 3000, 6)),     # largest size, thousands of runs
        (L.policy(9000, 4, 512, 3), *_case(2, 23000, 700, 4)),        # smaller, other policy
        # right after a many-run call: a streaming-shaped cache with a few dozen runs (the decision
        # kernel's direct path, which stages run starts, kept counts and offsets in the scratch)
        (L.policy(16000, 4, 1024, 4), stream_tc, stream_sc),
        # right after an eviction: a cache within the budget (everything kept; a stale emit flag
        # from the previous call must not be used)
        (L.policy(8000, 4, 1024, 4), keep_tc, rng.exponential(size=10).astype(np.float32)),
    ]
    for pol, tc, sc in cases:
        (n_ref, idx_ref, mask_ref), (n, idx, mask) = _select_both(L, pol, tc, sc)
        assert n_ref == min(pol.budget_M, tc.size) and n == n_ref
        assert np.array_equal(idx, idx_ref)
        assert np.array_equal(mask, mask_ref)


@pytest.mark.gpu
def test_static_select_reports_bad_chunk_then_recovers(L):
    """A chunk id out of range is reported as *n_retained == 0; the next call on the same scratch
    is again equal to the workspace entry point's result."""
    pol = L.policy(3000, 4, 256, 4)
    tc, sc = _case(3, 8000, 400, 3)
    bad = tc.copy()
    bad[5000] = 400                                    # == num_chunks: out of range
    dev = torch.device("cuda")
    idx = torch.zeros(3000, dtype=torch.int32, device=dev)
    n = torch.full((1,), -7, dtype=torch.int32, device=dev)
    L.deltas_select_retain_static(pol, bad.size, torch.from_numpy(bad).to(dev), torch.from_numpy(sc).to(dev),
                                  idx, n, None)
    torch.cuda.synchronize()
    assert int(n.item()) == 0
    (n_ref, idx_ref, mask_ref), (n2, idx2, mask2) = _select_both(L, pol, tc, sc)
    assert n2 == n_ref == 3000
    assert np.array_equal(idx2, idx_ref) and np.array_equal(mask2, mask_ref)
