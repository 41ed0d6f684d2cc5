"""Benchmark of the DeltaS hot path on GB300 (one JSON line on stdout, rank 0).

Workloads (``--workload``; synthetic inputs shaped like the paper's backbone, Sec. 4.1 / App. A):
* ``streaming`` (default) — Alg. 1 in steady state: per step one 512-token chunk through 24
  gated-delta layers x 32 value heads x 128 x 128 fp32 state (update + fused drift), the chunk
  score, the append to 8 full-attention caches (2 KV heads, D=256, bf16), retain selection at a
  32k-token budget with the paper's policy (n_s=4, n_w=1024, N=4) and in-place compaction.  This
  is the only workload whose step runs every step of the path.
* ``stack``  — 24 layers, 1024-token chunks: update + drift + score only.
* ``layer``  — 1 layer (16 key / 32 value heads, d=128), 1024-token chunks.
* ``kv``     — one eviction on a 64k-token cache (budget 16k, ties injected): select + compact.

Inputs are generated on the device from fixed seeds before timing, as a ring of 8 distinct
per-chunk input sets (each larger than nothing cached: the L2 is also flushed between timed
steps).  Timing: CUDA events on the launching stream around every step and every kernel, W
untimed warm-up steps, K timed steps, max over ranks.  ``--impl reference`` times the CPU
oracle (test infrastructure) on a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2609_27470_gb300 import configs, inputs  # noqa: E402

METRIC = "update+drift tokens/s and % tensor peak; KV-compaction GB/s vs HBM peak (1 GB300)"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
RING = 8
L2_FLUSH_BYTES = 256 << 20


# ----------------------------------------------------------------------------------- helpers

def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def source_sha(relpath):
    with open(os.path.join(ROOT, relpath), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def traffic_for(kernel_key, src):
    """dram bytes per launch from a committed ncu capture, or None if absent or stale."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p)).get(kernel_key)
    if not d or d.get("source_sha") != source_sha(src):
        return None
    return d.get("dram_bytes_per_launch")


class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.tmp = None

    def __enter__(self):
        try:
            self.tmp = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.tmp, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or self.tmp is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        self.tmp.flush()
        rows = [r.split(",") for r in open(self.tmp.name).read().strip().splitlines() if r.count(",") >= 8]
        os.unlink(self.tmp.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].strip() == "Active"})
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


class Timer:
    """Per-kernel CUDA events on the launching stream, accumulated over the timed steps."""

    def __init__(self, stream):
        self.stream = stream
        self.pending = []
        self.totals = {}
        self.counts = {}
        self.on = False

    def mark(self, name):
        if not self.on:
            return _NullCtx()
        return _EvCtx(self, name)

    def collect(self):
        for name, a, b in self.pending:
            self.totals[name] = self.totals.get(name, 0.0) + a.elapsed_time(b)
            self.counts[name] = self.counts.get(name, 0) + 1
        self.pending = []


class _NullCtx:
    def __enter__(self):
        return self

    def __exit__(self, *exc):
        return False


class _EvCtx:
    def __init__(self, t, name):
        self.t, self.name = t, name

    def __enter__(self):
        self.a = torch.cuda.Event(enable_timing=True)
        self.b = torch.cuda.Event(enable_timing=True)
        self.a.record(self.t.stream)
        return self

    def __exit__(self, *exc):
        self.b.record(self.t.stream)
        self.t.pending.append((self.name, self.a, self.b))
        return False


# ----------------------------------------------------------------------------------- workloads

class GdnRing:
    """R distinct per-chunk input sets on the device (generated from seeds, outside timing); set r
    has chunk_lens[r] tokens (one length for all when chunk_lens is an int)."""

    def __init__(self, cfg, chunk_lens, dev, seed):
        lens = [chunk_lens] * RING if isinstance(chunk_lens, int) else list(chunk_lens)
        self.sets = [inputs.gdn_chunk(cfg["L"], lens[r], cfg["Hk"], cfg["Hv"], cfg["d"], cfg["dtype"],
                                      inputs.seed_for(seed, r), device=dev) for r in range(RING)]

    def __getitem__(self, i):
        return self.sets[i % RING]

    def bytes_per_set(self):
        return sum(t.numel() * t.element_size() for t in self.sets[0].values())


def algorithmic_gdn_bytes(L, T, Hk, Hv, d, act_bytes, with_out):
    k = L * T * Hk * d * act_bytes
    q = k if with_out else 0
    v = L * T * Hv * d * act_bytes
    gb = L * T * Hv * 8
    st = 2 * L * Hv * d * d * 4
    part = L * Hv * 8
    o = L * T * Hv * d * act_bytes if with_out else 0
    return k + q + v + gb + st + part + o


def algorithmic_gdn_flops(L, T, Hv, d, with_out):
    return (6 if with_out else 4) * d * d * T * L * Hv


class StreamingWorkload:
    """One chunk per step through the whole path (update + drift, score, append, select, compact)
    on a cache kept at the budget: streaming (512-token chunks) and paper (118-132-token chunks,
    the length cycling through the ring).  With a per-head token signal (paper_key_norm,
    paper_value_norm: Sec. 4.3) the step is update (no drift), append with scores, per-plane
    select and per-plane compact."""

    def __init__(self, dev, L, cfg=None):
        cfg = dict(cfg or configs.STREAMING)
        self.cfg = cfg
        self.name = cfg["name"]
        self.L = L
        self.dev = dev
        C = cfg["chunk_len"]                                   # the longest chunk
        self.C = C
        self.lens = list(cfg.get("chunk_lens", (C,) * RING))
        assert len(self.lens) == RING and max(self.lens) <= C
        self.ring = GdnRing(cfg, self.lens, dev, seed=40)
        self.kv_ring = [inputs.kv_chunk(cfg["Lf"], cfg["Hkv"], self.lens[r], cfg["D"], cfg["kv_dtype"],
                                        inputs.seed_for(41, r), device=dev) for r in range(RING)]
        from paper_2609_27470_gb300.stream import DeltaSStream
        self.s = DeltaSStream(num_layers=cfg["L"], num_k_heads=cfg["Hk"], num_v_heads=cfg["Hv"], head_dim=cfg["d"],
                              act_dtype=torch.bfloat16, kv_layers=cfg["Lf"], kv_heads=cfg["Hkv"],
                              kv_head_dim=cfg["D"], kv_dtype=torch.bfloat16, budget_M=cfg["budget_M"],
                              n_sink=cfg["n_sink"], n_window=cfg["n_window"], n_buckets=cfg["n_buckets"],
                              chunk_len=C, max_chunks=cfg["n_chunks"],
                              state0=inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 42, device=dev),
                              device=dev, signal=cfg.get("signal", "drift"))
        # fill the cache to exactly the budget (setup, not timed): appended chunks with Exp(1)
        # scores, the last one cut to fit, so that every timed step evicts
        M = cfg["budget_M"]
        fills = []
        while sum(fills) < M:
            fills.append(min(self.lens[len(fills) % RING], M - sum(fills)))
        n_fill = len(fills)
        gen = torch.Generator(device=dev)
        gen.manual_seed(43)
        self.s.chunk_scores[:n_fill] = torch.empty(n_fill, device=dev).exponential_(1.0, generator=gen)
        for c, n in enumerate(fills):
            kn, vn = self.kv_ring[c % RING]
            kn, vn = kn[:, :, :n].contiguous(), vn[:, :, :n].contiguous()
            if self.s.per_head:
                L.deltas_append_kv_heads(self.s.kv, self.s.signal, self.s.k_cache, self.s.v_cache, self.s.tok_chunk,
                                         self.s.tok_pos, self.s.tok_score, self.s.cache_len, kn, vn, c,
                                         self.s.position)
            else:
                L.deltas_append_kv(self.s.kv, self.s.k_cache, self.s.v_cache, self.s.tok_chunk, self.s.tok_pos,
                                   self.s.cache_len, kn, vn, c, self.s.position)
            self.s.cache_len += n
            self.s.position += n
        self.s.chunk = n_fill
        self.step_i = 0
        self.moved = None

    def step(self, timer):
        x = self.ring[self.step_i]
        kn, vn = self.kv_ring[self.step_i % RING]
        T = self.lens[self.step_i % RING]
        s, L, c = self.s, self.L, self.s.chunk
        if s.per_head:
            self._step_heads(timer, x, kn, vn, T)
            return
        with timer.mark("gdn_update"):
            L.deltas_gdn_chunk_update(s.gdn, T, None, x["k"], x["v"], x["g"], x["beta"], s.state, None,
                                      s.partials, s.workspace, write_norms=s.write_norms)
        with timer.mark("score"):
            if s.signal == "write_norm":
                L.deltas_score_write_norms(s.gdn.num_layers, s.gdn.num_v_heads, s.write_norms, T, c, s.chunk_scores)
            else:
                L.deltas_score_chunks(s.gdn.num_layers, s.gdn.num_v_heads, s.partials, c, s.chunk_scores)
        with timer.mark("append"):
            L.deltas_append_kv(s.kv, s.k_cache, s.v_cache, s.tok_chunk, s.tok_pos, s.cache_len, kn, vn, c,
                               s.position)
        s.cache_len += T
        s.position += T
        s.chunk += 1
        with timer.mark("select"):
            L.deltas_select_retain(s.policy, s.cache_len, s.tok_chunk, s.chunk_scores[: c + 1], s.retain_idx,
                                   s.n_retained, None, s.workspace)
        with timer.mark("compact"):
            L.deltas_compact_kv(s.kv, s.k_cache, s.v_cache, s.tok_chunk, s.tok_pos, s.retain_idx, s.n_retained,
                                s.cache_len, s.workspace)
        s.cache_len = s.policy.budget_M
        self.step_i += 1

    def _step_heads(self, timer, x, kn, vn, T):
        s, L, c = self.s, self.L, self.s.chunk
        P = s.kv.num_layers * s.kv.num_kv_heads
        with timer.mark("gdn_update"):
            L.deltas_gdn_chunk_update(s.gdn, T, None, x["k"], x["v"], x["g"], x["beta"], s.state, None, None,
                                      s.workspace)
        with timer.mark("append"):
            L.deltas_append_kv_heads(s.kv, s.signal, s.k_cache, s.v_cache, s.tok_chunk, s.tok_pos, s.tok_score,
                                     s.cache_len, kn, vn, c, s.position)
        s.cache_len += T
        s.position += T
        s.chunk += 1
        with timer.mark("select"):
            L.deltas_select_retain_heads(s.policy, s.cache_len, s.tok_chunk.view(P, -1), s.tok_score.view(P, -1),
                                         s.retain_idx, s.n_retained, None, s.workspace)
        with timer.mark("compact"):
            L.deltas_compact_kv_heads(s.kv, s.k_cache, s.v_cache, s.tok_chunk, s.tok_pos, s.tok_score,
                                      s.retain_idx, s.n_retained, s.cache_len, s.workspace)
        s.cache_len = s.policy.budget_M
        self.step_i += 1

    def post_step(self):
        # rows the last compaction moved (slots j whose source differs from j; per plane with a
        # per-head signal); runs between the timed steps, on the device, without a host sync
        idx = self.s.retain_idx
        cnt = (idx != torch.arange(idx.shape[-1], device=idx.device, dtype=torch.int32)).sum()
        self.moved = cnt if self.moved is None else self.moved + cnt

    def launches_per_step(self):
        if self.s.per_head:
            return 2 + 1 + 1 + 3                                # update (2), append, select, compact (3)
        return 2 + 1 + 1 + 3 + 3                                # update (2), score, append, select (3), compact (3)

    def tokens_per_step(self):
        # the mean chunk length (exact when the timed steps are a multiple of the ring)
        return sum(self.lens) / len(self.lens)

    def kernel_roofline(self, name, avg_ms, peaks, steps):
        cfg = self.cfg
        if name == "gdn_update":
            T = self.tokens_per_step()
            by = algorithmic_gdn_bytes(cfg["L"], T, cfg["Hk"], cfg["Hv"], cfg["d"], 2, False)
            fl = algorithmic_gdn_flops(cfg["L"], T, cfg["Hv"], cfg["d"], False)
            return {"bound": "hbm", "achieved": by / (avg_ms * 1e-3) / 1e9, "peak": peaks["hbm_gbs"],
                    "unit": "GB/s", "bytes_per_launch": by,
                    "tensor_frac": fl / (avg_ms * 1e-3) / 1e12 / peaks["bf16_tflops_sustained"]}
        if name == "compact":
            moved = float(self.moved.item()) / steps if self.moved is not None else 0.0
            if self.s.per_head:      # moved (plane, row) pairs: a K row, a V row, 3 metadata words
                row = cfg["D"] * 2 * 2 + 12
            else:                    # moved slots: every plane's K and V row, 2 metadata words
                row = cfg["D"] * 2 * cfg["Lf"] * cfg["Hkv"] * 2 + 8
            by = 2 * moved * row
            return {"bound": "hbm", "achieved": by / (avg_ms * 1e-3) / 1e9, "peak": peaks["hbm_gbs"],
                    "unit": "GB/s", "bytes_per_launch": by, "moved_rows_per_launch": moved}
        return None

    def h2d_tensors(self, i=0):
        x = self.ring[i]
        kn, vn = self.kv_ring[i % RING]
        return [x["k"], x["v"], x["g"], x["beta"], kn, vn]

    def result_scalar(self):
        if self.s.per_head:                     # the score of the newest token of plane 0
            return self.s.tok_score.view(-1)[self.s.cache_len - 1: self.s.cache_len]
        return self.s.chunk_scores[self.s.chunk - 1: self.s.chunk]


class GdnOnlyWorkload:
    """stack / layer: one chunk through every layer per step (update + drift + score)."""

    def __init__(self, dev, L, cfg):
        self.cfg = cfg
        self.name = cfg["name"]
        self.L = L
        self.C = cfg["chunk_len"]
        self.ring = GdnRing(cfg, self.C, dev, seed=50)
        self.gdn = L.gdn_desc(cfg["L"], cfg["Hk"], cfg["Hv"], cfg["d"], torch.bfloat16)
        self.state = inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 51, device=dev)
        self.part = torch.zeros(cfg["L"], cfg["Hv"], 2, device=dev)
        self.scores = torch.zeros(cfg["n_chunks"], device=dev)
        self.with_out = bool(cfg.get("with_out"))
        size = (L.deltas_gdn_chunk_update_readout_workspace_size if self.with_out else
                L.deltas_gdn_chunk_update_workspace_size)(self.gdn, self.C)
        self.ws = L.alloc_workspace(size, dev)
        self.out = (torch.empty(cfg["L"], self.C, cfg["Hv"], cfg["d"], dtype=torch.bfloat16, device=dev)
                    if self.with_out else None)
        self.step_i = 0

    def step(self, timer):
        x = self.ring[self.step_i]
        with timer.mark("gdn_update"):
            self.L.deltas_gdn_chunk_update(self.gdn, self.C, x["q"] if self.with_out else None, x["k"], x["v"],
                                           x["g"], x["beta"], self.state, self.out, self.part, self.ws)
        with timer.mark("score"):
            self.L.deltas_score_chunks(self.cfg["L"], self.cfg["Hv"], self.part,
                                       self.step_i % self.cfg["n_chunks"], self.scores)
        self.step_i += 1

    def launches_per_step(self):
        return 2 + (1 if self.with_out else 0) + 1              # factor + chain (+ read-out) kernels, score

    def tokens_per_step(self):
        return self.C

    def kernel_roofline(self, name, avg_ms, peaks, steps):
        if name != "gdn_update":
            return None
        cfg = self.cfg
        by = algorithmic_gdn_bytes(cfg["L"], self.C, cfg["Hk"], cfg["Hv"], cfg["d"], 2, self.with_out)
        fl = algorithmic_gdn_flops(cfg["L"], self.C, cfg["Hv"], cfg["d"], self.with_out)
        return {"bound": "hbm", "achieved": by / (avg_ms * 1e-3) / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "bytes_per_launch": by, "tensor_frac": fl / (avg_ms * 1e-3) / 1e12 / peaks["bf16_tflops_sustained"]}

    def post_step(self):
        pass

    def h2d_tensors(self, i=0):
        x = self.ring[i]
        return ([x["q"]] if self.with_out else []) + [x["k"], x["v"], x["g"], x["beta"]]

    def result_scalar(self):
        i = (self.step_i - 1) % self.cfg["n_chunks"]
        return self.scores[i: i + 1]


class DriftWorkload:
    """drift: the standalone drift partials (deltas_state_drift) of a whole stack's states plus the
    chunk score, one chunk per step, from a ring of (S_before, S_after) pairs larger than L2."""
    name = "drift"

    def __init__(self, dev, L, cfg=None):
        cfg = dict(cfg or configs.DRIFT)
        self.cfg = cfg
        self.L = L
        self.gdn = L.gdn_desc(cfg["L"], cfg["Hk"], cfg["Hv"], cfg["d"], torch.bfloat16)
        self.pairs = [(inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 60 + 2 * i, device=dev),
                       inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 61 + 2 * i, device=dev))
                      for i in range(cfg["ring"])]
        self.part = torch.zeros(cfg["L"], cfg["Hv"], 2, device=dev)
        self.scores = torch.zeros(cfg["n_chunks"], device=dev)
        self.ws = L.alloc_workspace(L.deltas_state_drift_workspace_size(self.gdn), dev)
        self.step_i = 0

    def step(self, timer):
        sb, sa = self.pairs[self.step_i % len(self.pairs)]
        with timer.mark("drift"):
            self.L.deltas_state_drift(self.gdn, sb, sa, self.part, self.ws)
        with timer.mark("score"):
            self.L.deltas_score_chunks(self.cfg["L"], self.cfg["Hv"], self.part,
                                       self.step_i % self.cfg["n_chunks"], self.scores)
        self.step_i += 1

    def launches_per_step(self):
        return 1 + 1                                            # drift, score

    def tokens_per_step(self):
        return self.cfg["chunk_len"]

    def kernel_roofline(self, name, avg_ms, peaks, steps):
        if name != "drift":
            return None
        c = self.cfg
        by = 2.0 * c["L"] * c["Hv"] * c["d"] * c["d"] * 4 + c["L"] * c["Hv"] * 8   # both states read, partials written
        return {"bound": "hbm", "achieved": by / (avg_ms * 1e-3) / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "bytes_per_launch": by}

    def post_step(self):
        pass

    def h2d_tensors(self, i=0):
        return list(self.pairs[i % len(self.pairs)])

    def result_scalar(self):
        i = (self.step_i - 1) % self.cfg["n_chunks"]
        return self.scores[i: i + 1]


class KvWorkload:
    """One eviction on a full 64k-token cache per step (select + compact); the cache is restored
    from a pristine copy between steps (outside the timed events)."""
    name = "kv"

    def __init__(self, dev, L, cfg=None):
        cfg = dict(cfg or configs.KV)
        self.cfg = cfg
        self.L = L
        cap = cfg["n_chunks"] * cfg["chunk_len"]
        self.cap = cap
        self.k0, self.v0 = inputs.kv_cache(cfg["Lf"], cfg["Hkv"], cap, cfg["D"], "bf16", seed=21, device=dev)
        self.k, self.v = self.k0.clone(), self.v0.clone()
        self.tc0 = inputs.chunked_tok_chunk(cfg["n_chunks"], cfg["chunk_len"]).to(dev)
        self.tp0 = torch.arange(cap, dtype=torch.int32, device=dev)
        self.tc, self.tp = self.tc0.clone(), self.tp0.clone()
        self.scores = inputs.chunk_scores_with_ties(cfg["n_chunks"], seed=3).to(dev)
        self.kv = L.kv_desc(cfg["Lf"], cfg["Hkv"], cfg["D"], torch.bfloat16, cap)
        self.pol = L.policy(cfg["budget_M"], 4, 1024, 4)
        self.idx = torch.zeros(cfg["budget_M"], dtype=torch.int32, device=dev)
        self.n = torch.zeros(1, dtype=torch.int32, device=dev)
        self.ws = L.alloc_workspace(max(L.deltas_select_retain_workspace_size(cap),
                                        L.deltas_compact_kv_workspace_size(self.kv, cap)), dev)
        self.moved = None

    def reset(self):
        self.k.copy_(self.k0)
        self.v.copy_(self.v0)
        self.tc.copy_(self.tc0)
        self.tp.copy_(self.tp0)

    def step(self, timer):
        with timer.mark("select"):
            self.L.deltas_select_retain(self.pol, self.cap, self.tc, self.scores, self.idx, self.n, None, self.ws)
        with timer.mark("compact"):
            self.L.deltas_compact_kv(self.kv, self.k, self.v, self.tc, self.tp, self.idx, self.n, self.cap, self.ws)

    def launches_per_step(self):
        return 3 + 3                                            # selection: runs, retain, emit; compaction: init, need, main

    def tokens_per_step(self):
        return self.cap

    def kernel_roofline(self, name, avg_ms, peaks, steps):
        if name != "compact":
            return None
        moved = float(self.moved.item()) / steps if self.moved is not None else 0.0
        row = self.cfg["D"] * 2 * self.cfg["Lf"] * self.cfg["Hkv"] * 2 + 8
        by = 2 * moved * row
        return {"bound": "hbm", "achieved": by / (avg_ms * 1e-3) / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "bytes_per_launch": by, "moved_rows_per_launch": moved}

    def post_step(self):
        ar = torch.arange(self.cfg["budget_M"], device=self.idx.device, dtype=torch.int32)
        cnt = (self.idx != ar).sum()
        self.moved = cnt if self.moved is None else self.moved + cnt

    def h2d_tensors(self, i=0):
        return [self.scores]

    def result_scalar(self):
        return self.n


KERNEL_SOURCES = {"gdn_update": "paper_2609_27470_gb300/csrc/gdn_tc.cu",
                  "compact": "paper_2609_27470_gb300/csrc/compact.cu",
                  "select": "paper_2609_27470_gb300/csrc/select.cu",
                  "score": "paper_2609_27470_gb300/csrc/drift.cu",
                  "append": "paper_2609_27470_gb300/csrc/compact.cu",
                  "snapshot": "paper_2609_27470_gb300/csrc/snapshot.cu",
                  "drift": "paper_2609_27470_gb300/csrc/drift.cu",
                  "restore": "paper_2609_27470_gb300/csrc/snapshot.cu"}


def kernel_source(workload, name):
    """The source file of a timed kernel (the per-head selection has its own)."""
    if name == "select" and _cfg(workload).get("signal") in ("key_norm", "value_norm"):
        return "paper_2609_27470_gb300/csrc/select_heads.cu"
    return KERNEL_SOURCES[name]


class SnapshotWorkload:
    """Question-time snapshot and restore (Sec. 3.3) of a paper-shaped stream at its budget: the
    24 x 32 x 128 x 128 fp32 recurrent state (48 MiB), the 8,192-token caches of 8 layers x 4 KV
    heads (256 MiB), the slots' chunk ids and positions and 4,096 chunk scores.  A step saves the
    whole state and puts it back (deltas_copy_stream_state twice: one launch each)."""
    name = "snapshot"

    def __init__(self, dev, L, cfg=None):
        cfg = dict(cfg or configs.PAPER)
        self.cfg = cfg
        self.L = L
        from paper_2609_27470_gb300.stream import DeltaSStream, StreamSnapshot
        self.s = DeltaSStream(num_layers=cfg["L"], num_k_heads=cfg["Hk"], num_v_heads=cfg["Hv"], head_dim=cfg["d"],
                              act_dtype=torch.bfloat16, kv_layers=cfg["Lf"], kv_heads=cfg["Hkv"],
                              kv_head_dim=cfg["D"], kv_dtype=torch.bfloat16, budget_M=cfg["budget_M"],
                              n_sink=cfg["n_sink"], n_window=cfg["n_window"], n_buckets=cfg["n_buckets"],
                              chunk_len=cfg["chunk_len"], max_chunks=cfg["n_chunks"],
                              state0=inputs.initial_state(cfg["L"], cfg["Hv"], cfg["d"], 90, device=dev),
                              device=dev)
        s = self.s
        k, v = inputs.kv_cache(cfg["Lf"], cfg["Hkv"], s.capacity, cfg["D"], "bf16", seed=91, device=dev)
        s.k_cache.copy_(k)
        s.v_cache.copy_(v)
        del k, v
        M = cfg["budget_M"]
        s.tok_chunk[:M] = torch.arange(M, device=dev, dtype=torch.int32) // cfg["chunk_len"]
        s.tok_pos[:M] = torch.arange(M, device=dev, dtype=torch.int32) * 3
        gen = torch.Generator(device=dev)
        gen.manual_seed(92)
        s.chunk_scores.exponential_(1.0, generator=gen)
        s.cache_len, s.position, s.chunk = M, 3 * M, cfg["n_chunks"]
        self.snap = StreamSnapshot(s, full=True)

    def step(self, timer):
        with timer.mark("snapshot"):
            self.s.snapshot(into=self.snap)
        with timer.mark("restore"):
            self.s.restore(self.snap)

    def bytes_per_copy(self):
        c, s = self.cfg, self.s
        return (s.state.numel() * 4 + s.chunk * 4 + 2 * c["Lf"] * c["Hkv"] * s.cache_len * c["D"] * 2
                + 2 * s.cache_len * 4)

    def launches_per_step(self):
        return 2

    def tokens_per_step(self):
        return self.s.cache_len

    def kernel_roofline(self, name, avg_ms, peaks, steps):
        by = 2.0 * self.bytes_per_copy()                       # every byte read once and written once
        return {"bound": "hbm", "achieved": by / (avg_ms * 1e-3) / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "bytes_per_launch": by}

    def post_step(self):
        pass

    def h2d_tensors(self, i=0):
        return [self.s.chunk_scores]

    def result_scalar(self):
        return self.s.chunk_scores[:1]


def make_workload(name, dev, L):
    if name == "streaming":
        return StreamingWorkload(dev, L)
    if name == "paper":
        return StreamingWorkload(dev, L, configs.PAPER)
    if name in ("paper_write_norm", "paper_key_norm", "paper_value_norm"):
        return StreamingWorkload(dev, L, _cfg(name))
    if name == "stack":
        return GdnOnlyWorkload(dev, L, configs.STACK)
    if name == "stack_out":
        return GdnOnlyWorkload(dev, L, configs.STACK_OUT)
    if name == "layer":
        return GdnOnlyWorkload(dev, L, configs.LAYER)
    if name == "layer_out":
        return GdnOnlyWorkload(dev, L, configs.LAYER_OUT)
    if name == "kv":
        return KvWorkload(dev, L)
    if name == "drift":
        return DriftWorkload(dev, L)
    if name == "snapshot":
        return SnapshotWorkload(dev, L)
    raise ValueError(name)


# ----------------------------------------------------------------------------------- ranks

def max_over_ranks(local_ms: float, dev, world: int) -> float:
    """The slowest rank's timed-region duration (ms): every rank's clock counts."""
    t = torch.tensor([float(local_ms)], dtype=torch.float64, device=dev)
    if world > 1:
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank_step: float, steps: int, world: int, t_max_ms: float) -> float:
    """Units processed by all ranks together per second of the slowest rank's time.  Each rank runs
    its own independent stream (weak scaling: the per-rank work does not shrink as ranks are added)."""
    return units_per_rank_step * steps * world / (t_max_ms * 1e-3)


# ----------------------------------------------------------------------------------- end to end

def e2e_sequential(wl, host, steps, stream, timer_off, reset):
    """Per step: pinned host inputs -> device, the step, its score -> pinned host, all on one stream;
    the timed region of each step starts after the workload's reset."""
    host_out = torch.zeros(1, dtype=wl.result_scalar().dtype).pin_memory()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e_ms = 0.0
    for _ in range(steps):
        reset()
        e0.record(stream)
        i = getattr(wl, "step_i", 0)
        for h, d in zip(host[i % len(host)], wl.h2d_tensors(i)):
            d.copy_(h, non_blocking=True)
        wl.step(timer_off)
        host_out.copy_(wl.result_scalar(), non_blocking=True)
        e1.record(stream)
        e1.synchronize()
        e_ms += e0.elapsed_time(e1)
        _ = float(host_out[0])
    return e_ms


def e2e_pipelined(wl, host, steps, stream, dev, timer_off):
    """A stream of chunks as a serving loop runs it: every step's inputs are copied from pinned host
    memory on a copy stream (into the ring slot that step reads) while the previous step computes;
    each step's score is copied back to pinned host memory and read by the host one step later.
    Returns the time from the first copy to the last read-back (ms)."""
    cs = torch.cuda.Stream(dev)
    copied = [torch.cuda.Event() for _ in range(steps)]
    done = [torch.cuda.Event() for _ in range(steps)]
    host_out = [torch.zeros(1, dtype=wl.result_scalar().dtype).pin_memory() for _ in range(2)]
    e_start = torch.cuda.Event(enable_timing=True)
    e_end = torch.cuda.Event(enable_timing=True)
    slot0 = getattr(wl, "step_i", 0)
    e_start.record(cs)
    for i in range(steps):
        with torch.cuda.stream(cs):
            if i >= 2:
                cs.wait_event(done[i - 2])                 # at most two steps in flight
            for h, d in zip(host[(slot0 + i) % len(host)], wl.h2d_tensors(slot0 + i)):
                d.copy_(h, non_blocking=True)
            copied[i].record(cs)
        stream.wait_event(copied[i])
        wl.step(timer_off)
        host_out[i % 2].copy_(wl.result_scalar(), non_blocking=True)
        done[i].record(stream)
        if i >= 1:
            done[i - 1].synchronize()
            _ = float(host_out[(i - 1) % 2][0])
    e_end.record(stream)
    e_end.synchronize()
    _ = float(host_out[(steps - 1) % 2][0])
    return e_start.elapsed_time(e_end)


# ----------------------------------------------------------------------------------- CPU oracle

def _pool_time(fn, n_items, threads):
    """Seconds for fn(i), i < n_items, on `threads` threads (the oracle's C calls release the GIL)."""
    t0 = time.perf_counter()
    if threads <= 1:
        for i in range(n_items):
            fn(i)
    else:
        from concurrent.futures import ThreadPoolExecutor
        with ThreadPoolExecutor(max_workers=threads) as ex:
            list(ex.map(fn, range(n_items)))
    return time.perf_counter() - t0


def oracle_sample(workload: str, budget_s: float = 12.0, threads: int = 1):
    """Times the CPU oracle on a bounded sample of one step of the workload and extrapolates to a
    whole step: on one thread, or with the independent (layer, head) recurrences and compaction
    planes spread over `threads` threads.  Returns (tokens_per_s, sample description, seconds
    spent, extrapolation factor of the sampled part)."""
    import oracle
    t_start = time.perf_counter()
    cfg = _cfg(workload)
    parts = []
    total = 0.0
    factor = 1.0
    if workload == "drift":
        heads_total = cfg["L"] * cfg["Hv"]
        n = max(64, 8 * threads)
        sb = inputs.initial_state(1, n, cfg["d"], 60).double().numpy()
        sa = inputs.initial_state(1, n, cfg["d"], 61).double().numpy()
        t = _pool_time(lambda i: oracle.drift_partials(sb[:, i:i + 1], sa[:, i:i + 1]), n, threads)
        factor = heads_total / n
        total += t * factor
        p = np.ones((cfg["L"], cfg["Hv"], 2))
        t0 = time.perf_counter()
        oracle.chunk_score(p)
        total += time.perf_counter() - t0
        parts.append(f"drift of {n} (layer,head) state pairs x{factor:.0f} extrapolated; score of {cfg['L']} layers")
    head_signal = cfg.get("signal") in ("key_norm", "value_norm")
    if workload in ("streaming", "paper", "paper_write_norm", "paper_key_norm", "paper_value_norm", "stack",
                    "stack_out", "layer", "layer_out"):
        C = int(round(_tokens(workload)))
        heads_total = cfg["L"] * cfg["Hv"]
        n_heads = 2
        x = inputs.gdn_chunk(1, C, 1, 1, cfg["d"], "bf16", 77)
        f = {k: v.float().numpy() for k, v in x.items()}
        s0 = inputs.initial_state(1, 1, cfg["d"], 78).double().numpy()

        def one_head(_):
            if workload == "paper_write_norm":
                oracle.gdn_recurrence(None, f["k"], f["v"], f["g"], f["beta"], s0, want_write_norms=True)
            elif head_signal:                              # the state moves; no drift is formed
                oracle.gdn_recurrence(None, f["k"], f["v"], f["g"], f["beta"], s0)
            elif cfg.get("with_out"):                      # with the layer output
                S, _ = oracle.gdn_recurrence(f["q"], f["k"], f["v"], f["g"], f["beta"], s0, want_out=True)
                oracle.drift_partials(s0, S)
            else:
                S, _ = oracle.gdn_recurrence(None, f["k"], f["v"], f["g"], f["beta"], s0)
                oracle.drift_partials(s0, S)
        batch = max(n_heads, threads)
        reps, t_sum = 0, 0.0
        while True:
            t_sum += _pool_time(one_head, batch, threads)
            reps += batch
            if t_sum > budget_s * 0.5 or reps >= 64 * max(1, threads):
                break
        t_head = t_sum / reps
        factor = heads_total / reps
        total += t_head * heads_total
        parts.append(f"gdn: {reps} (layer,head) x {C} tokens on {threads} thread(s), x{factor:.0f} extrapolated")
    if workload == "snapshot":
        # the oracle's question handling copies the whole stream state (numpy .copy()); timed on
        # a 64 MiB slice and scaled to the bytes of one save and one restore
        M = cfg["budget_M"]
        per_copy = (cfg["L"] * cfg["Hv"] * cfg["d"] ** 2 * 8 + cfg["n_chunks"] * 4
                    + 2 * cfg["Lf"] * cfg["Hkv"] * M * cfg["D"] * 2 + 2 * M * 4)
        a = np.random.default_rng(7).standard_normal(8 << 20)
        t0 = time.perf_counter()
        reps = 0
        while reps < 2 or time.perf_counter() - t0 < budget_s * 0.25:
            a.copy()
            reps += 1
        t_byte = (time.perf_counter() - t0) / (reps * a.nbytes)
        total += 2 * per_copy * t_byte
        parts.append(f"numpy copy of 64 MiB x{reps}, scaled to 2 x {per_copy / 2**20:.0f} MiB "
                     "(fp64 state, as the oracle keeps it)")
    if workload in ("streaming", "paper", "paper_write_norm", "kv"):
        M = cfg["budget_M"]
        if workload != "kv":
            T = M + cfg["chunk_len"]
            rng = np.random.default_rng(5)
            lens = rng.integers(1, cfg["chunk_len"] + 1, size=4 * T // cfg["chunk_len"])
            tc = np.concatenate([np.full(n, c, np.int32) for c, n in enumerate(lens)])[-T:]
            sc = rng.exponential(size=len(lens)).astype(np.float32)
            pol = (M, cfg["n_sink"], cfg["n_window"], cfg["n_buckets"])
        else:
            T = cfg["n_chunks"] * cfg["chunk_len"]
            tc = inputs.chunked_tok_chunk(cfg["n_chunks"], cfg["chunk_len"]).numpy()
            sc = inputs.chunk_scores_with_ties(cfg["n_chunks"], seed=3).numpy()
            pol = (M, 4, 1024, 4)
        t0 = time.perf_counter()
        idx, _ = oracle.select_retain(*pol, tc, sc)
        t_sel = time.perf_counter() - t0
        planes_total = 2 * cfg["Lf"] * cfg["Hkv"]
        plane = np.random.default_rng(6).integers(-2**15, 2**15, size=(2, T, cfg["D"]), dtype=np.int16)
        n_pairs = max(1, min(threads, planes_total // 2))
        t_cmp = _pool_time(lambda i: oracle.compact_rows(plane, idx, T), n_pairs, threads) * planes_total / (2 * n_pairs)
        total += t_sel + t_cmp
        parts.append(f"select on {T} slots; compact {2 * n_pairs} of {planes_total} planes x{planes_total // (2 * n_pairs)}")
    if head_signal:
        # score the chunk's rows, then per (layer, KV head) plane: select among M + C slots with
        # per-token scores and gather the plane's K and V rows; one plane timed, x planes
        M, C, D = cfg["budget_M"], cfg["chunk_len"], cfg["D"]
        T = M + C
        P = cfg["Lf"] * cfg["Hkv"]
        rng = np.random.default_rng(8)
        lens = rng.integers(1, C + 1, size=4 * T // C)
        tc = np.concatenate([np.full(n, c, np.int32) for c, n in enumerate(lens)])[-T:]
        ts = rng.standard_normal(T).astype(np.float32)
        rows = rng.standard_normal((P, C, D)).astype(np.float32)
        t0 = time.perf_counter()
        oracle.row_norm_scores(rows, cfg["signal"])
        t_score = time.perf_counter() - t0
        t0 = time.perf_counter()
        idx, _ = oracle.select_retain_tokens(M, cfg["n_sink"], cfg["n_window"], cfg["n_buckets"], tc, ts)
        t_sel = time.perf_counter() - t0
        plane = rng.integers(-2**15, 2**15, size=(2, T, D), dtype=np.int16)
        meta = np.zeros((3, T, 1), np.int32)
        t0 = time.perf_counter()
        oracle.compact_rows(plane, idx, T)
        oracle.compact_rows(meta, idx, T)
        t_cmp = time.perf_counter() - t0
        total += t_score + P * (t_sel + t_cmp)
        parts.append(f"score {P}x{C} rows; select on {T} slots and compact K, V, metadata of 1 of {P} planes x{P}")
    return _tokens(workload) / total, "; ".join(parts), time.perf_counter() - t_start, factor


# ----------------------------------------------------------------------------------- main

def run_reference(args):
    """The oracle as it stands, on this host's cores, one sampled step per timed step: each timed
    step runs the oracle on a bounded sample of the workload's step (a few (layer, head)
    recurrences and compaction planes), and `value` extrapolates the sample to the whole step.
    ms_per_step is the wall time of the sampled steps actually run, so steps x ms_per_step is the
    time this arm took."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    vals, walls = [], []
    desc, factor = "", 1.0
    for _ in range(args.warmup):
        oracle_sample(args.workload, budget_s=1.0)
    for _ in range(args.steps):
        v, desc, wall, factor = oracle_sample(args.workload, budget_s=2.0)
        vals.append(v)
        walls.append(wall)
    value = float(np.median(vals))
    out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": 1e3 * float(np.mean(walls)),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference",
           "config": config_line(args.workload),
           "timing": {"per_step": "one bounded sample of the workload's step, extrapolated to the whole step",
                      "extrapolation_factor": factor,
                      "ms_per_full_step_extrapolated": 1e3 * _tokens(args.workload) / value},
           "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle", "sample": desc},
           "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def config_line(workload):
    """The workload description printed in "config" by both arms."""
    c = _cfg(workload)
    line = {"workload": workload, "l2": "flushed between timed steps (256 MiB write)",
            "inputs": "ring of 8 distinct per-chunk input sets, generated on device"}
    for key in ("L", "Hk", "Hv", "d", "chunk_len", "chunk_lens", "with_out", "Lf", "Hkv", "D", "budget_M", "n_sink",
                "n_window", "n_buckets", "signal"):
        if key in c:
            line[key] = c[key]
    if workload == "kv":
        line["cache_len"] = c["n_chunks"] * c["chunk_len"]
    if workload == "snapshot":
        line["cache_len"] = c["budget_M"]
        line["copied"] = "state, chunk scores, live cache rows, chunk ids, positions: snapshot + restore per step"
        line["inputs"] = "one stream state generated on device"
    return line


def _cfg(workload):
    return {"streaming": configs.STREAMING, "paper": configs.PAPER, "stack": configs.STACK,
            "stack_out": configs.STACK_OUT,
            "layer": configs.LAYER, "layer_out": configs.LAYER_OUT, "kv": configs.KV, "snapshot": configs.PAPER, "drift": configs.DRIFT,
            "paper_write_norm": configs.PAPER_WRITE_NORM, "paper_key_norm": configs.PAPER_KEY_NORM,
            "paper_value_norm": configs.PAPER_VALUE_NORM}[workload]


def _tokens(workload):
    """Tokens per step: the chunk length (the mean of the cycle for paper), the cache for kv."""
    cfg = _cfg(workload)
    if workload == "kv":
        return cfg["n_chunks"] * cfg["chunk_len"]
    if workload == "snapshot":
        return cfg["budget_M"]
    lens = cfg.get("chunk_lens")
    return sum(lens) / len(lens) if lens else cfg["chunk_len"]


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="streaming",
                    choices=["streaming", "paper", "paper_write_norm", "paper_key_norm", "paper_value_norm",
                             "stack", "stack_out", "layer", "layer_out", "kv", "snapshot", "drift"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.impl == "reference":
        run_reference(args)
        return

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    from paper_2609_27470_gb300 import _lib as L
    stream = torch.cuda.current_stream(dev)
    wl = make_workload(args.workload, dev, L)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    timer = Timer(stream)
    peaks, peaks_src = load_peaks()

    def reset():
        if hasattr(wl, "reset"):
            wl.reset()
        flush.fill_(1.0)

    for _ in range(args.warmup):
        reset()
        wl.step(timer)
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    # the timed steps carry events at their boundaries only (events between kernels would cut the
    # programmatic dependent launches apart); the per-kernel breakdown comes from a second,
    # instrumented pass below
    step_ms = []
    barrier()
    with ClockSampler(local) as clocks:
        wall0 = time.perf_counter()
        for _ in range(args.steps):
            reset()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            wl.step(timer)
            b.record(stream)
            step_ms.append((a, b))
            wl.post_step()
        barrier()
        wall = time.perf_counter() - wall0
    ms = [a.elapsed_time(b) for a, b in step_ms]
    # per-kernel breakdown: the same steps again with an event pair around every kernel
    n_bd = min(args.steps, 20)
    if hasattr(wl, "moved"):
        wl.moved = None
    timer.on = True
    for _ in range(n_bd):
        reset()
        wl.step(timer)
        wl.post_step()
    barrier()
    timer.on = False
    timer.collect()
    t_local = float(sum(ms))
    t_max = max_over_ranks(t_local, dev, world)
    value = whole_job_rate(wl.tokens_per_step(), args.steps, world, t_max)
    ms_per_step = t_max / args.steps

    # end to end through the public API: pinned host inputs copied in, score read back, every step
    # pinned host copies of the step inputs: one set, or one per ring slot when the chunk length
    # cycles (the paper workload)
    n_host = RING if len(set(getattr(wl, "lens", [0]))) > 1 else 1
    host = [[x.detach().cpu().pin_memory() for x in wl.h2d_tensors(r)] for r in range(n_host)]
    h2d = sum(x.numel() * x.element_size() for hs in host for x in hs) / len(host)   # mean bytes per step
    timer_off = Timer(stream)
    barrier()
    if hasattr(wl, "reset"):
        e_ms = e2e_sequential(wl, host, args.steps, stream, timer_off, reset)
        e2e_mode = "sequential: per step, copy in -> compute -> read back (cache restore excluded)"
    else:
        e_ms = e2e_pipelined(wl, host, args.steps, stream, dev, timer_off)
        e2e_mode = "pipelined: step i+1's inputs copied on a second stream while step i computes"
    e2e_value = whole_job_rate(wl.tokens_per_step(), args.steps, world, max_over_ranks(e_ms, dev, world))

    kernels = {}
    for name, tot in timer.totals.items():
        kernels[name] = {"avg_us": 1e3 * tot / timer.counts[name], "share": tot / max(t_local, 1e-9)}
    dominant = max(kernels, key=lambda k: kernels[k]["avg_us"] * timer.counts[k])
    rl = wl.kernel_roofline(dominant, kernels[dominant]["avg_us"] * 1e-3, peaks, n_bd)
    roofline = None
    if rl is not None:
        roofline = {"kernel": dominant, "bound": rl["bound"], "achieved": rl["achieved"], "peak": rl["peak"],
                    "unit": rl["unit"], "frac": rl["achieved"] / rl["peak"],
                    "traffic": traffic_for(f"{args.workload}:{dominant}", kernel_source(args.workload, dominant)),
                    "peak_source": f"{peaks_src} (hbm_gbs)",
                    "algorithmic_bytes_per_launch": rl["bytes_per_launch"]}
        if "tensor_frac" in rl:
            roofline["tensor_frac_algorithmic"] = rl["tensor_frac"]
    extra = {}
    for name in kernels:
        r = wl.kernel_roofline(name, kernels[name]["avg_us"] * 1e-3, peaks, n_bd)
        if r is not None:
            kernels[name]["achieved"] = r["achieved"]
            kernels[name]["unit"] = r["unit"]
            kernels[name]["frac_of_peak"] = r["achieved"] / r["peak"]
            if "moved_rows_per_launch" in r:
                kernels[name]["moved_rows_per_launch"] = r["moved_rows_per_launch"]
            if "tensor_frac" in r:
                kernels[name]["tensor_frac_algorithmic"] = r["tensor_frac"]

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, desc, _, _ = oracle_sample(args.workload)
        n_cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
        va, desc_a, _, _ = oracle_sample(args.workload, budget_s=6.0, threads=n_cores)
        cpu = {"value": v, "unit": "tokens/s", "cores": 1, "kind": "oracle", "sample": desc,
               "all_cores": {"value": va, "unit": "tokens/s", "cores": n_cores, "sample": desc_a}}

    if rank == 0:
        cfg_line = config_line(args.workload)
        out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
               "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
               "scaling": "weak", "vs_baseline": None, "dtype": "bf16 in / f32 state",
               "data": "synthetic (seeded, paper-shaped)", "config": cfg_line,
               "roofline": roofline, "kernels": kernels,
               "kernels_from": f"{n_bd} further steps with an event pair around every kernel (the timed "
                               "steps have events at their boundaries only)",
               "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": 4,
                       "mode": e2e_mode},
               "gpu_launches": wl.launches_per_step() * args.steps, "clocks": clocks.summary(),
               "wall_s_timed": wall, "cpu_baseline": cpu, "library": L.deltas_version()}
        print(json.dumps(out), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
