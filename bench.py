#!/usr/bin/env python
"""Benchmark of the region-sparse DiT denoising step on GB300.

Workload: PixArt-alpha-shaped DiT at 1024 px (64 x 64 = 4096 image tokens,
28 blocks, hidden 1152, 16 heads of 72, MLP 4608, 120 text tokens, 20
timesteps), batch 1, bf16 weights and a bf16 per-(layer, timestep) K/V/hidden
cache of 15.85 GB resident in HBM.  The dirty region of each sweep point is a
union of 1-3 seeded ellipses covering 5 / 10 / 20 / 40 % of the tokens,
presented to the localisation kernel as a cross-attention score map.

One step = localisation mask (rc_localize_mask) + one region-sparse
denoising step at timestep t = step mod 20, replayed from the CUDA graph of
rc_step (mode SPARSE) for that timestep, which reads the dirty list from the
localisation buffers; the headline value is steps/s at 20 % dirty.  The same
steps issued launch by launch (rc_step), the library's own dense path and
every sweep point are reported beside it.

Usage: python bench.py [--gpus N --steps K --warmup W] [--impl reference]
For N > 1 launch with torch.distributed.run: every rank runs an independent
replica (its own session and cache); value = all ranks' steps / max time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_29809_gb300 import synth  # noqa: E402

METRIC = "region-reuse DiT steps/s @4096 tok vs dirty %; % of BF16 tensor peak"
UNIT = "steps/s"
SEED = 1234 + 300
FRACS = (0.05, 0.10, 0.20, 0.40)
HEADLINE = 0.20
WORKLOAD = "pixart-alpha-1024px: 4096 tokens, 28 blocks, 20 timesteps, batch 1"
L2_NOTE = ("inputs larger than L2: each step streams 1.04 GB of weights and a different "
           "28 x 28.3 MB cache slice per timestep")


def linear_flops_per_token_block(d: synth.Dims, folded: bool = True) -> float:
    """2 x (3h^2 + h^2 [+ h^2] + h^2 + hF + Fh) per dirty token and block: the
    GEMM launches (QKV, out, [cross-q,] cross-out, fc1, fc2).  With the
    cross-query projection folded into the text keys (sparse steps) its 2 h^2
    run inside the cross-attention kernel instead."""
    h, F = d.hidden, d.mlp
    return 2.0 * ((5 if folded else 6) * h * h + 2 * h * F)


def attn_flops_per_token_block(d: synth.Dims, folded: bool = True) -> float:
    """Self-attention (4 N h) plus cross-attention (4 M h), with its query
    projection (2 h^2) when folded, per dirty token and block."""
    return (4.0 * d.tokens * d.hidden + 4.0 * d.text_len * d.hidden +
            (2.0 * d.hidden * d.hidden if folded else 0.0))


KERNEL_SOURCES = {
    "gemm": ["gemm_tc.cu", "tc_common.cuh", "common.cuh", "kernels.h"],
    "attention": ["attention_tc.cu", "tc_common.cuh", "common.cuh", "kernels.h"],
}
PROFILES = {"gemm": "gemm_tc_kernel_pixart1024_d831.md",
            "attention": "attn_tc_kernel_pixart1024_d831.md"}


def profiled_traffic(kernel: str):
    """DRAM bytes per launch from the committed ncu summary of `kernel`, or
    None when the kernel's sources changed since the counters were taken."""
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2608_29809_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    path = os.path.join(ROOT, "profiles", PROFILES[kernel])
    if not os.path.exists(path):
        return None
    meta = {}
    with open(path) as fh:
        for ln in fh:
            if ":" in ln and not ln.startswith(("|", "#", " ")):
                k, v = ln.split(":", 1)
                meta[k.strip()] = v.strip()
    if meta.get("kernel_source_sha256_16") != h.hexdigest()[:16]:
        return None
    try:
        return int(meta["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return {"hbm_gbs": j["hbm_gbs"], "bf16_tflops": j["bf16_tflops"],
                "bf16_tflops_sustained": j.get("bf16_tflops_sustained", j["bf16_tflops"]),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi samples (200 ms) of SM clock and throttle reasons."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.index)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in out.strip().splitlines():
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------ distributed
def dist_setup(n_gpus: int):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world != n_gpus:
        raise SystemExit(f"--gpus {n_gpus} but WORLD_SIZE={world}; launch N>1 with torchrun")
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank: float, ms: float, world: int) -> float:
    """Whole-job rate of independent replicas (weak scaling): the units all
    ranks processed over the slowest rank's time (ms)."""
    return units_per_rank * world / (max_over_ranks(ms, world) / 1e3)


# ------------------------------------------------------------------ our arm
class Workload:
    def __init__(self, R, d: synth.Dims, seed: int, dev: str, fracs=FRACS):
        self.R, self.d, self.dev = R, d, dev
        w = synth.make_weights(d, seed, device=dev)
        self.model = R.Model(d, w, sessions=1, device=dev)
        ctx, cache = self.model.ctx, self.model.cache
        for t in range(d.timesteps):
            for l in range(d.layers):
                H, K, V = synth.make_cache_slice(d, seed, 0, l, t, device=dev)
                R.rc_cache_fill(cache, 0, l, t, H, K, V)
        torch.cuda.synchronize()
        self.text = synth.make_text(d, seed, dev)
        R.rc_set_text(ctx, cache, 0, self.text)
        tv, ab = synth.ddim_tables(d.timesteps)
        R.rc_set_schedule(ctx, tv, ab)
        self.latent0 = synth.make_latent(d, seed, dev)
        self.latent = self.latent0.clone()
        N = d.tokens
        self.mask = torch.zeros(N, dtype=torch.uint8, device=dev)
        self.idx = torch.zeros(N, dtype=torch.int32, device=dev)
        self.cnt = torch.zeros(1, dtype=torch.int32, device=dev)
        self.ws = torch.empty(R.rc_localize_workspace_size(N, 8), dtype=torch.uint8, device=dev)
        self.sparse = np.full(d.timesteps, R.RC_MODE_SPARSE, np.uint8)
        self.dilation = 0
        self.scores = {}
        for f in fracs:
            blobs = synth.ellipse_blobs(d, seed, f)
            A, ids = synth.indicator_scores(d, blobs, seed)
            self.scores[f] = (torch.from_numpy(A).to(dev), ids, A)

    def localize(self, f, A=None, ids=None):
        d = self.d
        if ids is None:
            A_dev, ids, _ = self.scores[f]
            A = A_dev if A is None else A
        self.R.rc_localize_mask(A, 1, d.tokens, d.text_len, d.grid_h, d.grid_w, ids, 0.5,
                                self.dilation, self.mask, self.idx, self.cnt, self.ws)

    def step(self, i, f):
        t = i % self.d.timesteps
        if t == 0:
            self.latent.copy_(self.latent0)
        self.localize(f)
        self.R.rc_step(self.model.ctx, self.model.cache, 0, self.latent, t, self.sparse, self.idx,
                       -1, self.cnt)

    def make_graphs(self):
        """One CUDA graph of rc_step per timestep, SPARSE over the localisation
        buffers (their contents are read at each replay), and one DENSE."""
        R, d = self.R, self.d
        dense = np.full(d.timesteps, R.RC_MODE_DENSE, np.uint8)
        self.graphs = [R.rc_step_graph_create(self.model.ctx, self.model.cache, 0, self.latent,
                                              t, self.sparse, self.idx, -1, self.cnt)
                       for t in range(d.timesteps)]
        self.dense_graphs = [R.rc_step_graph_create(self.model.ctx, self.model.cache, 0,
                                                    self.latent, t, dense, None, 0, None)
                             for t in range(d.timesteps)]

    def free_graphs(self):
        for g in self.graphs + self.dense_graphs:
            self.R.rc_graph_destroy(g)
        self.graphs, self.dense_graphs = [], []

    def gstep(self, i, f):
        t = i % self.d.timesteps
        if t == 0:
            self.latent.copy_(self.latent0)
        self.localize(f)
        self.R.rc_graph_launch(self.graphs[t])

    def gstep_dense(self, i):
        t = i % self.d.timesteps
        if t == 0:
            self.latent.copy_(self.latent0)
        self.R.rc_graph_launch(self.dense_graphs[t])

    def step_dense(self, i):
        t = i % self.d.timesteps
        if t == 0:
            self.latent.copy_(self.latent0)
        self.R.rc_step_dense(self.model.ctx, self.model.cache, 0, self.latent, t)

    def step_capture(self, i):
        """A DENSE step that also captures the localisation scores of the
        headline mask's delta tokens (the first step of an editing turn)."""
        t = i % self.d.timesteps
        if t == 0:
            self.latent.copy_(self.latent0)
        if not hasattr(self, "cap_scores"):
            self.cap_scores = torch.empty(self.d.tokens, self.d.text_len, device=self.dev)
        ids = self.scores[HEADLINE][1]
        self.R.rc_step_capture(self.model.ctx, self.model.cache, 0, self.latent, t, ids,
                               self.cap_scores)


    def host_tier_rate(self, K, W, world, seed=SEED):
        R, d, dev = self.R, self.d, self.dev
        hc = R.rc_cache_create_host(self.model.ctx, 1)
        try:
            for t in range(d.timesteps):
                for l in range(d.layers):
                    H, K_, V = synth.make_cache_slice(d, seed, 0, l, t, device=dev)
                    R.rc_cache_fill(hc, 0, l, t, H, K_, V)
            R.rc_set_text(self.model.ctx, hc, 0, self.text)
            torch.cuda.synchronize()

            def step(i):
                t = i % d.timesteps
                if t == 0:
                    self.latent.copy_(self.latent0)
                self.localize(HEADLINE)
                R.rc_step(self.model.ctx, hc, 0, self.latent, t, self.sparse, self.idx, -1,
                          self.cnt)

            m = timed(step, K, W, world)
            R.rc_sync(self.model.ctx)
            thp = thp_state()  # while the pool is still mapped
        finally:
            R.rc_cache_destroy(hc)
        slot = d.tokens * d.hidden * 2
        h2d = (2 * (d.layers - 1) + 3) * slot
        return {"steps_per_s": round(job_rate(K, m, world), 3),
                "pool_bytes": d.timesteps * d.layers * 3 * slot,
                "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": 3 * int(self.cnt.item()) * d.hidden * 2 * d.layers,
                "h2d_gbs_over_step": round(h2d / (m / K / 1e3) / 1e9, 1),
                "step": "rc_localize_mask + rc_step(SPARSE) on rc_cache_create_host",
                "thp": thp}


def thp_state():
    """Transparent-huge-page mode of the host and the anonymous huge pages in
    use (read while the host-tier pool is mapped): the host tier's rate
    depends on whether its pool got huge pages."""
    out = {}
    for k in ("enabled", "defrag"):
        try:
            with open(f"/sys/kernel/mm/transparent_hugepage/{k}") as f:
                out[k] = f.read().strip()
        except OSError:
            out[k] = None
    try:
        with open("/proc/meminfo") as f:
            for ln in f:
                if ln.startswith(("AnonHugePages:", "Hugepagesize:")):
                    k, v = ln.split(":", 1)
                    out[k] = v.strip()
    except OSError:
        pass
    return out


def rate_batched(R, args, world, dev, K, W, n=8):
    """Batched serving: n concurrent 512 px sessions (1024 tokens, 28 blocks),
    each at its own timestep with its own text and a ragged dirty fraction
    from U(2 %, 35 %); one rc_step_batched per step against n rc_step calls."""
    from dataclasses import replace
    d = replace(synth.PIXART_512, timesteps=args.resident_steps)
    seed = SEED + 11
    w = synth.make_weights(d, seed, device=dev)
    model = R.Model(d, w, sessions=n, device=dev, max_batch=n)
    try:
        for s in range(n):
            R.rc_set_text(model.ctx, model.cache, s, synth.make_text(d, seed + s, dev))
            for t in range(d.timesteps):
                for l in range(d.layers):
                    H, K_, V = synth.make_cache_slice(d, seed, s, l, t, device=dev)
                    R.rc_cache_fill(model.cache, s, l, t, H, K_, V)
        tv, ab = synth.ddim_tables(d.timesteps)
        R.rc_set_schedule(model.ctx, tv, ab)
        rng = np.random.default_rng(seed)
        fracs = rng.uniform(0.02, 0.35, size=n)
        N = d.tokens
        idx, cnt, lat0, lat = [], [], [], []
        for s in range(n):
            blobs = synth.ellipse_blobs(d, seed + s, float(fracs[s]))
            A, ids = synth.indicator_scores(d, blobs, seed + s)
            ws = torch.empty(R.rc_localize_workspace_size(N, len(ids)), dtype=torch.uint8,
                             device=dev)
            mask = torch.zeros(N, dtype=torch.uint8, device=dev)
            idx.append(torch.zeros(N, dtype=torch.int32, device=dev))
            cnt.append(torch.zeros(1, dtype=torch.int32, device=dev))
            R.rc_localize_mask(torch.from_numpy(A).to(dev), A.shape[0], N, A.shape[2], d.grid_h,
                               d.grid_w, ids, 0.5, 0, mask, idx[s], cnt[s], ws)
            lat0.append(synth.make_latent(d, seed + s, dev))
            lat.append(lat0[s].clone())
        torch.cuda.synchronize()
        dirty = [int(c.item()) for c in cnt]
        sparse = np.full(d.timesteps, R.RC_MODE_SPARSE, np.uint8)

        def items(i):
            out = []
            for s in range(n):
                t = (i + 3 * s) % d.timesteps
                if t == 0:
                    lat[s].copy_(lat0[s])
                out.append(dict(session=s, latent=lat[s], t=t, mode=R.RC_MODE_SPARSE,
                                dirty_idx=idx[s], D=-1, dirty_count=cnt[s]))
            return out

        def batched(i):
            R.rc_step_batched(model.ctx, model.cache, items(i))

        def one_by_one(i):
            for it in items(i):
                R.rc_step(model.ctx, model.cache, it["session"], it["latent"], it["t"], sparse,
                          it["dirty_idx"], -1, it["dirty_count"])

        k = max(2, K // 2)
        m = timed(batched, k, W, world)
        rate_b = job_rate(n * k, m, world)
        m = timed(one_by_one, k, W, world)
        rate_1 = job_rate(n * k, m, world)
        R.rc_sync(model.ctx)
    finally:
        model.close()
    return {"workload": f"batched serving: {n} sessions x pixart-alpha-512px ({d.tokens} tokens, "
                        f"{d.layers} blocks, {d.timesteps} timesteps)",
            "dirty_tokens": dirty, "session_steps_per_s": round(rate_b, 3),
            "session_steps_per_s_one_by_one": round(rate_1, 3),
            "speedup_of_batching": round(rate_b / rate_1, 3),
            "step": "rc_step_batched over all sessions (vs one rc_step per session)"}


def pct(xs, q):
    """q-th percentile (nearest rank) of a list."""
    xs = sorted(xs)
    return xs[min(len(xs) - 1, max(0, int(np.ceil(q / 100.0 * len(xs))) - 1))]


def rate_server(R, args, world, dev, n=8, turns_per_session=2):
    """Persistent serving through the cross-session scheduler (rc_server_*):
    n 512 px sessions (1024 tokens, 28 blocks), turns arriving on a seeded
    schedule (exponential gaps, mean 2.5 ticks; a session's next turn queues
    until its previous one ends), each turn = T SPARSE steps over the
    session's own ragged region (dirty fraction from U(2 %, 35 %)).  Every
    tick is one rc_server_tick (one batched step over up to n running turns);
    CUDA events around each tick give the per-tick latency, and a turn's
    latency runs from the start of the tick at which it arrived to the end of
    its last tick."""
    from dataclasses import replace
    d = replace(synth.PIXART_512, timesteps=args.resident_steps)
    T = d.timesteps
    seed = SEED + 13
    w = synth.make_weights(d, seed, device=dev)
    model = R.Model(d, w, sessions=n, device=dev, max_batch=n)
    srv = None
    try:
        for s in range(n):
            R.rc_set_text(model.ctx, model.cache, s, synth.make_text(d, seed + s, dev))
            for t in range(T):
                for l in range(d.layers):
                    H, K_, V = synth.make_cache_slice(d, seed, s, l, t, device=dev)
                    R.rc_cache_fill(model.cache, s, l, t, H, K_, V)
        tv, ab = synth.ddim_tables(T)
        R.rc_set_schedule(model.ctx, tv, ab)
        rng = np.random.default_rng(seed)
        fracs = rng.uniform(0.02, 0.35, size=n)
        N = d.tokens
        idx, cnt, lat0, lat = [], [], [], []
        for s in range(n):
            blobs = synth.ellipse_blobs(d, seed + s, float(fracs[s]))
            A, ids = synth.indicator_scores(d, blobs, seed + s)
            ws = torch.empty(R.rc_localize_workspace_size(N, len(ids)), dtype=torch.uint8,
                             device=dev)
            mask = torch.zeros(N, dtype=torch.uint8, device=dev)
            idx.append(torch.zeros(N, dtype=torch.int32, device=dev))
            cnt.append(torch.zeros(1, dtype=torch.int32, device=dev))
            R.rc_localize_mask(torch.from_numpy(A).to(dev), A.shape[0], N, A.shape[2], d.grid_h,
                               d.grid_w, ids, 0.5, 0, mask, idx[s], cnt[s], ws)
            lat0.append(synth.make_latent(d, seed + s, dev))
            lat.append(lat0[s].clone())
        torch.cuda.synchronize()
        dirty = [int(c.item()) for c in cnt]
        sparse = np.full(T, R.RC_MODE_SPARSE, np.uint8)
        # seeded arrivals: (tick, session), sessions in turn order
        gaps = rng.exponential(2.5, size=n * turns_per_session)
        arrivals = [(int(np.floor(g)), k % n) for k, g in enumerate(np.cumsum(gaps) - gaps[0])]
        srv = R.rc_server_create(model.ctx, model.cache, n)

        def run(record):
            pending = list(arrivals)
            waiting, started, done = [], {}, []
            ev = []
            tick = 0
            while pending or waiting or R.rc_server_running(srv):
                while pending and pending[0][0] <= tick:
                    waiting.append(pending.pop(0))
                for a in list(waiting):
                    s = a[1]
                    if R.rc_server_state(srv, s) < 0:
                        lat[s].copy_(lat0[s])
                        R.rc_server_admit(srv, s, lat[s], sparse, idx[s], -1, cnt[s])
                        started[s] = (a[0], tick)
                        waiting.remove(a)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                stepped = R.rc_server_tick(srv, n)
                e1.record()
                ev.append((e0, e1, stepped))
                for s in list(started):
                    if R.rc_server_state(srv, s) < 0 and s in stepped:
                        done.append((started.pop(s), tick))
                tick += 1
            torch.cuda.synchronize()
            if not record:
                return None
            tick_ms = [a.elapsed_time(b) for a, b, st in ev if st]
            t0 = ev[0][0]
            start_of = [t0.elapsed_time(a) for a, _, _ in ev]
            end_of = [t0.elapsed_time(b) for _, b, _ in ev]
            turn_ms = [end_of[e] - start_of[a_tick] for (a_tick, _), e in done]
            total_ms = end_of[-1]
            steps = sum(len(st) for _, _, st in ev)
            return tick_ms, turn_ms, total_ms, steps, len(ev)

        run(False)  # warm-up pass (tensor maps, tables)
        tick_ms, turn_ms, total_ms, steps, ticks = run(True)
        R.rc_sync(model.ctx)
    finally:
        if srv:
            R.rc_server_destroy(srv)
        model.close()
    return {"workload": f"persistent serving: {n} sessions x pixart-alpha-512px ({d.tokens} "
                        f"tokens, {d.layers} blocks, {T} timesteps), "
                        f"{n * turns_per_session} turns on a seeded arrival schedule",
            "dirty_tokens": dirty, "turns": len(turn_ms), "ticks": ticks,
            "session_steps": steps,
            "session_steps_per_s": round(steps / (total_ms / 1e3) * world, 3),
            "tick_ms_p50": round(pct(tick_ms, 50), 3), "tick_ms_p99": round(pct(tick_ms, 99), 3),
            "turn_ms_p50": round(pct(turn_ms, 50), 2), "turn_ms_p99": round(pct(turn_ms, 99), 2),
            "step": "rc_server_tick: one rc_step_batched over up to 8 running turns, "
                    "least recently stepped first"}


def rate_session(wl, R, d, seed, turns=5):
    """Multi-turn editing session at 1024 px (4096 tokens, 28 blocks, T = 20),
    the cache updated in place from turn to turn.  Per turn: a new prompt
    (rc_set_text), a seeded similarity s ~ U(0, 1) giving k = 2 (1 + min(3,
    floor(4 (1 - s)))) fully recomputed leading steps -- the first one
    rc_step_capture (DENSE + the delta tokens' scores), the rest DENSE graphs
    -- then the turn's region (an ellipse map of f ~ U(5 %, 20 %): the
    random-init model's own attention is not localised) through
    rc_localize_mask, and SPARSE graphs for steps k .. T-1.  A second
    session runs the paper's Eq. 2 schedule instead: T_reuse = floor(0.2 T)
    REUSE steps, then the region localised from the cached states
    (rc_localize_scores + rc_localize_mask) and SPARSE steps."""
    T = d.timesteps
    rng = np.random.default_rng(seed)
    sims = rng.uniform(0.0, 1.0, size=turns)
    fr = rng.uniform(0.05, 0.20, size=turns)
    plans = []
    for j in range(turns):
        blobs = synth.ellipse_blobs(d, seed + 10 * j, float(fr[j]))
        A, ids = synth.indicator_scores(d, blobs, seed + 10 * j)
        # the workload's leading dense steps: k = 2 (1 + min(3, floor(4 (1 - s))))
        k = 2 * (1 + min(3, int(np.floor(4.0 * (1.0 - float(sims[j]))))))
        plans.append((k, torch.from_numpy(A).to(wl.dev), ids,
                      synth.make_text(d, seed + 10 * j, wl.dev)))
    cap = torch.empty(d.tokens, d.text_len, device=wl.dev)
    ctx, cache = wl.model.ctx, wl.model.cache

    def first_k():
        ks = []
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        for k, A, ids, text in plans:
            R.rc_set_text(ctx, cache, 0, text)
            wl.latent.copy_(wl.latent0)
            R.rc_step_capture(ctx, cache, 0, wl.latent, 0, ids[:8], cap)
            for t in range(1, k):
                R.rc_graph_launch(wl.dense_graphs[t])
            wl.localize(None, A=A, ids=ids)
            for t in range(k, T):
                R.rc_graph_launch(wl.graphs[t])
            ks.append(k)
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1), ks

    lat_scores = torch.empty(d.tokens, d.text_len, device=wl.dev)
    t_reuse = int(np.floor(0.2 * T))
    reuse = R.rc_reuse_schedule(0.0, 1.0, T, 0.2)

    def eq2():
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        for k, A, ids, text in plans:
            R.rc_set_text(ctx, cache, 0, text)
            wl.latent.copy_(wl.latent0)
            for t in range(t_reuse):
                R.rc_step(ctx, cache, 0, wl.latent, t, reuse, None, 0, None)
            R.rc_localize_scores(ctx, cache, 0, t_reuse, wl.latent, ids[:8], lat_scores)
            # the region of the random-init model's scores is not compact: the
            # turn's ellipse map stands in for the mask (the score pass is timed)
            wl.localize(None, A=A, ids=ids)
            for t in range(t_reuse, T):
                R.rc_graph_launch(wl.graphs[t])
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1)

    first_k()
    ms, ks = first_k()
    eq2()
    ms_eq2 = eq2()
    steps = turns * T
    return {"workload": f"{turns}-turn editing session, pixart-alpha-1024px ({d.tokens} tokens, "
                        f"{d.layers} blocks, {T} timesteps), cache updated in place",
            "first_k_dense": {"k_per_turn": ks, "session_ms": round(ms, 2),
                              "steps_per_s": round(steps / (ms / 1e3), 3),
                              "step": "rc_set_text, rc_step_capture, k-1 DENSE graphs, "
                                      "rc_localize_mask, T-k SPARSE graphs per turn"},
            "eq2_reuse_then_sparse": {"t_reuse": t_reuse, "session_ms": round(ms_eq2, 2),
                                      "steps_per_s": round(steps / (ms_eq2 / 1e3), 3),
                                      "step": "rc_set_text, T_reuse REUSE steps, "
                                              "rc_localize_scores, rc_localize_mask, "
                                              "T-T_reuse SPARSE graphs per turn"}}


def rate_2048(R, args, world, dev, K, W):
    """Headline-style steps (20 % dirty, graphs) and dense steps of the 2048 px
    model (128 x 128 = 16 384 tokens, all 20 timesteps resident)."""
    from dataclasses import replace
    d = replace(synth.PIXART_2048, timesteps=args.resident_steps)
    wl = Workload(R, d, SEED + 7, dev, fracs=(HEADLINE,))
    try:
        wl.make_graphs()
        k = max(2, K // 4)
        m = timed(lambda i: wl.gstep(i, HEADLINE), k, W, world)
        sparse = job_rate(k, m, world)
        D = int(wl.cnt.item())
        m = timed(wl.gstep_dense, k, min(W, 3), world)
        dense = job_rate(k, m, world)
        R.rc_sync(wl.model.ctx)
        wl.free_graphs()
    finally:
        wl.model.close()
    return {"workload": f"pixart-alpha-2048px: {d.tokens} tokens, {d.layers} blocks, "
                        f"{d.timesteps} timesteps, batch 1",
            "dirty_frac": HEADLINE, "dirty_tokens": D, "steps_per_s": round(sparse, 3),
            "dense_steps_per_s": round(dense, 3), "speedup_vs_dense": round(sparse / dense, 3),
            "cache_bytes": d.timesteps * d.layers * 3 * d.tokens * d.hidden * 2}


def rate_c1(R, world, dev, K, W, seed, with_oracle):
    """One PixArt-alpha block at 256 tokens (16 x 16) on a seeded ~15 % dirty
    rectangle: rc_block_forward_region with the block input restored before
    each launch sequence, blocks/s; beside it the oracle's region_block on
    the same shapes, timed whole on the host cores."""
    d = synth.ONE_BLOCK_256
    w = synth.make_weights(d, seed)
    text = synth.make_text(d, seed)
    mod6 = synth.make_mod6(d, w.layers[0]["table"], seed)
    x0 = synth.make_hidden(d, seed)
    slot = synth.make_cache_slice(d, seed, 0, 0, 0)
    idx = np.flatnonzero(synth.rectangle_mask(d, seed)).astype(np.int32)
    m = R.Model(d, w, device=dev)
    try:
        R.rc_cache_fill(m.cache, 0, 0, 0, *(a.to(dev) for a in slot))
        R.rc_set_text(m.ctx, m.cache, 0, text.to(dev))
        idx_d, mod6_d = torch.from_numpy(idx).to(dev), mod6.to(dev)
        x0_d = x0.to(dev)
        x = x0_d.clone()

        def blk(i):
            x.copy_(x0_d)
            R.rc_block_forward_region(m.ctx, m.cache, 0, 0, 0, x, idx_d, len(idx), None, mod6_d)

        k = 10 * K
        ms = timed(blk, k, W, world)
        R.rc_sync(m.ctx)
    finally:
        m.close()
    out = {"workload": f"one PixArt-alpha block, {d.tokens} tokens ({d.grid_h} x {d.grid_w}), "
                       "bf16 weights and cache, seeded rectangle",
           "dirty_tokens": int(len(idx)), "unit": "blocks/s",
           "blocks_per_s": round(job_rate(k, ms, world), 3),
           "ms_per_block": round(ms / k, 5),
           "timed": "copy of the block input + rc_block_forward_region, CUDA events"}
    if with_oracle:
        import oracle as O
        L64 = {kk: O.to64(v) for kk, v in w.layers[0].items()}
        cache = dict(zip("HKV", (O.to64(a) for a in slot)))
        tkv = O.text_kv(O.to64(text), L64)
        x64, m64 = O.to64(x0)[idx], O.to64(mod6)
        n, t0 = 0, time.perf_counter()
        while n < 3 or time.perf_counter() - t0 < 2.0:
            O.region_block(x64, idx.astype(np.int64), cache, L64, m64, tkv, d.heads)
            n += 1
        sec = (time.perf_counter() - t0) / n
        out["oracle"] = {"value": round(1.0 / sec, 3), "unit": "blocks/s",
                         "cores": os.cpu_count(), "kind": "oracle", "extrapolated": False,
                         "sample": f"{n} whole region blocks, float64 numpy",
                         "seconds_per_block": round(sec, 5)}
    return out


def rate_c2(R, args, world, dev, K, W, seed, with_oracle):
    """Whole steps of the 28-block model at 512 px (32 x 32 = 1024 tokens, all
    timesteps resident): localisation on a seeded score map with 3-8 delta
    tokens (threshold 0.5, one token of dilation) + the CUDA graph of rc_step
    (SPARSE), and the dense path; beside them one whole oracle step
    (localisation, 28 region blocks, final layer and DDIM update)."""
    from dataclasses import replace
    d = replace(synth.PIXART_512, timesteps=args.resident_steps)
    A, ids = synth.blob_scores(d, seed)
    wl = Workload(R, d, seed, dev, fracs=())
    try:
        wl.scores["c2"] = (torch.from_numpy(A).to(dev), ids, A)
        wl.dilation = 1
        wl.make_graphs()
        ms = timed(lambda i: wl.gstep(i, "c2"), K, W, world)
        sparse = job_rate(K, ms, world)
        D = int(wl.cnt.item())
        m = timed(wl.gstep_dense, K, min(W, 3), world)
        dense = job_rate(K, m, world)
        R.rc_sync(wl.model.ctx)
        wl.free_graphs()
    finally:
        wl.model.close()
    out = {"workload": f"pixart-alpha-512px: {d.tokens} tokens, {d.layers} blocks, "
                       f"{d.timesteps} timesteps, batch 1; dirty set localised from a seeded "
                       f"score map ({len(ids)} delta tokens, threshold 0.5, dilation 1)",
           "dirty_tokens": D, "dirty_frac": round(D / d.tokens, 4),
           "steps_per_s": round(sparse, 3), "ms_per_step": round(ms / K, 4),
           "dense_steps_per_s": round(dense, 3), "speedup_vs_dense": round(sparse / dense, 3)}
    if with_oracle:
        import oracle as O
        w = synth.make_weights(d, seed)
        L64 = [{kk: O.to64(v) for kk, v in L.items()} for L in w.layers]
        G64 = {kk: O.to64(v) for kk, v in w.glob.items()}
        pos = O.to64(w.pos)
        del w
        ctx = O.to64(synth.make_text(d, seed))
        tkv = [O.text_kv(ctx, L) for L in L64]
        t = 5
        cache = [dict(zip("HKV", (O.to64(a) for a in synth.make_cache_slice(d, seed, 0, l, t))))
                 for l in range(d.layers)]
        lat = O.to64(synth.make_latent(d, seed))
        tv, ab = synth.ddim_tables(d.timesteps)
        tv, ab = tv.astype(np.float64), ab.astype(np.float64)
        secs = []
        for _ in range(2):
            t0 = time.perf_counter()
            _, idx = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 1)
            O.step(G64, L64, pos, lat, t, O.MODE_SPARSE, idx, cache, tkv, tv, ab, d.heads,
                   d.grid_h, d.grid_w, d.patch, d.in_ch)
            secs.append(time.perf_counter() - t0)
        sec = min(secs)
        out["oracle"] = {"value": round(1.0 / sec, 5), "unit": UNIT, "cores": os.cpu_count(),
                         "kind": "oracle", "extrapolated": False, "dirty_tokens": int(len(idx)),
                         "sample": "2 whole steps (localisation, 28 region blocks, final "
                                   "layer, DDIM update), float64 numpy; the faster one",
                         "seconds_per_step": round(sec, 3)}
    return out


def kernel_rooflines(d, D, gemm_each, att_each, peak):
    """GEMM and attention rooflines of one probe pass: algorithmic FLOPs of
    D dirty rows per launch over the CUDA-event launch durations."""
    gemm_ms, gemm_n = sum(gemm_each), len(gemm_each)
    att_ms, att_n = sum(att_each), len(att_each)
    steps = att_n / (2 * d.layers)
    per_block = int(round(gemm_n / (steps * d.layers)))  # 5: cross-query folded, 6: not
    folded = per_block == 5
    lin = linear_flops_per_token_block(d, folded)
    lin_flops_launch = lin * D / per_block
    gemm_tflops = lin * D * d.layers * steps / (gemm_ms / 1e3) / 1e12
    att_tflops = (attn_flops_per_token_block(d, folded) * D * d.layers * steps /
                  (att_ms / 1e3) / 1e12)
    roofline = {"bound": "tensor", "achieved": round(gemm_tflops, 2), "peak": peak,
                "unit": "TFLOP/s", "frac": round(gemm_tflops / peak, 4),
                "traffic": profiled_traffic("gemm"),
                "kernel": "gemm (QKV, out, [cross-q,] cross-out, fc1, fc2 of every block)",
                "launches": gemm_n, "avg_launch_ms": round(gemm_ms / max(gemm_n, 1), 5),
                "flops_per_launch": lin_flops_launch,
                "cross_query_folded_into_attention": folded}
    roof_att = {"bound": "tensor", "achieved": round(att_tflops, 2), "peak": peak,
                "traffic": profiled_traffic("attention"),
                "unit": "TFLOP/s", "frac": round(att_tflops / peak, 4), "launches": att_n,
                "avg_launch_ms": round(att_ms / max(att_n, 1), 5)}
    # per-launch breakdown: launches come in block order (GEMMs: QKV, out,
    # cross-q, cross-out, fc1, fc2; attention: self, cross)
    h, F = d.hidden, d.mlp
    gemm_shapes = [("qkv", 3 * h, h), ("out", h, h)] + ([] if folded else [("cross_q", h, h)]) + [
        ("cross_out", h, h), ("fc1", F, h), ("fc2", h, F)]
    per_gemm = {}
    for j, (name, n_, k_) in enumerate(gemm_shapes):
        ts = gemm_each[j::per_block]
        us = 1e3 * sum(ts) / max(len(ts), 1)
        per_gemm[name] = {"shape": [D, n_, k_], "avg_us": round(us, 2),
                          "tflops": round(2.0 * D * n_ * k_ / (us * 1e-6) / 1e12, 1)}
    per_attn = {}
    for j, (name, nk) in enumerate([("self", d.tokens), ("cross", d.text_len)]):
        ts = att_each[j::2]
        us = 1e3 * sum(ts) / max(len(ts), 1)
        fl = 4.0 * D * nk * h + (2.0 * D * h * h if name == "cross" and folded else 0.0)
        per_attn[name] = {"queries": D, "keys": nk, "avg_us": round(us, 2),
                          "tflops": round(fl / (us * 1e-6) / 1e12, 1)}
    roofline["per_gemm"] = per_gemm
    roof_att["per_launch"] = per_attn
    return roofline, roof_att


def timed(fn, K, W, world):
    for i in range(W):
        fn(i)
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record()
    for i in range(K):
        fn(W + i)
    e.record()
    torch.cuda.synchronize()
    barrier(world)
    return s.elapsed_time(e)  # ms


def run_ours(args, world, rank, local):
    from paper_2608_29809_gb300 import regioncache as R
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    from dataclasses import replace
    d = replace(synth.PIXART_1024, timesteps=args.resident_steps)
    K, W = args.steps, args.warmup
    wl = Workload(R, d, SEED + rank, dev)
    peaks = load_peaks()
    if args.dense_only:
        m = timed(wl.step_dense, K, W, world)
        R.rc_sync(wl.model.ctx)
        if rank == 0:
            print(json.dumps({"metric": METRIC, "dense_only": True, "unit": UNIT,
                              "dense_steps_per_s": round(job_rate(K, m, world), 3),
                              "steps": K, "warmup": W}), flush=True)
        wl.model.close()
        return

    # headline: 20 % dirty, each step = localisation + the CUDA graph of
    # rc_step for the timestep; clock sampler running, no probe events
    wl.make_graphs()
    for i in range(W):
        wl.gstep(i, HEADLINE)
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    n0 = R.rc_launch_count()
    ms = timed(lambda i: wl.gstep(i, HEADLINE), K, 0, world)
    launches = R.rc_launch_count() - n0
    clk = clocks.stop()
    R.rc_sync(wl.model.ctx)
    D = int(wl.cnt.item())
    ms_max = max_over_ranks(ms, world)
    value = K * world / (ms_max / 1e3)
    # the same steps issued launch by launch (rc_step)
    m = timed(lambda i: wl.step(i, HEADLINE), K, W, world)
    direct = job_rate(K, m, world)
    if args.quick:
        if rank == 0:
            print(json.dumps({"metric": METRIC, "value": round(value, 3), "unit": UNIT,
                              "quick": True, "ms_per_step": round(ms_max / K, 4),
                              "direct_steps_per_s": round(direct, 3),
                              "dirty_tokens": D, "gpu_launches": int(launches)}), flush=True)
        wl.free_graphs()
        wl.model.close()
        return

    # kernel-level timing: the same K steps again, once with CUDA events around
    # every GEMM launch and once around every attention launch (events on the
    # launching stream; they serialise the launches they bracket, so these
    # passes are kept out of the headline)
    def probe(which, per_step, fn, nsteps):
        cap = nsteps * d.layers * per_step
        R.rc_probe_enable(wl.model.ctx, which, cap)
        timed(fn, nsteps, 0, 1)
        each = R.rc_probe_read_each(wl.model.ctx, cap)
        R.rc_probe_enable(wl.model.ctx, R.RC_PROBE_OFF, 0)
        return each

    gemm_each = probe(R.RC_PROBE_GEMM, 5, lambda i: wl.step(i, HEADLINE), K)
    att_each = probe(R.RC_PROBE_ATTENTION, 2, lambda i: wl.step(i, HEADLINE), K)
    ln_each = probe(R.RC_PROBE_LN, 2, lambda i: wl.step(i, HEADLINE), K)
    # the same kernels on all 4096 rows (the dense step)
    Kd = max(2, K // 4)
    # 6 GEMMs per block here: at 4096 host-known rows the cross-query projection
    # runs as its own paired GEMM instead of inside the cross-attention kernel
    gemm_each_d = probe(R.RC_PROBE_GEMM, 6, wl.step_dense, Kd)
    att_each_d = probe(R.RC_PROBE_ATTENTION, 2, wl.step_dense, Kd)

    # the same launch-by-launch steps with the gated residuals on whole tiles
    # (rc_set_deterministic: bit-reproducible results)
    R.rc_set_deterministic(wl.model.ctx, True)
    m = timed(lambda i: wl.step(i, HEADLINE), K, W, world)
    R.rc_set_deterministic(wl.model.ctx, False)
    direct_det = job_rate(K, m, world)

    # sweep and dense baseline (graphs, like the headline)
    sweep, dirty = {}, {}
    for f in FRACS:
        m = timed(lambda i, f=f: wl.gstep(i, f), K, W, world)
        sweep[f"{f:.2f}"] = round(job_rate(K, m, world), 3)
        dirty[f"{f:.2f}"] = int(wl.cnt.item())
    m = timed(wl.gstep_dense, max(2, K // 2), min(W, 3), world)
    dense = job_rate(max(2, K // 2), m, world)
    m = timed(wl.step_capture, max(2, K // 2), min(W, 3), world)
    capture = job_rate(max(2, K // 2), m, world)
    R.rc_sync(wl.model.ctx)

    # batched serving of 8 concurrent 512 px sessions
    batch = None
    if not args.no_batched:
        batch = rate_batched(R, args, world, dev, K, W)

    # persistent serving: turns arriving on a seeded schedule, through the
    # cross-session scheduler
    server = None
    if not args.no_server:
        server = rate_server(R, args, world, dev)

    # the same step at 2048 px (16 384 tokens, 63.4 GB cache resident)
    big = None
    if not args.no_2048:
        big = rate_2048(R, args, world, dev, K, W)

    # the two smaller configurations: one block at 256 tokens, whole steps at
    # 512 px, each with the oracle timed whole beside it
    small = None
    if not args.no_small:
        with_oracle = rank == 0 and world == 1 and not args.no_cpu_baseline
        small = {"c1_one_block_256": rate_c1(R, world, dev, K, W, SEED + 11, with_oracle),
                 "c2_512px": rate_c2(R, args, world, dev, K, W, SEED + 13, with_oracle)}

    # the same headline steps on a host-tier cache (pinned host pool, each
    # layer's K, V streamed into HBM windows while the previous layer runs)
    host_tier = None
    if not args.no_host_tier:
        host_tier = wl.host_tier_rate(K, W, world)

    # end to end through the C ABI with host buffers: per step the score map
    # and the latent go host -> device, the updated latent comes back
    A_host = torch.from_numpy(wl.scores[HEADLINE][2]).pin_memory()
    lat_host = wl.latent0.cpu().pin_memory()
    A_dev = torch.empty_like(A_host, device=dev)

    def e2e_step(i):
        t = i % d.timesteps
        if t == 0:
            lat_host.copy_(wl.latent0.cpu())
        A_dev.copy_(A_host, non_blocking=True)
        wl.latent.copy_(lat_host, non_blocking=True)
        wl.localize(HEADLINE, A_dev)
        R.rc_graph_launch(wl.graphs[t])
        lat_host.copy_(wl.latent, non_blocking=True)
        torch.cuda.current_stream().synchronize()

    for i in range(W):
        e2e_step(i)
    barrier(world)
    t0 = time.perf_counter()
    for i in range(K):
        e2e_step(i)
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)
    barrier(world)
    e2e = {"value": round(K * world / e2e_s, 3), "unit": UNIT,
           "h2d_bytes_per_step": int(A_host.numel() * 4 + lat_host.numel() * 4),
           "d2h_bytes_per_step": int(lat_host.numel() * 4)}

    # the 5-turn editing session at size (first k dense, then sparse), and
    # the same turns under Eq. 2 with the region localised from the cache
    session = None
    if not args.no_session:
        session = rate_session(wl, R, d, SEED + 17)

    # burst peak: each launch is timed on its own (tens of microseconds), far
    # shorter than the seconds-long loop the sustained figure needs
    peak = peaks["bf16_tflops"]
    roofline, roof_att = kernel_rooflines(d, D, gemm_each, att_each, peak)
    roofline.update({"timing": "CUDA events around each launch, separate pass of the same "
                               "K steps",
                     "peak_source": f"{peaks['source']} bf16_tflops (burst)"})
    roof_dense, roof_att_dense = kernel_rooflines(d, d.tokens, gemm_each_d, att_each_d, peak)
    # LayerNorm-modulation launches (HBM-bound class): bytes per launch are
    # the D rows read as f32 and written as bf16, plus the bf16 H rows the
    # first LN of a block stores into the cache
    ln_msa, ln_mlp = ln_each[0::2], ln_each[1::2]
    ln_bytes = {"msa": 8.0 * D * d.hidden, "mlp": 6.0 * D * d.hidden}
    ln_us = {"msa": 1e3 * sum(ln_msa) / max(len(ln_msa), 1),
             "mlp": 1e3 * sum(ln_mlp) / max(len(ln_mlp), 1)}
    ln_gbs = (ln_bytes["msa"] * len(ln_msa) + ln_bytes["mlp"] * len(ln_mlp)) / (
        sum(ln_each) / 1e3) / 1e9
    roof_ln = {"bound": "hbm", "achieved": round(ln_gbs, 1), "peak": peaks["hbm_gbs"],
               "unit": "GB/s", "frac": round(ln_gbs / peaks["hbm_gbs"], 4), "traffic": None,
               "launches": len(ln_each), "avg_us": {k: round(v, 2) for k, v in ln_us.items()},
               "bytes_per_launch": ln_bytes}
    out = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world,
        "steps": K, "warmup": W, "ms_per_step": round(ms_max / K, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: seeded random-init PixArt-alpha-shaped weights, cache, text, "
                "latent and ellipse-blob score maps",
        "config": {"workload": WORKLOAD, "tokens": d.tokens, "dirty_frac": HEADLINE,
                   "dirty_tokens": D, "layers": d.layers, "timesteps": d.timesteps,
                   "sessions_per_gpu": 1, "parallelism": "replicas" if world > 1 else "single",
                   "l2": L2_NOTE,
                   "step": "rc_localize_mask + rc_graph_launch (CUDA graph of rc_step SPARSE, "
                           "dirty list read from the localisation buffers)"},
        "sweep_steps_per_s": sweep, "sweep_dirty_tokens": dirty,
        "dense_steps_per_s": round(dense, 3),
        "dense_capture_steps_per_s": round(capture, 3),
        "host_tier": host_tier,
        "pixart2048": big,
        "small_configs": small,
        "batched_serving": batch,
        "persistent_serving": server,
        "editing_session": session,
        "direct_steps_per_s": round(direct, 3),
        "deterministic_direct_steps_per_s": round(direct_det, 3),
        "speedup_vs_dense": {k: round(v / dense, 3) for k, v in sweep.items()},
        "roofline": roofline, "roofline_attention": roof_att,
        "roofline_dense": {"rows": d.tokens, "gemm": roof_dense, "attention": roof_att_dense},
        "roofline_ln": roof_ln,
        "e2e": e2e, "gpu_launches": int(launches),
        "launches_per_step": round(launches / K, 2), "clocks": clk,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(d, SEED, HEADLINE, layers_sample=args.cpu_layers)
    if rank == 0:
        print(json.dumps(out), flush=True)
    wl.free_graphs()
    wl.model.close()


# ------------------------------------------------------------- oracle arm
def oracle_sample(d: synth.Dims, seed: int, f: float, layers_sample: int):
    """Oracle inputs for the first `layers_sample` blocks of the workload."""
    import oracle as O
    from dataclasses import replace
    ds = replace(d, layers=layers_sample)
    w = synth.make_weights(ds, seed)
    layers = [{k: O.to64(v) for k, v in L.items()} for L in w.layers]
    G = {k: O.to64(v) for k, v in w.glob.items()}
    pos = O.to64(w.pos)
    ctx = O.to64(synth.make_text(d, seed))
    tkv = [O.text_kv(ctx, L) for L in layers]
    cache = [dict(zip("HKV", (O.to64(a) for a in synth.make_cache_slice(d, seed, 0, l, 0))))
             for l in range(layers_sample)]
    blobs = synth.ellipse_blobs(d, seed, f)
    A, ids = synth.indicator_scores(d, blobs, seed)
    lat = O.to64(synth.make_latent(d, seed))
    return O, ds, layers, G, pos, tkv, cache, A, ids, lat


def cpu_baseline(d, seed, f, layers_sample=2):
    """The oracle, as it stands, on the host cores: localisation, `layers_sample`
    region blocks and the final layer of one step of the headline workload,
    scaled to a full 28-block step."""
    O, ds, layers, G, pos, tkv, cache, A, ids, lat = oracle_sample(d, seed, f, layers_sample)
    t0 = time.perf_counter()
    _, idx = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 0)
    t_loc = time.perf_counter() - t0
    temb = O.t_embed(999.0, G)
    tb = O.t_block(temb, G)
    x = O.patch_embed(lat, idx, G, pos, d.patch)
    t0 = time.perf_counter()
    for l in range(layers_sample):
        _, x = O.region_block(x, idx, cache[l], layers[l], layers[l]["table"] + tb, tkv[l],
                              d.heads)
    t_blk = (time.perf_counter() - t0) / layers_sample
    t0 = time.perf_counter()
    eps = O.final_layer(cache[-1]["H"], temb, G, d.grid_h, d.grid_w, d.patch, d.in_ch)
    O.ddim_update(lat, eps, 0.5, 0.6)
    t_fin = time.perf_counter() - t0
    step_s = t_loc + d.layers * t_blk + t_fin
    return {"value": round(1.0 / step_s, 6), "unit": UNIT, "cores": os.cpu_count(),
            "kind": "oracle", "extrapolated": True,
            "sample": f"one step of the headline workload ({int(f * 100)} % dirty, D={len(idx)}) "
                      f"timed as localisation + {layers_sample} of {d.layers} region blocks "
                      f"(scaled x{d.layers}/{layers_sample}) + final layer; float64 numpy",
            "seconds_per_step": round(step_s, 3)}


def run_reference(args, world, rank):
    if rank != 0:
        return
    d = synth.PIXART_1024
    layers_sample = 2
    O, ds, layers, G, pos, tkv, cache, A, ids, lat = oracle_sample(d, SEED, HEADLINE,
                                                                   layers_sample)
    t0 = time.perf_counter()
    _, idx = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 0)
    temb = O.t_embed(999.0, G)
    tb = O.t_block(temb, G)
    x = O.patch_embed(lat, idx, G, pos, d.patch)
    eps = O.final_layer(cache[-1]["H"], temb, G, d.grid_h, d.grid_w, d.patch, d.in_ch)
    O.ddim_update(lat, eps, 0.5, 0.6)
    t_fixed = time.perf_counter() - t0

    def one(i):
        l = i % layers_sample
        s = time.perf_counter()
        O.region_block(x, idx, cache[l], layers[l], layers[l]["table"] + tb, tkv[l], d.heads)
        return time.perf_counter() - s

    for i in range(args.warmup):
        one(i)
    ts = [one(i) for i in range(args.steps)]
    block_s = sum(ts) / len(ts)
    step_s = t_fixed + d.layers * block_s
    v = 1.0 / step_s
    sample = (f"each timed step is ONE of the {d.layers} oracle region blocks of a headline step "
              f"({int(HEADLINE * 100)} % dirty, D={len(idx)}; blocks {layers_sample} apart in "
              f"weights and cache); value = 1 / ({d.layers} x mean block time + localisation + "
              f"final layer), extrapolated to whole steps")
    # "steps" / "ms_per_step" describe what was timed (blocks); the value is
    # the extrapolated whole-step rate
    out = {"metric": METRIC, "value": round(v, 6), "unit": UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(block_s * 1e3, 3),
           "timed_unit": f"one region block (1/{d.layers} of a step)", "extrapolated": True,
           "ms_per_whole_step": round(step_s * 1e3, 3),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference",
           "config": {"workload": WORKLOAD, "tokens": d.tokens, "dirty_frac": HEADLINE,
                      "dirty_tokens": int(len(idx)), "layers": d.layers,
                      "timesteps": d.timesteps},
           "cpu_baseline": {"value": round(v, 6), "unit": UNIT, "cores": os.cpu_count(),
                            "kind": "oracle", "sample": sample, "extrapolated": True},
           "e2e": {"value": round(v, 6), "unit": UNIT, "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-layers", type=int, default=2)
    ap.add_argument("--quick", action="store_true",
                    help="headline only: no attention probe, sweep, dense, e2e or cpu baseline")
    ap.add_argument("--no-batched", action="store_true",
                    help="skip the batched-serving measurement (8 x 512 px sessions, 32 GB)")
    ap.add_argument("--no-2048", action="store_true",
                    help="skip the 2048 px (16 384-token, 63 GB cache) measurement")
    ap.add_argument("--no-host-tier", action="store_true",
                    help="skip the host-tier cache measurement (a pinned host pool)")
    ap.add_argument("--no-server", action="store_true",
                    help="skip the persistent-serving measurement (rc_server, 8 x 512 px)")
    ap.add_argument("--no-small", action="store_true",
                    help="skip the one-block 256-token and 512 px lines")
    ap.add_argument("--no-session", action="store_true",
                    help="skip the 5-turn editing-session measurement")
    ap.add_argument("--dense-only", action="store_true",
                    help="profiling mode: K launch-by-launch DENSE steps of the headline model "
                         "and nothing else (prints one line)")
    ap.add_argument("--resident-steps", type=int, default=20,
                    help="timesteps held in the cache (1 keeps a profiling run to ~2 GB)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        raise SystemExit("--warmup must be >= 3")
    world, rank, local = dist_setup(args.gpus)
    try:
        if args.impl == "reference":
            run_reference(args, world, rank)
        else:
            run_ours(args, world, rank, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
