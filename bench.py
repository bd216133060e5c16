"""Benchmark of the PACE hot path on GB300.

A step is one pass of the whole path over one pool: pool scoring
(pace_score_pool), budget + rejection (pace_select), then the fused LM-head
log-probs, GRPO advantages and clipped surrogate of the accepted rows
(pace_token_logprob).  The headline workload is the largest step that fits one
GPU, the MoE-shaped policy head (1024 trajectories = 128 prompts x 8, lognormal
responses of median 4096 capped at 16384, hidden 2048, vocab 151936, capacity
768): the metric is accepted tokens per second (rows in the loss / step time).
Further line items time the same step on the 7B-shaped math pool and the
multi-turn tool-use pool, pool scoring + selection alone on the sweep pools
(1k, 16k, 128k and 1M trajectories) against HBM bandwidth, prefix rescoring
(Eq. 6) and the LM-head backward.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

With N > 1 (torchrun, one process per GPU) the pool is partitioned by prompt
group across the ranks (each rank holds 1024 trajectories, the whole pool
N x 1024 with capacity N x 768): the ranks score their groups, reject the k
top-scored groups of the whole pool (six all-reduces of a 2048-bin histogram
and one exclusive sum of tie counts) and compute log-probs and loss on their
accepted rows, the loss from one all-reduce of two partial sums; weak scaling,
a barrier around the timed region and the slowest rank's clock.
``--impl reference`` times the CPU oracle on a bounded sample of the same
workload (rank 0 only).
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "moe"
OTHER_WORKLOADS = ("math7b", "multiturn")
PREFIX_WORKLOAD = "math7b"  # prefix rescoring and the backward are timed on the 7B math pool
# DRAM bytes (read + written) per row in the loss of the LM-head kernel (rows read by index),
# by (workload, vocabulary splits), from one-pass ncu captures (dram__bytes_read.sum +
# dram__bytes_write.sum) of the current kernel on the MoE-shaped head.  4 splits: one wave
# of 19,456 rows, 2.589991 GB read + 4.27 MB written; every round of items reads the
# vocabulary once, so the bytes grow with the rows and the wave's figure per row is scaled by
# the launch's rows.  2 splits: a single wave is not proportional to a long launch (the
# clusters of a split drift apart over it), so the figure is one full 3,958,414-row launch,
# 298.063 GB read + 129.3 MB written.  Emptied whenever the kernel changes, until it is
# captured again.  The tag reduction's per tag: 219.96 MB read + 3.12 MB written for the
# 54.93 M tags of the 16k sweep pool (the atomic-free kernel; its reads equal the algorithmic
# bytes, so the figure per tag carries to the larger pools).
LMHEAD_DRAM_BYTES_PER_ROW = {("moe", 4): (2589990656 + 4268800) / 19456,
                             ("moe", 2): (298063478784 + 129295872) / 3958414}
TAG_REDUCE_DRAM_BYTES_PER_TAG = (219963904 + 3123712) / 54929421
SWEEP_N = 1048576
SWEEP_SIZES = (1024, 16384, 131072, SWEEP_N)
METRIC = "accepted tokens/sec (logprob+loss) and % bf16 tensor peak; pool scoring traj/s + HBM GB/s"
UNIT = "tokens/s"


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (getattr(self, "out", "") or "").strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for name, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def _dist():
    from paper_2609_36830_gb300 import replicas
    return replicas.rank_env()


def _make_inputs(seed_offset, device, workload=WORKLOAD):
    """The pool of rank seed_offset (its own seed), its rows and the step's device inputs."""
    from paper_2609_36830_gb300 import pace, replicas, step, workloads
    spec = workloads.SPECS[workload]
    pool = workloads.make_pool(workload, seed=replicas.replica_seed(workload, seed_offset))
    rows = workloads.make_rows(pool)
    H, V = spec.hidden, spec.vocab
    hidden = workloads.bf16_normal_device((rows.n_rows, H), 1.0, pool.seed + 11, device=device)
    # the vocabulary matrix is the same on every rank (the policy's lm_head.weight)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H),
                                     replicas.replica_seed(workload, 0) + 12, device=device)
    behav = workloads.behaviour_logprob(rows, pool.trainer_version, workloads.uniform_center(V),
                                        pool.seed)
    x = step.build_inputs(pool, rows, hidden, w, behav, device=device)
    lp_params = pace.loss_params(eps_low=spec.eps_low, eps_high=spec.eps_high)
    return pool, rows, x, lp_params


def _step_for(x, pool, lp_params, ws, rank, device):
    """One GPU: the whole pool's step.  N ranks: this rank's part of the step over
    the pool partitioned by prompt group (every rank holds pool.n_traj trajectories)."""
    from paper_2609_36830_gb300 import sharded, step
    if ws == 1:
        return step.PaceStep(x, loss_params=lp_params, device=device)
    return sharded.ShardedPaceStep(x, rank * (pool.n_traj // pool.group_size), ws * pool.n_traj,
                                   ws * pool.n_target, loss_params=lp_params, device=device)


def _make_step(seed_offset, device, workload=WORKLOAD):
    pool, rows, x, lp_params = _make_inputs(seed_offset, device, workload)
    return pool, rows, x, _step_for(x, pool, lp_params, 1, 0, device)


class _L2Flush:
    """Evicts L2 (129 MB) between timed calls: writes one 256 MB buffer, then reads a
    second one, so the written lines are also written back before the timed call
    starts instead of being evicted (and charged) inside it."""

    def __init__(self, device):
        import torch
        self.w = torch.empty(256 << 20, dtype=torch.uint8, device=device)
        self.r = torch.ones(64 << 20, dtype=torch.float32, device=device)
        self.sink = torch.empty((), dtype=torch.float32, device=device)

    def __call__(self):
        import torch
        self.w.zero_()
        torch.sum(self.r, dim=0, out=self.sink)


def _sweep_scoring(steps, warmup, device, n_traj=SWEEP_N):
    """pace_score_pool + pace_select on one sweep pool; tag-reduction roofline.  L2 is
    flushed before every timed call (the small pools fit in it)."""
    import torch
    from paper_2609_36830_gb300 import pace, workloads
    pool = workloads.make_pool("sweep", n_traj=n_traj, device=device)
    n = pool.n_traj
    tok = int(pool.meta["offsets_host"][-1])
    c = torch.from_numpy(pool.c_version).to(device)
    sp = torch.from_numpy(pool.s_pre).to(device)
    win = torch.from_numpy(pool.window).to(device)
    params = pace.score_params(group_size=8)
    out = {k: torch.empty(n, dtype=torch.float64, device=device)
           for k in ("kgen", "kwait", "weight", "score")}
    out["unit_score"] = torch.empty(n // 8, dtype=torch.float64, device=device)
    L = pace.lib()
    ws = pace.workspace(L.pace_score_pool_workspace_size(n, win.numel()), device)
    sel = {"accepted": torch.empty(n, dtype=torch.int32, device=device),
           "rejected": torch.empty(n, dtype=torch.int32, device=device),
           "flags": torch.empty(n, dtype=torch.uint8, device=device)}
    ws_sel = pace.workspace(L.pace_select_workspace_size(n // 8), device)
    status = pace.new_status(device)
    bp = pace.budget_params(pool.n_target)
    flush = _L2Flush(device)

    def one():
        pace.score_pool(pool.tags, pool.offsets, c, sp, pool.trainer_version, win, params,
                        out=out, ws=ws, status=status)
        pace.select(out["unit_score"], 8, bp, out=sel, ws=ws_sel, status=status)

    for _ in range(warmup):
        one()
    torch.cuda.synchronize()
    k_b = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    k_e = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    s_b = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    s_e = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    for i in range(steps):
        flush()
        pace.set_profile_events(pace.PROFILE_TAG_REDUCE, k_b[i], k_e[i])
        s_b[i].record()
        one()
        s_e[i].record()
    pace.set_profile_events(pace.PROFILE_TAG_REDUCE)
    torch.cuda.synchronize()
    assert int(status.item()) == 0, pace.status_string(int(status.item()))
    k_ms = statistics.mean(b.elapsed_time(e) for b, e in zip(k_b, k_e))
    s_ms = statistics.mean(b.elapsed_time(e) for b, e in zip(s_b, s_e))
    # the same two calls replayed as one CUDA graph (no host launch gaps)
    g_ms = _timed(_capture(one, device).replay, steps, warmup, flush)
    assert int(status.item()) == 0, pace.status_string(int(status.item()))
    # algorithmic bytes of the tag reduction: every tag once, the offsets once,
    # the 16-byte per-trajectory slots written once
    k_bytes = 4 * tok + 8 * (n + 1) + 16 * n
    fused = n >= L.pace_score_fused_min_traj_default()
    res = {"workload": f"sweep pool {n} trajectories, {tok} tags", "traj_per_s": n / (s_ms / 1e3),
           # from 2^18 trajectories the tag reduction's launch also finalises the scores
           "tag_reduce_launch_finalises": bool(fused),
           "tag_reduce_traffic": (TAG_REDUCE_DRAM_BYTES_PER_TAG * tok
                                  if TAG_REDUCE_DRAM_BYTES_PER_TAG else None),
           "ms_per_call": s_ms, "ms_per_call_graph": g_ms, "tag_reduce_ms": k_ms,
           "tag_reduce_gbs": k_bytes / (k_ms / 1e3) / 1e9, "tag_reduce_bytes": k_bytes}
    if n_traj == SWEEP_N:
        res["admission_variants"] = _admission_variants(pool, tok, out, sel, status, flush,
                                                        steps, warmup, device)
    del pool, flush
    torch.cuda.empty_cache()
    return res


def _capture(fn, device):
    """fn's stream-ordered calls recorded as one CUDA graph (after one eager call on a
    side stream, so one-time launch set-up stays outside the capture)."""
    import torch
    side = torch.cuda.Stream(device=device)
    side.wait_stream(torch.cuda.current_stream(device))
    with torch.cuda.stream(side):
        fn()
    torch.cuda.current_stream(device).wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g


def _timed(fn, steps, warmup, flush=None):
    """Mean CUDA-event time (ms) of fn() over `steps` calls after `warmup`, L2 flushed
    before each timed call when a flush is given."""
    import torch
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(steps)]
    for b, e in evs:
        if flush is not None:
            flush()
        b.record()
        fn()
        e.record()
    torch.cuda.synchronize()
    return statistics.mean(b.elapsed_time(e) for b, e in evs)


def _admission_variants(pool, tok, out, sel, status, flush, steps, warmup, device):
    """The two alternative admission rules and the diagnostics on the 1M sweep pool:
    Stale-k (tag stream + one pass over trajectories, HBM), the retained-vs-rejected
    staleness histogram (one pass over 1M values), and the literal sliding-window
    quantile rule (one block: sort a 512-score window, decide candidates in draw
    order; latency-bound by design) for one step's 64 prompt groups and for 16,384."""
    import torch
    from paper_2609_36830_gb300 import pace
    n = pool.n_traj
    L = pace.lib()
    kbar = torch.empty(n, dtype=torch.float64, device=device)
    adm = torch.empty(n, dtype=torch.uint8, device=device)
    ws = pace.workspace(L.pace_stale_k_workspace_size(n), device)
    k_ms = _timed(lambda: pace.stale_k(pool.tags, pool.offsets, pool.trainer_version, 8.0,
                                       kbar=kbar, admitted=adm, ws=ws, status=status),
                  steps, warmup, flush)
    k_bytes = 4 * tok + 8 * (n + 1) + 16 * n + 9 * n
    hist = torch.empty(2 * 64, dtype=torch.int32, device=device)
    h_ms = _timed(lambda: pace.staleness_histogram(out["kgen"], sel["flags"], 0.0, 32.0, 64,
                                                   hist=hist, status=status),
                  steps, warmup, flush)
    h_bytes = 9 * n
    res = {"stale_k": {"workload": f"{n} trajectories, {tok} tags, k = 8",
                       "ms_per_call": k_ms, "traj_per_s": n / (k_ms / 1e3),
                       "gbs": k_bytes / (k_ms / 1e3) / 1e9},
           "staleness_histogram": {"workload": f"K_gen of {n} trajectories, 64 bins, "
                                               "retained / rejected",
                                   "ms_per_call": h_ms, "values_per_s": n / (h_ms / 1e3),
                                   "gbs": h_bytes / (h_ms / 1e3) / 1e9}}
    qa = {}
    for n_cand in (64, 16384):
        cand = out["unit_score"][:n_cand].contiguous()
        win = pace.ScoreWindow(512, device)
        dec = torch.empty(n_cand, dtype=torch.uint8, device=device)
        kap = torch.empty(1, dtype=torch.float64, device=device)
        pace.quantile_admit(out["unit_score"][-512:].contiguous(), 0.0, 512, win, min_obs=32,
                            decision=torch.empty(512, dtype=torch.uint8, device=device),
                            kappa=kap, status=status)  # fill the window
        q_ms = _timed(lambda: pace.quantile_admit(cand, 0.25, n_cand * 3 // 4, win, min_obs=32,
                                                  decision=dec, kappa=kap, status=status),
                      steps, warmup)
        qa[str(n_cand)] = {"ms_per_call": q_ms, "units_per_s": n_cand / (q_ms / 1e3)}
    res["quantile_admit"] = {"workload": "window of 512 unit scores, r = 0.25, draw until 3/4 "
                                         "of the candidates are retained", "candidates": qa}
    torch.cuda.synchronize()
    assert int(status.item()) == 0, pace.status_string(int(status.item()))
    return res


def _prefix_scoring(steps, warmup, device):
    """pace_prefix_score (Eq. 6) on every interrupted prefix of the math pool: the
    rollout-side overhead the paper measures for PACE (prefix rescoring)."""
    import torch
    from paper_2609_36830_gb300 import pace, workloads
    spec = workloads.SPECS[PREFIX_WORKLOAD]
    pool = workloads.make_pool(PREFIX_WORKLOAD)
    rows = workloads.make_rows(pool)
    pre = workloads.make_prefixes(pool, rows)
    H, V = spec.hidden, spec.vocab
    hidden = workloads.bf16_normal_device((pre.n_rows, H), 1.0, pool.seed + 31, device=device)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), pool.seed + 32, device=device)
    targets = torch.from_numpy(rows.targets[pre.rows]).to(device)
    behav = torch.from_numpy((workloads.uniform_center(V) + np.random.default_rng(3)
                              .standard_normal(pre.n_rows) * 0.3).astype(np.float32)).to(device)
    b = pace.make_batch(torch.from_numpy(pre.seq_offsets).to(device), pre.n_rows,
                        mask=torch.from_numpy(pre.mask).to(device))
    s_pre = torch.empty(len(pre.traj), dtype=torch.float32, device=device)
    lp = torch.empty(pre.n_rows, dtype=torch.float32, device=device)
    ws = pace.workspace(pace.lib().pace_prefix_score_workspace_size(pre.n_rows, len(pre.traj),
                                                                    H, V), device)
    status = pace.new_status(device)
    for _ in range(warmup):
        pace.prefix_score(b, hidden, w, targets, behav, cap_tokens=1024, s_pre=s_pre, logprob=lp,
                          ws=ws, status=status)
    torch.cuda.synchronize()
    scored = int((lp != 0).sum().item())
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    kv = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    for i in range(steps):
        pace.set_profile_events(pace.PROFILE_LMHEAD, *kv[i])
        ev[i][0].record()
        pace.prefix_score(b, hidden, w, targets, behav, cap_tokens=1024, s_pre=s_pre, logprob=lp,
                          ws=ws, status=status)
        ev[i][1].record()
    pace.set_profile_events(pace.PROFILE_LMHEAD)
    torch.cuda.synchronize()
    assert int(status.item()) == 0, pace.status_string(int(status.item()))
    ms = statistics.mean(a.elapsed_time(z) for a, z in ev)
    k_ms = statistics.mean(a.elapsed_time(z) for a, z in kv)
    res = {"workload": f"{len(pre.traj)} interrupted prefixes of the {PREFIX_WORKLOAD} pool, "
                       f"{pre.n_rows} rows, first 1024 eligible tokens scored",
           "prefixes": len(pre.traj), "rows_scored": scored, "ms_per_call": ms,
           "rows_scored_per_s": scored / (ms / 1e3), "lmhead_ms": k_ms,
           "lmhead_tflops": 2.0 * H * V * scored / (k_ms / 1e3) / 1e12}
    del hidden, w, ws
    torch.cuda.empty_cache()
    return res


def _lmhead_backward(steps, warmup, device):
    """pace_surrogate_backward + pace_token_logprob_backward on the math step's accepted rows:
    3 x 2 H V FLOP per row in the loss (recomputed logits, G W, G^T H)."""
    import torch
    from paper_2609_36830_gb300 import pace
    pool, rows, x, st = _make_step(0, device, workload=PREFIX_WORKLOAD)
    st.run()
    torch.cuda.synchronize()
    M = st.rows_in_loss()
    H, V = x.hidden.shape[1], x.w_vocab.shape[0]
    lse = torch.empty(x.mask.numel(), dtype=torch.float32, device=device)
    ws_f = pace.workspace(pace.token_logprob_workspace_size(x.mask.numel(), st.n_traj, H, V),
                          device)
    pace.token_logprob(st.batch, x.hidden, x.w_vocab, x.targets, 1.0, logprob=st.logprob, lse=lse,
                       ws=ws_f, status=st.status)
    del ws_f
    dlp = pace.surrogate_backward(st.batch, st.logprob, st.loss_args, status=st.status)
    gh = torch.empty(x.mask.numel(), H, dtype=torch.float32, device=device)
    gw = torch.empty(V, H, dtype=torch.float32, device=device)
    ws = pace.workspace(pace.lib().pace_token_logprob_backward_workspace_size(
        x.mask.numel(), st.n_traj, H, V), device)
    for _ in range(warmup):
        pace.token_logprob_backward(st.batch, x.hidden, x.w_vocab, x.targets, lse, dlp,
                                    grad_hidden=gh, grad_w=gw, ws=ws, status=st.status)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    for b, e in ev:
        b.record()
        pace.token_logprob_backward(st.batch, x.hidden, x.w_vocab, x.targets, lse, dlp,
                                    grad_hidden=gh, grad_w=gw, ws=ws, status=st.status)
        e.record()
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0, pace.status_string(int(st.status.item()))
    ms = statistics.mean(b.elapsed_time(e) for b, e in ev)
    flops = 3 * 2.0 * H * V * M
    res = {"workload": f"{PREFIX_WORKLOAD} step's {M} rows in the loss, H {H}, V {V}",
           "ms_per_call": ms, "rows_per_s": M / (ms / 1e3),
           "tflops": flops / (ms / 1e3) / 1e12, "flops_per_call": flops}
    del gh, gw, ws, x, st
    torch.cuda.empty_cache()
    return res


def _other_workloads(steps, warmup, device, peak_s):
    """The whole step on the 7B-shaped math pool (512 trajectories, hidden 3584) and
    the multi-turn tool-use pool (256 trajectories, tool segments masked): the same
    call sequence and launch configuration as the headline step."""
    import torch
    from paper_2609_36830_gb300 import pace
    res = {}
    for name in OTHER_WORKLOADS:
        pool, rows, x, st = _make_step(0, device, workload=name)
        for _ in range(warmup):
            st.run()
        torch.cuda.synchronize()
        M = st.rows_in_loss()
        H, V = x.hidden.shape[1], x.w_vocab.shape[0]
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps)]
        lm = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps)]
        for (b, e), (lb, le) in zip(ev, lm):
            pace.set_profile_events(pace.PROFILE_LMHEAD, lb, le)
            b.record()
            st.run()
            e.record()
        pace.set_profile_events(pace.PROFILE_LMHEAD)
        torch.cuda.synchronize()
        assert int(st.status.item()) == 0, pace.status_string(int(st.status.item()))
        ms = statistics.mean(b.elapsed_time(e) for b, e in ev)
        lm_ms = statistics.mean(b.elapsed_time(e) for b, e in lm)
        tf = 2.0 * H * V * M / (lm_ms / 1e3) / 1e12
        res[name] = {"workload": f"{name}: {pool.n_traj} trajectories, capacity {pool.n_target}, "
                                 f"hidden {H}, vocab {V}",
                     "rows_in_loss_per_step": M, "rows_total": int(rows.n_rows),
                     "ms_per_step": ms, "tokens_per_s": M / (ms / 1e3),
                     "lmhead_tflops": tf, "lmhead_frac_of_sustained": tf / peak_s}
        del pool, rows, x, st
        torch.cuda.empty_cache()
    return res


class OracleSampleStep:
    """The oracle's step on a bounded sample of the workload's batch: full admission of
    the pool (scores, budget, top-k) then the fp64 log-probs of n_rows sampled rows in
    the loss and their clipped-surrogate terms.  The vocabulary matrix comes from the
    same seeded generator as the GPU arm's; hidden rows are drawn on the host."""

    def __init__(self, workload, n_rows, seed_offset=0):
        import oracle
        from paper_2609_36830_gb300 import replicas, workloads
        oracle.build()
        spec = workloads.SPECS[workload]
        self.spec = spec
        self.pool = workloads.make_pool(workload,
                                        seed=replicas.replica_seed(workload, seed_offset))
        self.rows = workloads.make_rows(self.pool)
        H, V = spec.hidden, spec.vocab
        seed_w = replicas.replica_seed(workload, 0) + 12
        try:
            import torch
            has_gpu = torch.cuda.is_available()
        except ImportError:
            has_gpu = False
        if has_gpu:
            w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), seed_w)
            self.wb = w.view(torch.int16).cpu().numpy().view(np.uint16)
            del w
        else:
            self.wb = workloads.bf16_normal_host((V, H), 1.0 / math.sqrt(H), seed_w)
        self.behav = workloads.behaviour_logprob(self.rows, self.pool.trainer_version,
                                                 workloads.uniform_center(V), self.pool.seed)
        self.n_rows = n_rows
        self.M = None

    def run(self, i, n_threads):
        """One sample step; returns (seconds, rows in the loss of the whole batch)."""
        import oracle
        from paper_2609_36830_gb300 import workloads
        pool, rows = self.pool, self.rows
        t0 = time.perf_counter()
        st, *_, us = oracle.score_pool(pool.tags, pool.meta["offsets_host"], pool.c_version,
                                       pool.s_pre, pool.trainer_version, pool.window,
                                       group_size=pool.group_size)
        U = pool.n_traj // pool.group_size
        _, _, _, k = oracle.budget(pool.n_traj, pool.n_target, 0.0, 0.9, 0.0, U)
        _, _, _, flags = oracle.select(us, pool.group_size, k)
        in_loss = np.repeat(flags, np.diff(rows.row_offsets)).astype(bool) & \
            rows.mask.astype(bool)
        self.M = int(in_loss.sum())
        rng = np.random.default_rng(i)
        sample = np.sort(rng.choice(np.nonzero(in_loss)[0], size=self.n_rows, replace=False))
        hb = workloads.bf16_normal_host((self.n_rows, self.spec.hidden), 1.0,
                                        pool.seed + 11 + i)
        _, lp, _ = oracle.token_logprob(hb, self.wb, rows.targets[sample], n_threads=n_threads)
        _, adv = oracle.group_advantages(pool.reward, pool.group_size, seq_accepted=flags)
        so = np.arange(self.n_rows + 1, dtype=np.int64)
        seq = np.searchsorted(rows.row_offsets, sample, side="right") - 1
        oracle.surrogate(lp, self.behav[sample], so, adv[seq],
                         eps_low=float(np.float32(self.spec.eps_low)),
                         eps_high=float(np.float32(self.spec.eps_high)))
        return time.perf_counter() - t0, self.M


def _cpu_baseline(n_rows_sample):
    """The oracle as it stands on this host's cores: one sample step of the headline
    workload on every core, and a smaller one on one core."""
    cores = os.cpu_count() or 1
    ref = OracleSampleStep(WORKLOAD, n_rows_sample)
    t, M = ref.run(0, cores)
    n1 = max(n_rows_sample // 16, 1)
    one = OracleSampleStep(WORKLOAD, n1)
    t1, _ = one.run(1, 1)
    return {"value": n_rows_sample / t, "unit": UNIT, "cores": cores, "kind": "oracle",
            "cpu": _cpu_model(),
            "sample": f"one step of the {WORKLOAD} pool: full admission of its "
                      f"{ref.pool.n_traj} trajectories, then fp64 log-probs and surrogate "
                      f"terms of {n_rows_sample} of the {M} rows in the loss ({t:.1f} s); "
                      f"value = sampled rows per second of that step",
            "single_core": {"value": n1 / t1, "unit": UNIT, "cores": 1,
                            "sample": f"the same with {n1} rows on one thread ({t1:.1f} s)"}}


def _cpu_model():
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return None


def _config(ws):
    """The workload both arms name (the same object in the GPU and reference lines)."""
    from paper_2609_36830_gb300 import workloads
    spec = workloads.SPECS[WORKLOAD]
    return {"workload": "moe: 1024 trajectories (128 prompts x 8) per GPU, lognormal responses "
                        "(median 4096, cap 16384), capacity 768, hidden 2048, vocab 151936, "
                        "j=300, EFF scoring gamma 4, groups of 8, clip 0.2/0.28",
            "global_batch": spec.n_traj * ws,
            "parallelism": ("dp1: one GPU, whole pool" if ws == 1 else
                            f"dp{ws}: pool partitioned by prompt group across {ws} GPUs, "
                            "global top-k by histogram all-reduce, loss by partial-sum "
                            "all-reduce"),
            "l2": "inputs larger than L2 (hidden states 21.7 GB per GPU per step)"}


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return
    cores = os.cpu_count() or 1
    rows_per_step = args.ref_rows
    ref = OracleSampleStep(WORKLOAD, rows_per_step)
    times = []
    M = None
    for i in range(args.warmup + args.steps):
        t, M = ref.run(i, cores)
        if i >= args.warmup:
            times.append(t)
    t = statistics.mean(times)
    value = rows_per_step / t
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": t * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": _config(ws),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "cpu": _cpu_model(),
                             "sample": f"per step: full admission of the {ref.pool.n_traj}-"
                                       f"trajectory pool, then fp64 log-probs and surrogate "
                                       f"terms of {rows_per_step} of its {M} rows in the loss; "
                                       f"value = sampled rows per second of the timed steps"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_gpu(args):
    import torch
    import torch.distributed as dist
    from paper_2609_36830_gb300 import pace, replicas
    ws, rank, local = _dist()
    if ws > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    device = f"cuda:{local}"
    peaks, peak_src = _peaks()

    pool, rows, x, lp_params = _make_inputs(rank, device)
    st = _step_for(x, pool, lp_params, ws, rank, device)
    H, V = x.hidden.shape[1], x.w_vocab.shape[0]
    # the LM head's vocabulary split count, measured on this GPU (untimed; one GPU:
    # the ranks of a sharded step keep the automatic choice so that they agree)
    splits, split_ms = (st.tune_lmhead_splits() if ws == 1 else (0, {}))
    k_units = None
    for _ in range(args.warmup):
        k_units, _ = st.run()
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0, pace.status_string(int(st.status.item()))
    M = st.rows_in_loss()

    K = args.steps
    k_b = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    k_e = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    t_b = torch.cuda.Event(enable_timing=True)
    t_e = torch.cuda.Event(enable_timing=True)
    launches0 = pace.kernel_launches()
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t_b.record()
        for i in range(K):
            pace.set_profile_events(pace.PROFILE_LMHEAD, k_b[i], k_e[i])
            st.run()
        t_e.record()
        torch.cuda.synchronize()
    pace.set_profile_events(pace.PROFILE_LMHEAD)
    launches = pace.kernel_launches() - launches0
    assert int(st.status.item()) == 0, pace.status_string(int(st.status.item()))
    ms = t_b.elapsed_time(t_e) / K
    job_rows, ms = replicas.job_totals(M, ms, device)
    if ws > 1:
        dist.barrier()
    lm_each = [b.elapsed_time(e) for b, e in zip(k_b, k_e)]
    lm_ms = statistics.mean(lm_each)
    flops = 2.0 * H * V * M
    achieved = flops / (lm_ms / 1e3) / 1e12
    peak_s = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
    value = job_rows / (ms / 1e3)
    loss_value = float(st.loss.item())

    # End to end through the same C ABI with host buffers: every step's inputs are
    # copied from pinned host memory and its log-probs and loss copied back.  The
    # copy of step i+1's inputs (on a copy stream) overlaps step i's compute.  The
    # step alternates between two device input sets, each with its own step
    # driver, as a trainer that prefetches its next batch would do: the copy
    # into a set waits only for the step that last read it.
    names = ("tags", "offsets", "c_version", "s_pre", "window", "row_offsets", "mask",
             "targets", "behav_lp", "reward", "hidden", "w_vocab")
    host = {}
    for name in names:
        t = getattr(x, name)
        h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        host[name] = h
    x2 = dataclasses.replace(x, **{name: torch.empty_like(getattr(x, name)) for name in names})
    st2 = _step_for(x2, pool, lp_params, ws, rank, device)
    sets = [(x, st), (x2, st2)]
    h2d = sum(h.numel() * h.element_size() for h in host.values())
    lp_host = torch.empty(x.mask.numel(), dtype=torch.float32, pin_memory=True)
    loss_host = torch.empty(1, dtype=torch.float64, pin_memory=True)
    d2h = lp_host.numel() * 4 + 8
    e_steps = max(2, K)
    copy_stream = torch.cuda.Stream(device=device)
    comp = torch.cuda.current_stream(device)
    staged = [torch.cuda.Event() for _ in range(e_steps)]
    done = [torch.cuda.Event() for _ in range(e_steps)]

    def h2d_copy(i):
        xi = sets[i % 2][0]
        with torch.cuda.stream(copy_stream):
            if i >= 2:
                copy_stream.wait_event(done[i - 2])  # the last step that read this set
            for name in names:
                getattr(xi, name).copy_(host[name], non_blocking=True)
            staged[i].record(copy_stream)

    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e_b = torch.cuda.Event(enable_timing=True)
    e_e = torch.cuda.Event(enable_timing=True)
    e_b.record()
    h2d_copy(0)
    for i in range(e_steps):
        sti = sets[i % 2][1]
        comp.wait_event(staged[i])
        if i + 1 < e_steps:
            h2d_copy(i + 1)
        sti.run()
        done[i].record(comp)
        lp_host.copy_(sti.logprob, non_blocking=True)
        loss_host.copy_(sti.loss, non_blocking=True)
    e_e.record()
    torch.cuda.synchronize()
    assert int(st2.status.item()) == 0, pace.status_string(int(st2.status.item()))
    e_ms = e_b.elapsed_time(e_e) / e_steps
    _, e_ms = replicas.job_totals(M, e_ms, device)
    del host, x2, st2, sets

    sweep = prefix = backward = others = cpu = None
    # the split count was tuned on this head shape only: the heads measured below
    # (hidden 3584) take the automatic choice
    pace.set_lmhead_splits(0)
    if not args.no_sweep and rank == 0 and ws == 1:
        del x, st
        torch.cuda.empty_cache()
        sizes = []
        for n_sw in SWEEP_SIZES:
            r_sw = _sweep_scoring(max(3, min(K, 5)) if n_sw == SWEEP_N else 10, 3, device, n_sw)
            r_sw["tag_reduce_frac_of_hbm"] = r_sw["tag_reduce_gbs"] / peaks["hbm_gbs"]
            r_sw["hbm_peak_gbs"] = peaks["hbm_gbs"]
            if n_sw == SWEEP_N:
                sweep = r_sw
            else:
                sizes.append({k: r_sw[k] for k in ("workload", "traj_per_s", "ms_per_call",
                                                   "ms_per_call_graph",
                                                   "tag_reduce_ms", "tag_reduce_gbs",
                                                   "tag_reduce_frac_of_hbm")})
        sweep["smaller_pools"] = sizes
        prefix = _prefix_scoring(max(3, min(K, 5)), 3, device)
        backward = _lmhead_backward(3, 1, device)
        backward["frac_of_sustained"] = backward["tflops"] / peak_s
        others = _other_workloads(3, 2, device, peak_s)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = _cpu_baseline(args.cpu_rows)

    if rank == 0:
        chosen = splits or 4  # the automatic choice at this size is 4 (pick_splits)
        traffic = LMHEAD_DRAM_BYTES_PER_ROW.get((WORKLOAD, chosen))
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": _config(ws),
            "step_detail": {"rows_in_loss_per_step": job_rows, "rows_in_loss_rank0": M,
                            "rows_total_rank0": int(rows.n_rows), "k_units_rejected": k_units,
                            "loss": loss_value,
                            "lmhead_splits": {"chosen": splits,
                                              "tuning_ms_per_step": {str(k): v for k, v
                                                                     in split_ms.items()}}},
            "roofline": {"bound": "tensor", "kernel": "lmhead_lse_kernel", "achieved": achieved,
                         "peak": peak_s, "unit": "TFLOP/s", "frac": achieved / peak_s,
                         "peak_source": f"{peak_src} bf16_tflops_sustained",
                         "frac_of_burst": achieved / peaks["bf16_tflops"],
                         "kernel_ms": lm_ms, "kernel_ms_each": lm_each,
                         "flops_per_launch": flops,
                         "traffic": traffic * M if traffic else None,
                         "traffic_note": "dram read+write bytes per launch: bytes per row in the "
                                         "loss from a one-pass ncu capture of the current kernel "
                                         "at the split count used (4: one 19,456-row wave; 2: "
                                         "one full-length launch), times the rows of this "
                                         "launch"},
            "cpu_baseline": cpu,
            "e2e": {"value": job_rows / (e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "ms_per_step": e_ms},
            "gpu_launches": launches,
            "clocks": clk.summary(),
            "pool_scoring": sweep,
            "prefix_scoring": prefix,
            "lmhead_backward": backward,
            "other_workloads": others,
        }
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.destroy_process_group()


def run_case(args):
    """One kernel's launch configuration on a small case (for profiler captures)."""
    import torch
    from paper_2609_36830_gb300 import pace, workloads
    device = "cuda:0"
    torch.cuda.set_device(0)
    peaks, _ = _peaks()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    if args.case == "step_tiny":
        # the smallest workload (64 trajectories, H 256, V 2048): a step is a few
        # tens of microseconds of kernels, so launch latency matters; time it
        # eagerly and as one CUDA-graph replay
        from paper_2609_36830_gb300 import step
        pool = workloads.make_pool("tiny")
        rows = workloads.make_rows(pool)
        H, V = pool.spec.hidden, pool.spec.vocab
        hidden = workloads.bf16_normal_device((rows.n_rows, H), 1.0, pool.seed + 11, device)
        w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), pool.seed + 12, device)
        behav = workloads.behaviour_logprob(rows, pool.trainer_version,
                                            workloads.uniform_center(V), pool.seed)
        x = step.build_inputs(pool, rows, hidden, w, behav, device=device)
        st = step.PaceStep(x, loss_params=pace.loss_params(eps_low=0.2, eps_high=0.2),
                           device=device)
        M = None
        res = {}
        for mode in ("eager", "graph"):
            fn = st.run if mode == "eager" else st.capture().replay
            for _ in range(max(args.warmup, 3)):
                fn()
            torch.cuda.synchronize()
            b, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            n_rep = max(args.steps, 100)
            b.record()
            for _ in range(n_rep):
                fn()
            e.record()
            torch.cuda.synchronize()
            res[mode] = b.elapsed_time(e) / n_rep * 1e3
            M = st.rows_in_loss()
        assert int(st.status.item()) == 0
        print(json.dumps({"case": "step_tiny", "rows_in_loss": M, "us_per_step": res,
                          "tokens_per_s": {k: M / (v / 1e6) for k, v in res.items()}}),
              flush=True)
        return
    if args.case == "lmhead":
        spec = workloads.SPECS[args.case_workload]
        H, V, rows = spec.hidden, spec.vocab, args.case_rows
        hidden = workloads.bf16_normal_device((rows, H), 1.0, 101, device)
        w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), 102, device)
        gen = torch.Generator(device=device)
        gen.manual_seed(103)
        targets = torch.randint(0, V, (rows,), generator=gen, device=device, dtype=torch.int32)
        # --case-mask: every row in the loss, but read through the compacted row
        # index (the path masked and rejected rows take) instead of TMA boxes
        mask = torch.ones(rows, dtype=torch.uint8, device=device) if args.case_mask else None
        if args.case_mask_period:
            # prompt-like gaps: rows r with r % period < gap are outside the loss
            r = torch.arange(rows, device=device)
            mask = (r % args.case_mask_period >= args.case_mask_gap).to(torch.uint8)
        b = pace.make_batch(torch.tensor([0, rows], dtype=torch.int64, device=device), rows,
                            mask=mask)
        lp = torch.empty(rows, dtype=torch.float32, device=device)
        ws = pace.workspace(pace.token_logprob_workspace_size(rows, 1, H, V), device)
        status = pace.new_status(device)
        pace.set_lmhead_splits(args.case_splits)
        for i in range(args.warmup + args.steps):
            if i >= args.warmup:
                pace.set_profile_events(pace.PROFILE_LMHEAD, *evs[i - args.warmup])
            pace.token_logprob(b, hidden, w, targets, 1.0, logprob=lp, ws=ws, status=status)
        pace.set_profile_events(pace.PROFILE_LMHEAD)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        ms = statistics.mean(a.elapsed_time(z) for a, z in evs)
        n_loss = int(mask.sum().item()) if mask is not None else rows
        tf = 2.0 * n_loss * H * V / (ms / 1e3) / 1e12
        print(json.dumps({"case": "lmhead", "workload": args.case_workload, "rows": rows,
                          "rows_in_loss": n_loss, "H": H,
                          "V": V, "rows_by_index": mask is not None,
                          "mask_period": args.case_mask_period, "kernel_ms": ms,
                          "tflops": tf, "frac_burst": tf / peaks["bf16_tflops"]}), flush=True)
    elif args.case == "lmhead_bwd":
        spec = workloads.SPECS[WORKLOAD]
        H, V, rows = spec.hidden, spec.vocab, args.case_rows
        hidden = workloads.bf16_normal_device((rows, H), 1.0, 101, device)
        w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), 102, device)
        gen = torch.Generator(device=device)
        gen.manual_seed(103)
        targets = torch.randint(0, V, (rows,), generator=gen, device=device, dtype=torch.int32)
        dlp = torch.randn(rows, generator=gen, device=device) * 1e-6
        b = pace.make_batch(torch.tensor([0, rows], dtype=torch.int64, device=device), rows)
        lp = torch.empty(rows, dtype=torch.float32, device=device)
        lse = torch.empty(rows, dtype=torch.float32, device=device)
        status = pace.new_status(device)
        pace.token_logprob(b, hidden, w, targets, 1.0, logprob=lp, lse=lse, status=status)
        gh = torch.empty(rows, H, dtype=torch.float32, device=device)
        gw = torch.empty(V, H, dtype=torch.float32, device=device)
        ws = pace.workspace(pace.lib().pace_token_logprob_backward_workspace_size(rows, 1, H, V),
                            device)
        for i in range(args.warmup + args.steps):
            if i == args.warmup:
                torch.cuda.synchronize()
                t0 = torch.cuda.Event(enable_timing=True)
                t1 = torch.cuda.Event(enable_timing=True)
                t0.record()
            pace.token_logprob_backward(b, hidden, w, targets, lse, dlp, grad_hidden=gh,
                                        grad_w=gw, ws=ws, status=status)
        t1.record()
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        ms = t0.elapsed_time(t1) / args.steps
        tf = 3 * 2.0 * rows * H * V / (ms / 1e3) / 1e12
        print(json.dumps({"case": "lmhead_bwd", "rows": rows, "H": H, "V": V, "ms": ms,
                          "tflops": tf}), flush=True)
    elif args.case == "select":
        # pace_select_k alone: --case-units unit scores drawn uniformly in [0, 30),
        # groups of 8, half the units rejected
        U = args.case_units
        gen = torch.Generator(device=device)
        gen.manual_seed(104)
        scores = torch.rand(U, generator=gen, device=device, dtype=torch.float64) * 30.0
        out = {"accepted": torch.empty(U * 8, dtype=torch.int32, device=device),
               "rejected": torch.empty(U * 8, dtype=torch.int32, device=device),
               "flags": torch.empty(U * 8, dtype=torch.uint8, device=device)}
        ws = pace.workspace(pace.lib().pace_select_workspace_size(U), device)
        status = pace.new_status(device)
        ms = _timed(lambda: pace.select_k(scores, 8, U // 2, out=out, ws=ws, status=status),
                    args.steps, args.warmup)
        assert int(status.item()) == 0
        print(json.dumps({"case": "select", "units": U, "group_size": 8, "ms_per_call": ms}),
              flush=True)
    elif args.case == "pool":
        # pace_score_pool + pace_select on one sweep pool, L2 evicted before each call,
        # eagerly and as one CUDA-graph replay
        res = _sweep_scoring(args.steps, args.warmup, device, n_traj=args.case_traj)
        print(json.dumps({"case": "pool", **res,
                          "tag_reduce_frac_of_hbm": res["tag_reduce_gbs"] / peaks["hbm_gbs"]}),
              flush=True)
    else:
        pool = workloads.make_pool("sweep", n_traj=args.case_traj, device=device)
        n = pool.n_traj
        tok = int(pool.meta["offsets_host"][-1])
        c = torch.from_numpy(pool.c_version).to(device)
        sp = torch.from_numpy(pool.s_pre).to(device)
        win = torch.from_numpy(pool.window).to(device)
        status = pace.new_status(device)
        flush = _L2Flush(device)
        for i in range(args.warmup + args.steps):
            flush()
            if i >= args.warmup:
                pace.set_profile_events(pace.PROFILE_TAG_REDUCE, *evs[i - args.warmup])
            out = pace.score_pool(pool.tags, pool.offsets, c, sp, pool.trainer_version, win,
                                  pace.score_params(group_size=8), status=status)
        pace.set_profile_events(pace.PROFILE_TAG_REDUCE)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        ms = statistics.mean(a.elapsed_time(z) for a, z in evs)
        nbytes = 4 * tok + 8 * (n + 1) + 16 * n
        print(json.dumps({"case": "tagreduce", "n_traj": n, "tokens": tok, "kernel_ms": ms,
                          "gbs": nbytes / (ms / 1e3) / 1e9,
                          "frac_hbm": nbytes / (ms / 1e3) / 1e9 / peaks["hbm_gbs"]}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--cpu-rows", type=int, default=512)
    ap.add_argument("--ref-rows", type=int, default=96,
                    help="rows of the batch the reference arm's oracle computes per step")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--case", choices=["lmhead", "lmhead_bwd", "tagreduce", "step_tiny", "pool",
                                       "select"],
                    default=None,
                    help="time one kernel on a small case (profiler captures)")
    ap.add_argument("--case-rows", type=int, default=4864)
    ap.add_argument("--case-mask", action="store_true",
                    help="lmhead case: pass a mask of ones, so rows are read by index")
    ap.add_argument("--case-mask-period", type=int, default=0,
                    help="lmhead case: mask out the first --case-mask-gap rows of every period")
    ap.add_argument("--case-mask-gap", type=int, default=256)
    ap.add_argument("--case-workload", default=WORKLOAD, choices=["math7b", "multiturn", "moe"])
    ap.add_argument("--case-traj", type=int, default=16384)
    ap.add_argument("--case-units", type=int, default=131072)
    ap.add_argument("--case-splits", type=int, default=0,
                    help="LM-head vocabulary splits for --case lmhead (0 = automatic)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
        return
    from paper_2609_36830_gb300 import build as pace_build
    pace_build.build()
    if args.case:
        run_case(args)
        return
    run_gpu(args)


if __name__ == "__main__":
    main()
