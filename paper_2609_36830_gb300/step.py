"""One PACE trainer step through the C ABI, on one GPU.

Algorithm 1, trainer side, followed by the unchanged policy objective:
  1. pace_score_pool     staleness scores of every pooled trajectory and the
                         group means (Lemma 1 / Eq. 2, Eqs. 7-10);
  2. pace_select         occupancy budget (Eqs. 3-4) and rejection of the
                         top-scored groups; per-trajectory accepted flags;
  3. pace_token_logprob  for the rows of accepted trajectories that are in the
                         loss: the fused LM-head log-probs, GRPO advantages
                         over accepted group members, the clipped surrogate.
All buffers are allocated once here (the library allocates nothing) and every
call is queued on one stream; the only host work inside a step is the budget
arithmetic, which needs no device value.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import numpy as np
import torch

from . import pace


@dataclass
class StepInputs:
    """Device-resident inputs of a step (see pace.h for each array's meaning)."""
    tags: torch.Tensor         # int32 [n_tokens]
    offsets: torch.Tensor      # int64 [n_traj+1]
    c_version: torch.Tensor    # int32 [n_traj]
    s_pre: torch.Tensor        # float32 [n_traj]
    window: torch.Tensor       # float32 [W]
    row_offsets: torch.Tensor  # int64 [n_traj+1]
    mask: torch.Tensor         # uint8 [n_rows]
    targets: torch.Tensor      # int32 [n_rows]
    behav_lp: torch.Tensor     # float32 [n_rows]
    reward: torch.Tensor       # float32 [n_traj]
    hidden: torch.Tensor       # bf16 [n_rows, H]
    w_vocab: torch.Tensor      # bf16 [V, H]
    trainer_version: int
    n_target: int
    group_size: int


class PaceStep:
    """Buffers and calls of one trainer step; call ``run`` once per step.

    The pool in ``x`` may be refreshed in place between steps (new tags, versions,
    rows); ``n_target``, ``beta`` and ``r_max`` follow the paper's Eqs. 3-4 and the
    admission settings."""

    def __init__(self, x: StepInputs, score_params=None, loss_params=None, beta=0.0,
                 r_max=0.9, temperature=1.0, device="cuda"):
        self.x = x
        self.dev = device
        self.n_traj = x.offsets.numel() - 1
        self.G = x.group_size
        self.U = self.n_traj // self.G
        self.n_rows = x.mask.numel()
        self.H = x.hidden.shape[1]
        self.V = x.w_vocab.shape[0]
        self.temperature = float(temperature)
        self.sp = score_params or pace.score_params(group_size=self.G)
        self.lp_params = loss_params or pace.loss_params()
        self.beta, self.r_max = float(beta), float(r_max)
        self.r_hat = 0.0
        d = device
        f64 = dict(dtype=torch.float64, device=d)
        self.score_out = {k: torch.empty(self.n_traj, **f64)
                          for k in ("kgen", "kwait", "weight", "score")}
        self.score_out["unit_score"] = torch.empty(self.U, **f64)
        L = pace.lib()
        self.ws_score = pace.workspace(
            L.pace_score_pool_workspace_size(self.n_traj, x.window.numel()), d)
        self.sel_out = {"accepted": torch.empty(self.n_traj, dtype=torch.int32, device=d),
                        "rejected": torch.empty(self.n_traj, dtype=torch.int32, device=d),
                        "flags": torch.empty(self.n_traj, dtype=torch.uint8, device=d)}
        self.ws_select = pace.workspace(L.pace_select_workspace_size(self.U), d)
        self.logprob = torch.empty(self.n_rows, dtype=torch.float32, device=d)
        self.loss = torch.zeros(1, **f64)
        self.adv = torch.empty(self.n_traj, dtype=torch.float32, device=d)
        self.ws_lm = pace.workspace(
            pace.token_logprob_workspace_size(self.n_rows, self.n_traj, self.H, self.V), d)
        self.status = pace.new_status(d)
        self.batch = pace.make_batch(x.row_offsets, self.n_rows,
                                     seq_accepted=self.sel_out["flags"], mask=x.mask)
        self.loss_args = pace.make_loss_args(x.behav_lp, x.reward, self.G, self.lp_params,
                                             self.loss, adv_out=self.adv)
        self.k_units = None

    def run(self, stream=None):
        """Queue one step; returns (k_units, r_hat).  Nothing is synchronised.

        r_hat (Eq. 4) is carried into the next call's budget as r-hat_{j-1}."""
        x = self.x
        pace.score_pool(x.tags, x.offsets, x.c_version, x.s_pre, x.trainer_version, x.window,
                        self.sp, out=self.score_out, ws=self.ws_score, status=self.status,
                        stream=stream)
        bp = pace.budget_params(x.n_target, beta=self.beta, r_max=self.r_max,
                                r_hat_prev=self.r_hat)
        r_hat, k, _, _, _ = pace.select(self.score_out["unit_score"], self.G, bp,
                                        out=self.sel_out, ws=self.ws_select,
                                        status=self.status, stream=stream)
        pace.token_logprob(self.batch, x.hidden, x.w_vocab, x.targets, self.temperature,
                           loss=self.loss_args, logprob=self.logprob, ws=self.ws_lm,
                           status=self.status, stream=stream)
        self.k_units = k
        self.r_hat = r_hat
        return k, r_hat

    def tune_lmhead_splits(self, candidates=(2, 4), reps=2):
        """Time whole steps with each candidate vocabulary-split count of the LM head
        (pace_set_lmhead_splits) on this GPU, alternating candidates ``reps`` times,
        and keep the fastest for the process.  The count changes no result beyond
        rounding order, only the GPU's power-capped clock during the long LM-head
        launch, which differs from GPU to GPU.  Returns (best, {count: mean ms})."""
        times = {c: [] for c in candidates}
        for _ in range(reps):
            for c in candidates:
                pace.set_lmhead_splits(c)
                b = torch.cuda.Event(enable_timing=True)
                e = torch.cuda.Event(enable_timing=True)
                self.run()  # settle after the change
                b.record()
                self.run()
                e.record()
                torch.cuda.synchronize()
                times[c].append(b.elapsed_time(e))
        mean = {c: sum(v) / len(v) for c, v in times.items()}
        best = min(candidates, key=lambda c: (mean[c], c))
        pace.set_lmhead_splits(best)
        return best, mean

    def capture(self):
        """One step recorded as a CUDA graph (torch.cuda.CUDAGraph) for replay on a
        pool of fixed shape whose inputs are refreshed in place: every call of the
        step is stream-ordered with no host synchronisation, so a replay re-runs the
        whole step with one launch.  The budget k is host arithmetic and is frozen
        at capture, so capture needs beta = 0 (with beta > 0 the occupancy EMA of
        Eq. 4 would move k from step to step)."""
        if self.beta != 0.0:
            raise ValueError("capture needs beta = 0: the budget is frozen into the graph")
        side = torch.cuda.Stream(device=self.dev)
        side.wait_stream(torch.cuda.current_stream(self.dev))
        with torch.cuda.stream(side):
            self.run()  # one-time launch set-up outside the capture
        torch.cuda.current_stream(self.dev).wait_stream(side)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run()
        return g

    def rows_in_loss(self) -> int:
        """Rows the step's LM head processed (host count, synchronising)."""
        flags = self.sel_out["flags"].to(torch.int64)
        per_traj = torch.repeat_interleave(flags, torch.diff(self.x.row_offsets),
                                           output_size=self.n_rows)
        return int((per_traj * self.x.mask.to(torch.int64)).sum().item())


def build_inputs(pool, rows, hidden, w_vocab, behav_lp, device="cuda") -> StepInputs:
    """Uploads a workloads.Pool / Rows pair (host arrays) plus device tensors."""
    def dv(a, dtype=None):
        if isinstance(a, torch.Tensor):
            return a.to(device)
        t = torch.from_numpy(np.ascontiguousarray(a))
        return (t.to(dtype) if dtype is not None else t).to(device)
    return StepInputs(
        tags=dv(pool.tags), offsets=dv(pool.meta["offsets_host"]), c_version=dv(pool.c_version),
        s_pre=dv(pool.s_pre), window=dv(pool.window), row_offsets=dv(rows.row_offsets),
        mask=dv(rows.mask), targets=dv(rows.targets), behav_lp=dv(behav_lp),
        reward=dv(pool.reward), hidden=hidden, w_vocab=w_vocab,
        trainer_version=pool.trainer_version, n_target=pool.n_target,
        group_size=pool.group_size)
