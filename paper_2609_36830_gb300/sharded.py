"""Data-parallel PACE step over a pool partitioned across ranks by prompt group.

Rank r holds the contiguous units (prompt groups) [u0_r, u0_r + U_r) of the
whole pool, with their trajectories, rows and hidden states.  The admission
rule stays the rule of the whole pool (Sec. 3.1, Eqs. 3-4, Algorithm 1):
  1. pace_score_pool on the rank's trajectories: the scores need nothing from
     other ranks (the prefix-score window is replicated);
  2. the budget k from the whole pool's counts (host arithmetic, the same on
     every rank);
  3. the k top-scored units of the whole pool: six radix passes, each followed
     by a sum of one 2048-bin histogram over the ranks (all-reduce), then the
     ties at the pivot taken lowest id first from the tie counts of lower ranks
     (one exclusive sum of an int64 per rank);
  4. the fused log-prob + clipped surrogate on the rank's accepted rows: whole
     groups live on one rank, so the GRPO advantages are local, and the loss is
     the quotient of the (numerator, denominator) partials summed over the ranks
     (one all-reduce of two fp64 values).
The rejected and accepted sets equal those of the unsharded pool, and the loss
equals the unsharded loss up to the order of the final fp64 sums.

A rank's calls are written as a generator that yields at every exchange:
``(ALL_REDUCE, t)`` asks for t summed over the ranks in place, and
``(EXCLUSIVE_SUM, (src, dst))`` for dst = the sum of src over the lower ranks.
``run_process_group`` serves the requests with torch.distributed (NCCL for CUDA
tensors, gloo for CPU tensors); ``run_lockstep`` serves several shards held by
one process, advancing them together, so a sharded step can be checked on one
GPU without any kernel waiting on another.
"""
from __future__ import annotations

import dataclasses
from typing import Iterable, List, Sequence

import torch

from . import pace

ALL_REDUCE = "all_reduce_sum"
EXCLUSIVE_SUM = "exclusive_sum"


def run_process_group(gen, group=None):
    """Drives one rank's generator, serving its exchanges with torch.distributed."""
    import torch.distributed as dist
    world = dist.get_world_size(group)
    rank = dist.get_rank(group)
    for kind, t in gen:
        if kind == ALL_REDUCE:
            dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
        elif kind == EXCLUSIVE_SUM:
            src, dst = t
            parts = [torch.empty_like(src) for _ in range(world)]
            dist.all_gather(parts, src, group=group)
            dst.zero_()
            for p in parts[:rank]:
                dst.add_(p)
        else:
            raise ValueError(f"unknown exchange {kind!r}")


def run_lockstep(gens: List[Iterable]):
    """Drives the generators of all shards held by this process together: each
    exchange is served once every shard has reached it (all shards in one
    process, on one stream: nothing waits on anything but the host)."""
    gens = [iter(g) for g in gens]
    while True:
        reqs = [next(g, None) for g in gens]
        if all(r is None for r in reqs):
            return
        if any(r is None for r in reqs):
            raise RuntimeError("shards left the protocol at different points")
        kinds = {r[0] for r in reqs}
        if len(kinds) != 1:
            raise RuntimeError(f"shards asked for different exchanges: {sorted(kinds)}")
        kind = kinds.pop()
        if kind == ALL_REDUCE:
            total = torch.stack([r[1] for r in reqs]).sum(dim=0)
            for r in reqs:
                r[1].copy_(total)
        elif kind == EXCLUSIVE_SUM:
            run = torch.zeros_like(reqs[0][1][0])
            for r in reqs:
                src, dst = r[1]
                dst.copy_(run)
                run = run + src
        else:
            raise ValueError(f"unknown exchange {kind!r}")


class LibraryShardOps:
    """The per-rank calls of the sharded rejection, on the GPU (libpace)."""

    @staticmethod
    def pass_(unit_score, p, k, prev, cur, ws, status, stream):
        pace.select_shard_pass(unit_score, p, k, prev, cur, ws, status=status, stream=stream)

    @staticmethod
    def ties(unit_score, last, tied, ws, status, stream):
        pace.select_shard_ties(unit_score, last, tied, ws, status=status, stream=stream)

    @staticmethod
    def write(unit_score, group_size, k, tied_before, id_base, out, ws, n_rejected, status,
              stream):
        pace.select_shard_write(unit_score, group_size, k, tied_before, id_base, out, ws,
                                n_rejected_out=n_rejected, status=status, stream=stream)


class ShardSelectBuffers:
    """Device buffers of one rank's sharded rejection (allocated once)."""

    def __init__(self, n_units: int, group_size: int, device):
        n = max(n_units * group_size, 1)
        self.out = {"accepted": torch.empty(n, dtype=torch.int32, device=device),
                    "rejected": torch.empty(n, dtype=torch.int32, device=device),
                    "flags": torch.empty(n, dtype=torch.uint8, device=device)}
        self.hist = [torch.zeros(pace.SHARD_HIST_BINS, dtype=torch.int32, device=device)
                     for _ in range(2)]
        self.tied = torch.zeros(1, dtype=torch.int64, device=device)
        self.tied_before = torch.zeros(1, dtype=torch.int64, device=device)
        self.n_rejected = torch.zeros(1, dtype=torch.int64, device=device)
        self.ws = (pace.select_shard_workspace(n_units, device)
                   if torch.device(device).type == "cuda" else None)


def select_protocol(unit_score, group_size: int, k: int, id_base: int, buf: ShardSelectBuffers,
                    status=None, stream=None, ops=LibraryShardOps):
    """Generator: one rank's part of the whole pool's top-k rejection (the calls
    of pace_select_shard_*, yielding at the histogram sums and the tie scan).
    Afterwards buf.out holds this shard's accepted / rejected ids (global ids)
    and per-trajectory accepted flags, buf.n_rejected its rejected units."""
    prev = None
    for p in range(pace.SHARD_PASSES):
        cur = buf.hist[p % 2]
        ops.pass_(unit_score, p, k, prev, cur, buf.ws, status, stream)
        yield ALL_REDUCE, cur
        prev = cur
    ops.ties(unit_score, prev, buf.tied, buf.ws, status, stream)
    yield EXCLUSIVE_SUM, (buf.tied, buf.tied_before)
    ops.write(unit_score, group_size, k, buf.tied_before, id_base, buf.out, buf.ws,
              buf.n_rejected, status, stream)


class ShardedPaceStep:
    """One rank's part of a data-parallel PACE step (see the module docstring).

    ``x`` holds this rank's trajectories, rows and hidden states (step.StepInputs;
    its ``n_target`` is ignored); the window and the vocabulary matrix are the
    same on every rank.  ``unit_base`` is the global id of the rank's first unit,
    ``n_traj_total`` and ``n_target_total`` the whole pool's trajectory count and
    capacity (Eq. 3).  Drive ``steps()`` with ``run_process_group`` (one process
    per GPU) or with ``run_lockstep`` (several shards in one process)."""

    def __init__(self, x, unit_base: int, n_traj_total: int, n_target_total: int,
                 score_params=None, loss_params=None, beta=0.0, r_max=0.9, temperature=1.0,
                 device="cuda"):
        self.x = x
        self.dev = device
        self.n_traj = x.offsets.numel() - 1
        self.G = x.group_size
        self.U = self.n_traj // self.G
        self.unit_base = int(unit_base)
        self.n_traj_total = int(n_traj_total)
        self.n_target_total = int(n_target_total)
        if self.n_traj_total % self.G:
            raise ValueError("the whole pool must hold whole groups")
        self.n_rows = x.mask.numel()
        self.H = x.hidden.shape[1]
        self.V = x.w_vocab.shape[0]
        self.temperature = float(temperature)
        self.sp = score_params or pace.score_params(group_size=self.G)
        self.lp_params = loss_params or pace.loss_params()
        self.beta, self.r_max = float(beta), float(r_max)
        self.r_hat = 0.0
        f64 = dict(dtype=torch.float64, device=device)
        self.score_out = {k: torch.empty(self.n_traj, **f64)
                          for k in ("kgen", "kwait", "weight", "score")}
        self.score_out["unit_score"] = torch.empty(max(self.U, 1), **f64)[: self.U]
        L = pace.lib()
        self.ws_score = pace.workspace(
            L.pace_score_pool_workspace_size(self.n_traj, x.window.numel()), device)
        self.sel = ShardSelectBuffers(self.U, self.G, device)
        self.logprob = torch.empty(self.n_rows, dtype=torch.float32, device=device)
        self.loss = torch.zeros(1, **f64)
        self.partial = torch.zeros(2, **f64)
        self.adv = torch.empty(max(self.n_traj, 1), dtype=torch.float32,
                               device=device)[: self.n_traj]
        self.ws_lm = pace.workspace(
            pace.token_logprob_workspace_size(self.n_rows, self.n_traj, self.H, self.V), device)
        self.status = pace.new_status(device)
        self.batch = pace.make_batch(x.row_offsets, self.n_rows,
                                     seq_accepted=self.sel.out["flags"], mask=x.mask)
        self.loss_args = pace.make_loss_args(x.behav_lp, x.reward, self.G, self.lp_params,
                                             self.loss, adv_out=self.adv,
                                             partial_out=self.partial)
        self.k_units = None

    def steps(self, stream=None):
        """Generator of one step; afterwards ``loss`` holds the whole batch's loss on
        every rank and ``sel.out["flags"]`` this shard's accepted trajectories."""
        x = self.x
        pace.score_pool(x.tags, x.offsets, x.c_version, x.s_pre, x.trainer_version, x.window,
                        self.sp, out=self.score_out, ws=self.ws_score, status=self.status,
                        stream=stream)
        bp = pace.budget_params(self.n_target_total, beta=self.beta, r_max=self.r_max,
                                r_hat_prev=self.r_hat)
        _, r_hat, k = pace.budget(self.n_traj_total, self.n_traj_total // self.G, bp)
        yield from select_protocol(self.score_out["unit_score"], self.G, k,
                                   self.unit_base * self.G, self.sel, status=self.status,
                                   stream=stream)
        pace.token_logprob(self.batch, x.hidden, x.w_vocab, x.targets, self.temperature,
                           loss=self.loss_args, logprob=self.logprob, ws=self.ws_lm,
                           status=self.status, stream=stream)
        yield ALL_REDUCE, self.partial
        pace.loss_from_partial(self.partial, self.loss, stream=stream)
        self.k_units = k
        self.r_hat = r_hat

    def run(self, group=None):
        """One step with the exchanges over torch.distributed; returns (k, r_hat)."""
        run_process_group(self.steps(), group)
        return self.k_units, self.r_hat

    def rows_in_loss(self) -> int:
        """Rows this rank's LM head processed (host count, synchronising)."""
        flags = self.sel.out["flags"][: self.n_traj].to(torch.int64)
        per_traj = torch.repeat_interleave(flags, torch.diff(self.x.row_offsets),
                                           output_size=self.n_rows)
        return int((per_traj * self.x.mask.to(torch.int64)).sum().item())


def split_inputs(x, bounds: Sequence[int]):
    """The StepInputs of each shard of one pool: shard i holds the units
    [bounds[i], bounds[i + 1]) with their trajectories, tags and rows (fresh,
    aligned copies); the window and the vocabulary matrix are shared."""
    G = x.group_size
    offs = x.offsets.cpu()
    roffs = x.row_offsets.cpu()
    shards = []
    for u0, u1 in zip(bounds[:-1], bounds[1:]):
        t0, t1 = u0 * G, u1 * G
        k0, k1 = int(offs[t0]), int(offs[t1])
        r0, r1 = int(roffs[t0]), int(roffs[t1])
        shards.append(dataclasses.replace(
            x, tags=x.tags[k0:k1].clone(), offsets=(x.offsets[t0:t1 + 1] - k0).clone(),
            c_version=x.c_version[t0:t1].clone(), s_pre=x.s_pre[t0:t1].clone(),
            row_offsets=(x.row_offsets[t0:t1 + 1] - r0).clone(), mask=x.mask[r0:r1].clone(),
            targets=x.targets[r0:r1].clone(), behav_lp=x.behav_lp[r0:r1].clone(),
            reward=x.reward[t0:t1].clone(), hidden=x.hidden[r0:r1].clone()))
    return shards
