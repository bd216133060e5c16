"""The data-parallel step's kernels on one GPU: a pool split into 2-4 shards,
each shard's calls driven in lockstep in one process (sharded.run_lockstep
sums the histograms and the partials between the calls; no kernel waits on
another).  The union of the shards' selections must equal the oracle's top-k
on the unsharded pool id for id, and the loss assembled from the shards'
partials must match the single-GPU step's loss (same log-probs, same rows)
and the oracle's surrogate over every row of the unsharded batch."""
import math

import numpy as np
import pytest
import torch

import oracle
from pace_cases import DEV, as_np, to_dev
from paper_2609_36830_gb300 import pace, sharded, step, workloads

pytestmark = pytest.mark.gpu


def _select_sharded(us, G, k, bounds):
    bufs, gens = [], []
    for u0, u1 in zip(bounds[:-1], bounds[1:]):
        buf = sharded.ShardSelectBuffers(u1 - u0, G, DEV)
        score = to_dev(np.ascontiguousarray(us[u0:u1]))
        gens.append(sharded.select_protocol(score, G, k, u0 * G, buf))
        bufs.append((buf, score))
    sharded.run_lockstep(gens)
    torch.cuda.synchronize()
    acc, rej, flags = [], [], []
    for (buf, score), u0, u1 in zip(bufs, bounds[:-1], bounds[1:]):
        n = (u1 - u0) * G
        nr = int(buf.n_rejected.item()) * G
        acc.append(as_np(buf.out["accepted"][: n - nr]))
        rej.append(as_np(buf.out["rejected"][:nr]))
        flags.append(as_np(buf.out["flags"][:n]))
    return np.concatenate(acc), np.concatenate(rej), np.concatenate(flags)


@pytest.mark.parametrize("U,G,bounds_frac", [(1000, 8, (0, 0.5, 1)),
                                             (4097, 1, (0, 0.25, 0.25, 0.6, 1)),
                                             (131072, 8, (0, 0.3, 0.7, 1)),
                                             (300, 2, (0, 0.1, 0.2, 0.9, 1))])
@pytest.mark.parametrize("law", ["ties", "spread"])
def test_sharded_selection_matches_unsharded_oracle(U, G, bounds_frac, law):
    rng = np.random.default_rng(U + G + len(law))
    if law == "ties":
        us = rng.integers(0, 12, size=U).astype(np.float64) / 8.0
    else:
        us = rng.exponential(2.0, size=U)
    us[: min(3, U)] = [-0.0, 0.0, 0.0][: min(3, U)]
    bounds = [int(round(f * U)) for f in bounds_frac]
    for k in sorted({0, 1, U // 3, U // 2 + 1, U - 1, U}):
        oacc, orej, oflag = oracle.select(us, G, k)[1:]
        acc, rej, flags = _select_sharded(us, G, k, bounds)
        np.testing.assert_array_equal(acc, oacc)
        np.testing.assert_array_equal(rej, orej)
        np.testing.assert_array_equal(flags, oflag)


def _inputs(name, n_traj):
    pool = workloads.make_pool(name, n_traj=n_traj)
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, pool.seed + 11)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), pool.seed + 12)
    behav = workloads.behaviour_logprob(rw, pool.trainer_version, workloads.uniform_center(V),
                                        pool.seed)
    return pool, rw, behav, step.build_inputs(pool, rw, hidden, w, behav)


@pytest.mark.parametrize("name,n_traj,n_shards", [("tiny", None, 2), ("tiny", None, 4),
                                                  ("math7b", 512, 4)])
def test_sharded_step_matches_single_gpu_step_and_oracle(name, n_traj, n_shards):
    pool, rw, behav, x = _inputs(name, n_traj)
    lp_params = pace.loss_params(eps_low=pool.spec.eps_low, eps_high=pool.spec.eps_high)
    single = step.PaceStep(x, loss_params=lp_params)
    single.run()
    U = pool.n_traj // pool.group_size
    bounds = [round(i * U / n_shards) for i in range(n_shards + 1)]
    shards = [sharded.ShardedPaceStep(xs, u0, pool.n_traj, pool.n_target, loss_params=lp_params)
              for xs, u0 in zip(sharded.split_inputs(x, bounds), bounds[:-1])]
    sharded.run_lockstep([s.steps() for s in shards])
    torch.cuda.synchronize()
    assert int(single.status.item()) == 0
    assert all(int(s.status.item()) == 0 for s in shards)
    assert len({s.k_units for s in shards}) == 1 and shards[0].k_units == single.k_units
    flags = np.concatenate([as_np(s.sel.out["flags"][: s.n_traj]) for s in shards])
    np.testing.assert_array_equal(flags, as_np(single.sel_out["flags"]))
    *_, ous = oracle.score_pool(pool.tags, pool.meta["offsets_host"], pool.c_version,
                                pool.s_pre, pool.trainer_version, pool.window,
                                group_size=pool.group_size)
    oflag = oracle.select(ous, pool.group_size, single.k_units)[3]
    np.testing.assert_array_equal(flags, oflag)
    # the log-probs of each shard's rows are those of the single step (a shard's
    # LM-head launch may split the vocabulary differently: rounding only)
    lp = np.concatenate([as_np(s.logprob) for s in shards])
    np.testing.assert_allclose(lp, as_np(single.logprob), rtol=0, atol=1e-4)
    # every shard holds the whole batch's loss
    losses = [float(s.loss.item()) for s in shards]
    assert len(set(losses)) == 1
    ref = float(single.loss.item())
    assert abs(losses[0] - ref) <= 1e-4 * max(abs(ref), 1e-300)
    # and the oracle's surrogate over all rows of the unsharded batch (GPU log-probs)
    _, oadv = oracle.group_advantages(pool.reward, pool.group_size, seq_accepted=oflag,
                                      eps=float(np.float32(1e-6)))
    st, oloss, _, oterm = oracle.surrogate(lp, behav, rw.row_offsets, oadv, mask=rw.mask,
                                           seq_accepted=oflag,
                                           eps_low=float(np.float32(pool.spec.eps_low)),
                                           eps_high=float(np.float32(pool.spec.eps_high)))
    assert st == 0
    in_loss = np.repeat(oflag, np.diff(rw.row_offsets)).astype(bool) & rw.mask.astype(bool)
    scale = max(abs(oloss), float(np.abs(oterm[in_loss]).mean()))
    assert abs(losses[0] - oloss) <= 1e-3 * scale


def test_sharded_selection_reports_nan_scores():
    """A NaN unit score on any shard is reported through that shard's status word
    (first pass), as the single-GPU selection does."""
    us = np.linspace(0.0, 5.0, 600)
    us[450] = np.nan
    bounds = [0, 300, 600]
    statuses, gens, bufs = [], [], []
    for u0, u1 in zip(bounds[:-1], bounds[1:]):
        buf = sharded.ShardSelectBuffers(u1 - u0, 2, DEV)
        st = pace.new_status(DEV)
        gens.append(sharded.select_protocol(to_dev(np.ascontiguousarray(us[u0:u1])), 2, 100,
                                            u0 * 2, buf, status=st))
        statuses.append(st)
        bufs.append(buf)
    sharded.run_lockstep(gens)
    torch.cuda.synchronize()
    assert int(statuses[0].item()) == 0
    assert int(statuses[1].item()) == pace.ERR_NAN_INPUT
