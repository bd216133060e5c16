"""One whole PACE step (score -> budget/select -> fused log-prob + loss) at
the full-size workloads (7B single-turn at occupancies 1.0 / 1.33 / 2.0 of
capacity, multi-turn with tool segments at 1.0 / 2.5, the MoE head), in
exactly the launch configuration bench.py times: the selection must match the
oracle id for id, sampled log-probs within 5e-3, the fused loss must equal
the standalone surrogate on the same log-probs, and it must match the oracle's
surrogate computed over every row from the GPU log-probs (verified on the
sample) and the same behaviour log-probs, within 1e-3 relative (to the larger
of |loss| and the mean |term| of the rows in the loss).  Then the occupancy EMA
(Eq. 4) carried across steps."""
import math

import numpy as np
import pytest
import torch

import oracle
from pace_cases import DEV, as_np
from paper_2609_36830_gb300 import pace, step, workloads

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,n_traj", [("math7b", 384), ("math7b", 512), ("math7b", 768),
                                         ("multiturn", 256), ("multiturn", 480), ("moe", 1024)])
def test_full_size_step(name, n_traj):
    pool = workloads.make_pool(name, n_traj=n_traj)
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, pool.seed + 11)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), pool.seed + 12)
    behav = workloads.behaviour_logprob(rw, pool.trainer_version, workloads.uniform_center(V),
                                        pool.seed)
    x = step.build_inputs(pool, rw, hidden, w, behav)
    lp_params = pace.loss_params(eps_low=pool.spec.eps_low, eps_high=pool.spec.eps_high)
    st = step.PaceStep(x, loss_params=lp_params)
    k, r_hat = st.run()
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    # selection parity
    ost, *_, ous = oracle.score_pool(pool.tags, pool.meta["offsets_host"], pool.c_version,
                                     pool.s_pre, pool.trainer_version, pool.window,
                                     group_size=pool.group_size)
    U = pool.n_traj // pool.group_size
    _, _, orh, ok = oracle.budget(pool.n_traj, pool.n_target, 0.0, 0.9, 0.0, U)
    assert (k, r_hat) == (ok, orh)
    _, oacc, orej, oflag = oracle.select(ous, pool.group_size, ok)
    np.testing.assert_array_equal(as_np(st.sel_out["flags"]), oflag)
    # sampled log-probs
    lp = as_np(st.logprob)
    in_loss = np.repeat(oflag, np.diff(rw.row_offsets)).astype(bool) & rw.mask.astype(bool)
    assert (lp[~in_loss] == 0).all() and np.isfinite(lp).all()
    rng = np.random.default_rng(17)
    sample = np.sort(rng.choice(np.nonzero(in_loss)[0], size=32, replace=False))
    hb = hidden[torch.from_numpy(sample).to(DEV)].view(torch.int16).cpu().numpy().view(np.uint16)
    wb = w.view(torch.int16).cpu().numpy().view(np.uint16)
    _, olp, _ = oracle.token_logprob(hb, wb, rw.targets[sample])
    assert np.abs(lp[sample] - olp).max() <= 5e-3
    # fused loss == standalone surrogate on the same log-probs (same stream)
    loss2 = torch.zeros(1, dtype=torch.float64, device=DEV)
    la = pace.make_loss_args(x.behav_lp, x.reward, pool.group_size, lp_params, loss2)
    pace.surrogate_loss(st.batch, st.logprob, la)
    torch.cuda.synchronize()
    assert float(st.loss.item()) == float(loss2.item())
    assert math.isfinite(float(st.loss.item()))
    assert st.rows_in_loss() == int(in_loss.sum())
    # fused loss against the oracle's surrogate over all rows (GRPO
    # advantages over the accepted members of each group)
    _, oadv = oracle.group_advantages(pool.reward, pool.group_size, seq_accepted=oflag,
                                      eps=float(np.float32(1e-6)))
    sst, oloss, _, oterm = oracle.surrogate(lp, behav, rw.row_offsets, oadv, mask=rw.mask,
                                            seq_accepted=oflag,
                                            eps_low=float(np.float32(pool.spec.eps_low)),
                                            eps_high=float(np.float32(pool.spec.eps_high)),
                                            dual_clip=10.0)
    assert sst == 0
    scale = max(abs(oloss), float(np.abs(oterm[in_loss]).mean()))
    assert abs(float(st.loss.item()) - oloss) <= 1e-3 * scale, (float(st.loss.item()), oloss)


def test_ema_budget_carried_across_steps():
    """Eq. 4 across steps: r-hat_j = beta r-hat_{j-1} + (1 - beta) r_j.  The step
    driver carries r-hat from one call to the next while the pool occupancy changes;
    the oracle runs the same recurrence and the rejected groups must match."""
    beta, n_target = 0.5, 24
    o_rhat, r_hat_prev = 0.0, 0.0
    for i, n_traj in enumerate([96, 64, 48, 80, 96, 24]):
        pool = workloads.make_pool("tiny", seed=900 + i, n_traj=n_traj)
        rw = workloads.make_rows(pool)
        H, V = pool.spec.hidden, pool.spec.vocab
        hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, 40 + i)
        w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), 41)
        behav = workloads.behaviour_logprob(rw, pool.trainer_version,
                                            workloads.uniform_center(V), i)
        x = step.build_inputs(pool, rw, hidden, w, behav)
        x.n_target = n_target
        st = step.PaceStep(x, beta=beta)
        st.r_hat = r_hat_prev  # a new pool shape needs new buffers; the state carries over
        k, r_hat = st.run()
        torch.cuda.synchronize()
        assert int(st.status.item()) == 0
        U = n_traj // pool.group_size
        _, _, o_rhat, ok = oracle.budget(n_traj, n_target, beta, 0.9, o_rhat, U)
        assert (k, r_hat) == (ok, o_rhat), i
        assert st.r_hat == r_hat
        _, _, _, _, _, ous = oracle.score_pool(pool.tags, pool.meta["offsets_host"],
                                               pool.c_version, pool.s_pre,
                                               pool.trainer_version, pool.window,
                                               group_size=pool.group_size)
        _, _, _, oflag = oracle.select(ous, pool.group_size, ok)
        np.testing.assert_array_equal(as_np(st.sel_out["flags"]), oflag)
        r_hat_prev = r_hat
    assert o_rhat > 0.0  # the carried state reached the last, under-target step


def test_repeated_run_advances_ema():
    """Calling run() twice on one pool applies Eq. 4 twice."""
    pool = workloads.make_pool("tiny", seed=77, n_traj=96)
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, 78)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), 79)
    behav = workloads.behaviour_logprob(rw, pool.trainer_version, workloads.uniform_center(V), 1)
    x = step.build_inputs(pool, rw, hidden, w, behav)
    st = step.PaceStep(x, beta=0.75)
    U = 96 // pool.group_size
    o = 0.0
    for _ in range(3):
        k, r_hat = st.run()
        _, _, o, ok = oracle.budget(96, x.n_target, 0.75, 0.9, o, U)
        assert (k, r_hat) == (ok, o)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0


def test_split_tuner_keeps_a_candidate_and_results():
    """PaceStep.tune_lmhead_splits times the candidates on this GPU, keeps the
    fastest for the process, and the step's results do not depend on it."""
    pool = workloads.make_pool("tiny")
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, 3)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), 4)
    behav = workloads.behaviour_logprob(rw, pool.trainer_version, workloads.uniform_center(V), 5)
    st = step.PaceStep(step.build_inputs(pool, rw, hidden, w, behav))
    st.run()
    torch.cuda.synchronize()
    lp0 = st.logprob.clone()
    try:
        best, mean = st.tune_lmhead_splits(candidates=(2, 4), reps=1)
        assert best in (2, 4) and set(mean) == {2, 4}
        assert all(v > 0 for v in mean.values())
        st.run()
        torch.cuda.synchronize()
        assert int(st.status.item()) == 0
        assert float((st.logprob - lp0).abs().max()) <= 2e-5
    finally:
        pace.set_lmhead_splits(0)
