"""GRPO advantages and the clipped surrogate on the GPU vs the oracle.

Advantages are fp64 on both sides and rounded to float32 once: bit-identical.
The surrogate's per-token terms are fp32 on the GPU and fp64 in the oracle;
the loss must agree within 1e-3 relative (observed ~1e-7) and the ratios
within 1e-5 relative.  Inputs here are seeded synthetic log-probs, so the
oracle computes the full loss even at the largest batch sizes."""
import numpy as np
import pytest
import torch

import oracle
from pace_cases import DEV, as_np, to_dev
from paper_2609_36830_gb300 import pace, workloads

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("G,n_seq,p_acc", [(8, 64, 1.0), (8, 512, 0.75), (12, 1200, 0.5),
                                           (1, 300, 0.8), (16, 16, 0.3)])
@pytest.mark.parametrize("unbiased", [True, False])
def test_advantages_bitwise(G, n_seq, p_acc, unbiased):
    rng = np.random.default_rng(G * 1000 + n_seq)
    r = (rng.random(n_seq) < 0.4).astype(np.float32)
    r[: G] = 1.0  # an all-equal group
    acc = (rng.random(n_seq) < p_acc).astype(np.uint8)
    eps = np.float32(1e-6)
    adv = pace.group_advantages(to_dev(r), G, seq_accepted=to_dev(acc), adv_eps=eps,
                                std_unbiased=unbiased)
    st, oadv = oracle.group_advantages(r, G, seq_accepted=acc, eps=float(eps), unbiased=unbiased)
    assert st == 0
    np.testing.assert_array_equal(as_np(adv), oadv.astype(np.float32))


def _batch(rows, seed, accept_p=0.75):
    pool = workloads.make_pool(*rows)
    rw = workloads.make_rows(pool)
    rng = np.random.default_rng(seed)
    lp = (workloads.uniform_center(pool.spec.vocab or 1000)
          + rng.standard_normal(rw.n_rows)).astype(np.float32)
    behav = workloads.behaviour_logprob(rw, pool.trainer_version,
                                        workloads.uniform_center(pool.spec.vocab or 1000), seed)
    acc = (rng.random(pool.n_traj) < accept_p).astype(np.uint8)
    return pool, rw, lp, behav, acc


@pytest.mark.parametrize("rows", [("tiny", None), ("math7b", 512), ("multiturn", 480),
                                  ("moe", None)])
@pytest.mark.parametrize("agg", [pace.AGG_TOKEN_MEAN, pace.AGG_SEQ_MEAN_TOKEN_MEAN])
def test_surrogate_matches_oracle(rows, agg):
    pool, rw, lp, behav, acc = _batch(rows, 3)
    params = pace.loss_params(eps_low=pool.spec.eps_low, eps_high=pool.spec.eps_high,
                              agg=agg)
    loss = torch.zeros(1, dtype=torch.float64, device=DEV)
    ratio = torch.empty(rw.n_rows, dtype=torch.float32, device=DEV)
    adv = torch.empty(pool.n_traj, dtype=torch.float32, device=DEV)
    la = pace.make_loss_args(to_dev(behav), to_dev(pool.reward), pool.group_size, params, loss,
                             adv_out=adv, ratio_out=ratio)
    b = pace.make_batch(to_dev(rw.row_offsets), rw.n_rows, seq_accepted=to_dev(acc),
                        mask=to_dev(rw.mask))
    status = pace.new_status(DEV)
    pace.surrogate_loss(b, to_dev(lp), la, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    st, oadv = oracle.group_advantages(pool.reward, pool.group_size, seq_accepted=acc,
                                       eps=float(np.float32(1e-6)))
    np.testing.assert_array_equal(as_np(adv), oadv.astype(np.float32))
    st, oloss, oratio, _ = oracle.surrogate(lp, behav, rw.row_offsets, oadv,
                                            mask=rw.mask, seq_accepted=acc,
                                            eps_low=float(np.float32(pool.spec.eps_low)),
                                            eps_high=float(np.float32(pool.spec.eps_high)),
                                            dual_clip=10.0, agg=agg)
    assert st == 0
    gl = float(loss.item())
    assert abs(gl - oloss) <= 1e-3 * max(abs(oloss), 1e-12), (gl, oloss)
    np.testing.assert_allclose(as_np(ratio), oratio, rtol=1e-5, atol=0)


def test_on_policy_identity_on_gpu():
    pool, rw, lp, _, acc = _batch(("tiny", None), 9, accept_p=1.0)
    loss = torch.zeros(1, dtype=torch.float64, device=DEV)
    ratio = torch.empty(rw.n_rows, dtype=torch.float32, device=DEV)
    adv = torch.empty(pool.n_traj, dtype=torch.float32, device=DEV)
    la = pace.make_loss_args(to_dev(lp), to_dev(pool.reward), pool.group_size,
                             pace.loss_params(), loss, adv_out=adv, ratio_out=ratio)
    b = pace.make_batch(to_dev(rw.row_offsets), rw.n_rows, mask=to_dev(rw.mask))
    pace.surrogate_loss(b, to_dev(lp), la)
    torch.cuda.synchronize()
    r = as_np(ratio)[rw.mask.astype(bool)]
    assert (r == 1.0).all()
    st, oadv = oracle.group_advantages(pool.reward, pool.group_size, eps=float(np.float32(1e-6)))
    a_row = np.repeat(oadv, np.diff(rw.row_offsets))[rw.mask.astype(bool)]
    expect = -a_row.sum() / a_row.size
    assert abs(float(loss.item()) - expect) <= 1e-9 + 1e-6 * abs(expect)


def test_empty_loss_is_zero_and_bad_offsets_reported():
    so = np.array([0, 3, 5], np.int64)
    loss = torch.full((1,), 7.0, dtype=torch.float64, device=DEV)
    la = pace.make_loss_args(to_dev(np.zeros(5, np.float32)), to_dev(np.ones(2, np.float32)), 2,
                             pace.loss_params(), loss)
    b = pace.make_batch(to_dev(so), 5, mask=to_dev(np.zeros(5, np.uint8)))
    pace.surrogate_loss(b, to_dev(np.zeros(5, np.float32)), la)
    torch.cuda.synchronize()
    assert float(loss.item()) == 0.0
    bad = np.array([0, 4, 3], np.int64)
    b = pace.make_batch(to_dev(bad), 5)
    status = pace.new_status(DEV)
    pace.surrogate_loss(b, to_dev(np.zeros(5, np.float32)), la, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == pace.ERR_INVALID_ARG
