"""Pins of the oracle's log-probability, advantage and surrogate functions.

* log-probs against the fp64 log_softmax of a library (torch, CPU) on random
  non-square shapes, the W = 0 closed form (-log V), one-hot hidden rows
  (logits become one column of W) and temperature scaling;
* GRPO advantages against numpy's mean / std (ddof = 1) and two-member closed
  forms;
* the clipped surrogate against hand-worked branch cases and the on-policy
  identity (behaviour = current gives ratio 1 and loss = -sum m A / sum m).
"""
import math

import numpy as np
import pytest
import torch

import oracle


def _bf16_bits(x):
    """float32 array -> (bf16 bit patterns as uint16, the float32 values they hold)."""
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    bits = t.view(torch.int16).numpy().view(np.uint16).copy()
    return bits, t.to(torch.float32).numpy()


@pytest.mark.parametrize("rows,H,V,tau", [(5, 24, 37, 1.0), (9, 64, 130, 1.0), (4, 16, 11, 0.7)])
def test_logprob_matches_library_log_softmax(rows, H, V, tau):
    rng = np.random.default_rng(rows * 1000 + V)
    hb, hf = _bf16_bits(rng.standard_normal((rows, H)))
    wb, wf = _bf16_bits(rng.standard_normal((V, H)) / math.sqrt(H) * 3.0)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    st, lp, lse = oracle.token_logprob(hb, wb, y, temperature=tau, n_threads=3)
    assert st == oracle.OK
    z = torch.from_numpy(hf.astype(np.float64)) @ torch.from_numpy(wf.astype(np.float64)).T
    ref = torch.log_softmax(z / tau, dim=-1)
    expect = ref[torch.arange(rows), torch.from_numpy(y).long()].numpy()
    np.testing.assert_allclose(lp, expect, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, torch.logsumexp(z / tau, dim=-1).numpy(), rtol=0, atol=1e-12)


def test_logprob_zero_weights_is_uniform():
    rng = np.random.default_rng(0)
    V, H = 2048, 64
    hb, _ = _bf16_bits(rng.standard_normal((7, H)))
    wb = np.zeros((V, H), np.uint16)
    y = rng.integers(0, V, size=7).astype(np.int32)
    st, lp, lse = oracle.token_logprob(hb, wb, y)
    assert st == oracle.OK
    np.testing.assert_allclose(lp, -math.log(V), rtol=0, atol=1e-13)


def test_logprob_one_hot_rows_pick_a_column():
    rng = np.random.default_rng(1)
    V, H = 50, 32
    wb, wf = _bf16_bits(rng.standard_normal((V, H)))
    eye = np.eye(H, dtype=np.float32)[[3, 0, 31]]
    hb, _ = _bf16_bits(eye)
    y = np.array([7, 0, 49], np.int32)
    st, lp, _ = oracle.token_logprob(hb, wb, y)
    assert st == oracle.OK
    for i, k in enumerate([3, 0, 31]):
        col = wf[:, k].astype(np.float64)
        expect = col[y[i]] - (col.max() + math.log(np.exp(col - col.max()).sum()))
        assert abs(lp[i] - expect) < 1e-12


def test_logprob_row_subset_and_bad_target():
    rng = np.random.default_rng(2)
    hb, _ = _bf16_bits(rng.standard_normal((10, 16)))
    wb, _ = _bf16_bits(rng.standard_normal((20, 16)))
    y = rng.integers(0, 20, size=10).astype(np.int32)
    _, full, _ = oracle.token_logprob(hb, wb, y)
    st, sub, _ = oracle.token_logprob(hb, wb, y, rows=[9, 2, 2])
    assert st == oracle.OK
    np.testing.assert_array_equal(sub, full[[9, 2, 2]])
    y[4] = 20
    assert oracle.token_logprob(hb, wb, y)[0] == oracle.ERR_INVALID_ARG


def test_group_advantages_against_numpy():
    rng = np.random.default_rng(4)
    G = 8
    r = (rng.random(64) < 0.4).astype(np.float32)
    r[:8] = 1.0  # an all-equal group
    st, adv = oracle.group_advantages(r, G, eps=1e-6, unbiased=True)
    assert st == oracle.OK
    for g in range(0, 64, G):
        x = r[g:g + G].astype(np.float64)
        expect = (x - x.mean()) / (x.std(ddof=1) + 1e-6)
        np.testing.assert_allclose(adv[g:g + G], expect, rtol=1e-15, atol=1e-15)
    assert (adv[:8] == 0).all()
    st, adv_pop = oracle.group_advantages(r, G, eps=1e-6, unbiased=False)
    x = r[8:16].astype(np.float64)
    np.testing.assert_allclose(adv_pop[8:16], (x - x.mean()) / (x.std() + 1e-6), rtol=1e-15)


def test_group_advantages_accepted_members_only():
    r = np.array([1, 0, 1, 1, 0, 0, 1, 0], np.float32)
    acc = np.array([1, 1, 0, 0, 1, 0, 0, 0], np.uint8)
    st, adv = oracle.group_advantages(r, 4, seq_accepted=acc, eps=0.0, unbiased=True)
    assert st == oracle.OK
    # group 0: members {1, 0}: mean 1/2, sample std sqrt(1/2)
    assert abs(adv[0] - 0.5 / math.sqrt(0.5)) < 1e-15
    assert abs(adv[1] + 0.5 / math.sqrt(0.5)) < 1e-15
    assert adv[2] == adv[3] == 0.0  # rejected
    assert adv[4] == 0.0  # single accepted member
    assert (adv[5:] == 0).all()


@pytest.mark.parametrize("a,rho,expect", [
    (1.0, 1.5, -1.28),   # upper clip at 1 + eps_high
    (-1.0, 0.5, 0.8),    # lower clip at 1 - eps_low
    (-1.0, 20.0, 10.0),  # dual clip caps the loss at -c A
    (1.0, 0.5, -0.5),    # ratio below 1 - eps for a positive advantage: unclipped term wins
    (2.0, 1.1, -2.2),    # inside the trust region
    (-0.5, 1.5, 0.75),   # negative advantage, ratio above 1 + eps: unclipped p1 = 0.75
])
def test_surrogate_branches(a, rho, expect):
    lp = np.array([math.log(rho)])
    behav = np.array([0.0])
    st, loss, ratio, term = oracle.surrogate(lp, behav, [0, 1], [a], eps_low=0.2, eps_high=0.28,
                                             dual_clip=10.0)
    assert st == oracle.OK
    assert abs(ratio[0] - rho) < 1e-12
    assert abs(loss - expect) < 1e-12 and abs(term[0] - expect) < 1e-12


def test_surrogate_on_policy_identity():
    rng = np.random.default_rng(5)
    n_seq = 12
    lens = rng.integers(1, 30, size=n_seq)
    so = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    lp = -rng.random(so[-1]) * 10
    mask = (rng.random(so[-1]) < 0.7).astype(np.uint8)
    acc = (rng.random(n_seq) < 0.8).astype(np.uint8)
    adv = rng.standard_normal(n_seq)
    st, loss, ratio, term = oracle.surrogate(lp, lp, so, adv, mask=mask, seq_accepted=acc)
    assert st == oracle.OK
    rows_in = np.repeat(acc, lens).astype(bool) & mask.astype(bool)
    assert (ratio[rows_in] == 1.0).all()
    a_row = np.repeat(adv, lens)
    expect = -(a_row[rows_in]).sum() / rows_in.sum()
    assert abs(loss - expect) < 1e-12
    st, loss_s, _, _ = oracle.surrogate(lp, lp, so, adv, mask=mask, seq_accepted=acc,
                                        agg=oracle.AGG_SEQ_MEAN_TOKEN_MEAN)
    per_seq = [-adv[i] for i in range(n_seq)
               if acc[i] and mask[so[i]:so[i + 1]].any()]
    assert abs(loss_s - np.mean(per_seq)) < 1e-12


def test_surrogate_empty_and_ratio_clamp():
    st, loss, _, _ = oracle.surrogate([0.0, 0.0], [0.0, 0.0], [0, 2], [1.0],
                                      mask=np.zeros(2, np.uint8))
    assert st == oracle.OK and loss == 0.0
    st, loss, ratio, _ = oracle.surrogate([100.0], [0.0], [0, 1], [-1.0])
    assert ratio[0] == math.exp(20.0) and loss == 10.0
