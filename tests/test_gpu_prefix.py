"""Prefix Forgetting Score (Eq. 6) on the GPU vs the oracle: prefixes of the
pool's interrupted rollouts re-scored under an updated policy.  s_pre within
5e-3 (the log-prob tolerance bounds a mean of absolute differences), the same
NaN pattern (fewer than 32 eligible tokens), and the 1,024 / 2,048 caps."""
import math

import numpy as np
import pytest
import torch

import oracle
from pace_cases import DEV, as_np, bf16_dev, to_dev
from paper_2609_36830_gb300 import pace, workloads

pytestmark = pytest.mark.gpu
TOL = 5e-3


def _case(name, n_traj, H, V, seed):
    pool = workloads.make_pool(name, n_traj=n_traj)
    rows = workloads.make_rows(pool)
    pre = workloads.make_prefixes(pool, rows)
    hb = workloads.bf16_normal_host((pre.n_rows, H), 1.0, seed)
    wb = workloads.bf16_normal_host((V, H), 1.0 / math.sqrt(H), seed + 1)
    targets = (rows.targets[pre.rows] % V).astype(np.int32)
    behav = (workloads.uniform_center(V)
             + np.random.default_rng(seed).standard_normal(pre.n_rows) * 0.3).astype(np.float32)
    return pool, pre, hb, wb, targets, behav


@pytest.mark.parametrize("name,n_traj,cap", [("tiny", None, 1024), ("math7b", 64, 1024),
                                             ("multiturn", 32, 2048), ("math7b", 64, 100)])
def test_prefix_score_matches_oracle(name, n_traj, cap):
    H, V = 256, 2048
    pool, pre, hb, wb, targets, behav = _case(name, n_traj, H, V, 5)
    b = pace.make_batch(to_dev(pre.seq_offsets), pre.n_rows, mask=to_dev(pre.mask))
    status = pace.new_status(DEV)
    lp = torch.empty(pre.n_rows, dtype=torch.float32, device=DEV)
    s = pace.prefix_score(b, bf16_dev(hb), bf16_dev(wb), to_dev(targets), to_dev(behav),
                          min_tokens=32, cap_tokens=cap, logprob=lp, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    st, olp, _ = oracle.token_logprob(hb, wb, targets)
    assert st == 0
    st, os_ = oracle.prefix_score(olp, behav, pre.seq_offsets, mask=pre.mask, min_tokens=32,
                                  cap_tokens=cap)
    assert st == 0
    g = as_np(s).astype(np.float64)
    assert (np.isnan(g) == np.isnan(os_)).all()
    ok = ~np.isnan(os_)
    assert ok.sum() > 0
    assert np.abs(g[ok] - os_[ok]).max() <= TOL
    # rows beyond each prefix's cap were not scored (lp left at 0)
    glp = as_np(lp)
    for i in range(len(pre.traj)):
        r0, r1 = pre.seq_offsets[i], pre.seq_offsets[i + 1]
        elig = np.nonzero(pre.mask[r0:r1])[0]
        beyond = elig[cap:] + r0
        assert (glp[beyond] == 0).all()


def test_full_size_prefix_rescoring_sampled():
    """7B-shaped head (H 3584, V 152064), every interrupted prefix of the math pool:
    the eligibility pattern exactly, log-probs on sampled scored rows."""
    pool = workloads.make_pool("math7b")
    rows = workloads.make_rows(pool)
    pre = workloads.make_prefixes(pool, rows)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((pre.n_rows, H), 1.0, 31)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), 32)
    targets = rows.targets[pre.rows]
    behav = (workloads.uniform_center(V)
             + np.random.default_rng(3).standard_normal(pre.n_rows) * 0.3).astype(np.float32)
    b = pace.make_batch(to_dev(pre.seq_offsets), pre.n_rows, mask=to_dev(pre.mask))
    lp = torch.empty(pre.n_rows, dtype=torch.float32, device=DEV)
    status = pace.new_status(DEV)
    s = pace.prefix_score(b, hidden, w, to_dev(targets), to_dev(behav), cap_tokens=1024,
                          logprob=lp, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    # eligibility decided by the oracle from the masks alone (log-probs do not matter)
    zeros = np.zeros(pre.n_rows)
    _, pattern = oracle.prefix_score(zeros, zeros, pre.seq_offsets, mask=pre.mask,
                                     min_tokens=32, cap_tokens=1024)
    g = as_np(s)
    assert (np.isnan(g) == np.isnan(pattern)).all()
    assert np.isfinite(g[~np.isnan(pattern)]).all() and (g[~np.isnan(pattern)] > 0).all()
    glp = as_np(lp)
    scored = np.nonzero(glp != 0)[0]
    rng = np.random.default_rng(7)
    sample = np.sort(rng.choice(scored, size=24, replace=False))
    hb = hidden[torch.from_numpy(sample).to(DEV)].view(torch.int16).cpu().numpy().view(np.uint16)
    wb = w.view(torch.int16).cpu().numpy().view(np.uint16)
    _, olp, _ = oracle.token_logprob(hb, wb, targets[sample])
    assert np.abs(glp[sample] - olp).max() <= TOL
