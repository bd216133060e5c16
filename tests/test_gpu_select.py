"""Budget + top-k rejection on the GPU vs the oracle: the k, r-hat and every
accepted / rejected trajectory id must be identical (ties: lower id first)."""
import numpy as np
import pytest
import torch

import oracle
from pace_cases import DEV, as_np, oracle_score, pool_score_case, to_dev
from paper_2609_36830_gb300 import pace, workloads

pytestmark = pytest.mark.gpu


def _gpu_select_k(scores, G, k, expect_status=0):
    status = pace.new_status(DEV)
    acc, rej, flags = pace.select_k(to_dev(scores), G, k, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == expect_status
    return as_np(acc), as_np(rej), as_np(flags)


def _check_k(scores, G, k):
    acc, rej, flags = _gpu_select_k(scores, G, k)
    st, oacc, orej, oflag = oracle.select(scores, G, k)
    assert st == 0
    np.testing.assert_array_equal(acc, oacc)
    np.testing.assert_array_equal(rej, orej)
    np.testing.assert_array_equal(flags, oflag)


@pytest.mark.parametrize("U", [1, 2, 7, 64, 511, 512, 513, 2048, 5000, 131072, 1048576])
@pytest.mark.parametrize("dist", ["ties", "continuous", "constant"])
def test_select_k_matches_oracle(U, dist):
    rng = np.random.default_rng(U + len(dist))
    if dist == "ties":
        s = rng.integers(0, 9, size=U).astype(np.float64) / 4.0
    elif dist == "continuous":
        s = rng.random(U) * 40.0
    else:
        s = np.full(U, 2.5)
    ks = sorted({0, 1, U // 3, U // 2, U - 1, U} - {-1})
    G = 8 if U <= 131072 else 1
    for k in ks:
        if 0 <= k <= U:
            _check_k(s, G, k)


def test_select_handles_negative_zero_and_subnormals():
    s = np.array([0.0, -0.0, 5e-324, 1e-310, 0.0, 3.0, -0.0, 5e-324] * 100, np.float64)
    for k in (1, 3, 100, 401, 799):
        _check_k(s, 1, k)


@pytest.mark.parametrize("name,n", [("tiny", None), ("math7b", 512), ("math7b", 768),
                                    ("multiturn", 480), ("moe", None), ("sweep", 16384)])
@pytest.mark.parametrize("beta,r_prev", [(0.0, 0.0), (0.5, 0.2)])
def test_select_with_budget_on_workloads(name, n, beta, r_prev):
    pool = workloads.make_pool(name, n_traj=n)
    g, o = pool_score_case(pool)
    U = pool.n_traj // pool.group_size
    bp = pace.budget_params(pool.n_target, beta=beta, r_max=0.9, r_hat_prev=r_prev)
    status = pace.new_status(DEV)
    r_hat, k, acc, rej, flags = pace.select(to_dev(g["unit_score"]), pool.group_size, bp,
                                            status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    st, r, orh, ok = oracle.budget(pool.n_traj, pool.n_target, beta, 0.9, r_prev, U)
    assert (r_hat, k) == (orh, ok)
    st, oacc, orej, oflag = oracle.select(o["unit_score"], pool.group_size, ok)
    np.testing.assert_array_equal(as_np(acc), oacc)
    np.testing.assert_array_equal(as_np(rej), orej)
    np.testing.assert_array_equal(as_np(flags), oflag)


def test_nan_scores_are_reported():
    s = np.arange(600, dtype=np.float64)
    s[17] = np.nan
    _gpu_select_k(s, 1, 10, expect_status=pace.ERR_NAN_INPUT)
    s = np.arange(40, dtype=np.float64)
    s[3] = np.nan
    _gpu_select_k(s, 2, 5, expect_status=pace.ERR_NAN_INPUT)
