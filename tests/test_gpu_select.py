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


# 1..512 units: the one-block rank kernel; 513..131072: the one-cluster adaptive
# radix select (1-8 CTAs); above: the multi-block radix select.
@pytest.mark.parametrize("U", [1, 2, 7, 64, 511, 512, 513, 2048, 5000, 16384, 16385, 70001,
                               131072, 131073, 1048576])
@pytest.mark.parametrize("dist", ["ties", "continuous", "constant", "ulps", "signed_wide"])
def test_select_k_matches_oracle(U, dist):
    rng = np.random.default_rng(U + len(dist))
    if dist == "ties":
        s = rng.integers(0, 9, size=U).astype(np.float64) / 4.0
    elif dist == "continuous":
        s = rng.random(U) * 40.0
    elif dist == "ulps":  # keys that differ only in their last two bits
        s = 1.0 + rng.integers(0, 4, size=U) * np.finfo(np.float64).eps
    elif dist == "signed_wide":  # both signs, magnitudes from 1e-300 to 1e300
        s = np.where(rng.random(U) < 0.5, -1.0, 1.0) * 10.0 ** rng.uniform(-300, 300, size=U)
    else:
        s = np.full(U, 2.5)
    ks = sorted({0, 1, U // 3, U // 2, U - 1, U} - {-1})
    G = 8 if U <= 131072 else 1
    for k in ks:
        if 0 <= k <= U:
            _check_k(s, G, k)


@pytest.mark.parametrize("U", [513, 1000, 2047, 4095, 4096, 4097])
@pytest.mark.parametrize("dist", ["ties", "continuous", "ulps", "signed_wide"])
def test_one_cta_pools(U, dist):
    """One CTA holds the pool (G = 1) around the sizes where a cluster of one
    CTA gives way to larger clusters: ids exact."""
    rng = np.random.default_rng(7 * U + len(dist))
    if dist == "ties":
        s = rng.integers(0, 5, size=U).astype(np.float64)
    elif dist == "continuous":
        s = rng.random(U) * 40.0
    elif dist == "ulps":
        s = 1.0 + rng.integers(0, 4, size=U) * np.finfo(np.float64).eps
    else:
        s = np.where(rng.random(U) < 0.5, -1.0, 1.0) * 10.0 ** rng.uniform(-300, 300, size=U)
    for k in (1, 2, U // 3, U // 2, U - 1, U):
        _check_k(s, 1, k)


@pytest.mark.parametrize("reps", [50, 100, 1000])  # 400, 800 and 8000 units
def test_select_handles_negative_zero_and_subnormals(reps):
    s = np.array([0.0, -0.0, 5e-324, 1e-310, 0.0, 3.0, -0.0, 5e-324] * reps, np.float64)
    n = s.size
    for k in (1, 3, 100, n // 2 + 1, n - 1):
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
    for n in (600, 20000):
        s = np.arange(n, dtype=np.float64)
        s[17] = np.nan
        _gpu_select_k(s, 1, 10, expect_status=pace.ERR_NAN_INPUT)
    s = np.arange(40, dtype=np.float64)
    s[3] = np.nan
    _gpu_select_k(s, 2, 5, expect_status=pace.ERR_NAN_INPUT)


@pytest.mark.parametrize("U", [513, 16384])
def test_mid_size_pools_take_no_workspace(U):
    """Pools of up to 16,384 units are selected by one block without the caller's
    workspace: a NULL workspace of 0 bytes is accepted and gives the oracle's ids."""
    import ctypes
    rng = np.random.default_rng(U)
    s = rng.integers(0, 50, size=U).astype(np.float64) / 8.0
    k = U // 3
    G = 2
    scores = to_dev(s)
    acc = torch.full((U * G,), -7, dtype=torch.int32, device=DEV)
    rej = torch.full((U * G,), -7, dtype=torch.int32, device=DEV)
    flags = torch.full((U * G,), 9, dtype=torch.uint8, device=DEV)
    status = pace.new_status(DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = pace.lib().pace_select_k(ctypes.c_void_p(scores.data_ptr()), U, G, k,
                                  ctypes.c_void_p(acc.data_ptr()), ctypes.c_void_p(rej.data_ptr()),
                                  ctypes.c_void_p(flags.data_ptr()), None, 0,
                                  ctypes.c_void_p(status.data_ptr()), stream)
    assert st == pace.OK, pace.status_string(st)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    _, oacc, orej, oflag = oracle.select(s, G, k)
    np.testing.assert_array_equal(as_np(acc)[:(U - k) * G], oacc)
    np.testing.assert_array_equal(as_np(rej)[:k * G], orej)
    np.testing.assert_array_equal(as_np(flags), oflag)


@pytest.mark.parametrize("U,G", [(600, 3), (3000, 12), (3000, 100), (5000, 7), (16384, 3),
                                 (700, 1500)])
def test_select_group_sizes(U, G):
    """Group sizes that do and do not divide 1024 (the writers step through
    positions 1024 at a time), clusters of 1 to 8 CTAs on the one-launch path."""
    rng = np.random.default_rng(U * 31 + G)
    s = rng.integers(0, 200, size=U).astype(np.float64) / 16.0
    for k in (1, U // 4, U - 1):
        _check_k(s, G, k)


@pytest.mark.parametrize("U,G", [(5000, 2), (70000, 1), (300000, 1)])
def test_select_without_optional_outputs(U, G):
    """rejected_ids and traj_accepted may be NULL: the accepted ids alone, on the
    one-CTA, multi-CTA and radix paths."""
    import ctypes
    rng = np.random.default_rng(U + 3)
    s = rng.random(U) * 30.0
    k = U // 5
    scores = to_dev(s)
    acc = torch.full((U * G,), -7, dtype=torch.int32, device=DEV)
    L = pace.lib()
    ws = pace.workspace(L.pace_select_workspace_size(U), DEV)
    status = pace.new_status(DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = L.pace_select_k(ctypes.c_void_p(scores.data_ptr()), U, G, k,
                         ctypes.c_void_p(acc.data_ptr()), None, None,
                         ctypes.c_void_p(ws.data_ptr()), ws.numel(),
                         ctypes.c_void_p(status.data_ptr()), stream)
    assert st == pace.OK, pace.status_string(st)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    _, oacc, _, _ = oracle.select(s, G, k)
    got = as_np(acc)
    np.testing.assert_array_equal(got[:(U - k) * G], oacc)
    assert (got[(U - k) * G:] == -7).all()  # nothing written past the accepted ids


def test_select_random_shapes():
    """Random pool sizes across the one-launch range (513..131,072 units, clusters of
    1-8 CTAs), random group sizes, budgets and score distributions: ids exact."""
    rng = np.random.default_rng(2026)
    for case in range(40):
        U = int(rng.integers(513, 131073)) if case % 4 else int(rng.integers(513, 4096))
        G = int(rng.choice([1, 2, 3, 8, 12]))
        if U * G > 600_000:
            G = 1
        kind = case % 5
        if kind == 0:
            s = rng.random(U) * 40.0
        elif kind == 1:
            s = rng.integers(0, 12, size=U).astype(np.float64) / 8.0
        elif kind == 2:
            s = np.round(rng.normal(10.0, 3.0, size=U), 3)
        elif kind == 3:
            s = rng.choice([0.0, 1.5, 1.5 + 2.0 ** -40, 7.25], size=U)
        else:
            s = np.exp(rng.normal(0.0, 20.0, size=U))
        k = int(rng.integers(1, U))
        _check_k(s, G, k)


@pytest.mark.parametrize("U,G", [(3000, 4), (3000, 8), (20000, 12), (131072, 8)])
def test_select_outputs_at_unaligned_addresses(U, G):
    """Groups that are a multiple of 4 are written four ids at a time when the
    buffers allow it; buffers 4 bytes (ids) or 1 byte (flags) off alignment take
    the element-wise writer.  Both give the oracle's ids."""
    import ctypes
    rng = np.random.default_rng(U * 7 + G)
    s = rng.integers(0, 300, size=U).astype(np.float64) / 4.0
    k = U // 3
    n = U * G
    scores = to_dev(s)
    acc = torch.full((n + 4,), -7, dtype=torch.int32, device=DEV)
    rej = torch.full((n + 4,), -7, dtype=torch.int32, device=DEV)
    flags = torch.full((n + 4,), 9, dtype=torch.uint8, device=DEV)
    status = pace.new_status(DEV)
    L = pace.lib()
    ws = pace.workspace(L.pace_select_workspace_size(U), DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for off_ids, off_flags in ((0, 0), (1, 0), (0, 1)):
        st = L.pace_select_k(ctypes.c_void_p(scores.data_ptr()), U, G, k,
                             ctypes.c_void_p(acc.data_ptr() + 4 * off_ids),
                             ctypes.c_void_p(rej.data_ptr() + 4 * off_ids),
                             ctypes.c_void_p(flags.data_ptr() + off_flags),
                             ctypes.c_void_p(ws.data_ptr()), ws.numel(),
                             ctypes.c_void_p(status.data_ptr()), stream)
        assert st == pace.OK, pace.status_string(st)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        _, oacc, orej, oflag = oracle.select(s, G, k)
        np.testing.assert_array_equal(as_np(acc)[off_ids:off_ids + (U - k) * G], oacc)
        np.testing.assert_array_equal(as_np(rej)[off_ids:off_ids + k * G], orej)
        np.testing.assert_array_equal(as_np(flags)[off_flags:off_flags + n], oflag)
