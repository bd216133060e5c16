"""Stale-k admission, staleness histograms and the literal sliding-window
quantile rule on the GPU vs the oracle: kbar fp64 bits, admitted flags,
histogram counts, kappa, decisions and the window ring state all identical."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from pace_cases import DEV, as_np, assert_bits_equal, oracle_score, to_dev
from paper_2609_36830_gb300 import pace, workloads

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_pool.json")


def _hand_arrays():
    h = json.load(open(GOLDEN))
    tr = h["trajectories"]
    tags = np.concatenate([np.array(t["tags"], np.int32) for t in tr])
    offsets = np.concatenate([[0], np.cumsum([len(t["tags"]) for t in tr])]).astype(np.int64)
    return tags, offsets, h["trainer_version"]


def _pools():
    out = [("hand",) + _hand_arrays()]
    for name, n in [("tiny", None), ("math7b", 512), ("multiturn", 480), ("sweep", 16384)]:
        p = workloads.make_pool(name, n_traj=n)
        out.append((name, p.tags, p.meta["offsets_host"], p.trainer_version))
    return out


@pytest.mark.parametrize("k_max", [0.0, 1.0, 2.5, 4.0, 8.0, 31.5])
def test_stale_k_matches_oracle(k_max):
    for name, tags, offsets, j in _pools():
        status = pace.new_status(DEV)
        kbar, adm = pace.stale_k(to_dev(tags), to_dev(offsets), j, k_max, status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        st, okbar, oadm = oracle.stale_k(tags, offsets, j, k_max)
        assert st == 0
        assert_bits_equal(as_np(kbar), okbar, f"{name} kbar")
        np.testing.assert_array_equal(as_np(adm), oadm)


def test_stale_k_reports_tag_above_trainer_version():
    tags, offsets, j = _hand_arrays()
    status = pace.new_status(DEV)
    pace.stale_k(to_dev(tags), to_dev(offsets), j - 1, 1.0, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == pace.ERR_VERSION_ORDER


@pytest.mark.parametrize("n_bins,lo,hi", [(1, 0.0, 1.0), (7, 0.0, 8.0), (64, 0.5, 6.0),
                                          (4096, 0.0, 32.0)])
def test_histograms_match_oracle(n_bins, lo, hi):
    pool = workloads.make_pool("sweep", n_traj=16384)
    o = oracle_score(pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
                     pool.trainer_version, pool.window, group_size=8)
    U = pool.n_traj // 8
    _, _, _, k = oracle.budget(pool.n_traj, pool.n_target, 0.0, 0.9, 0.0, U)
    _, _, _, flags = oracle.select(o["unit_score"], 8, k)
    for key in ("kwait", "kgen", "score"):
        vals = o[key]
        hist = pace.staleness_histogram(to_dev(vals), to_dev(flags), lo, hi, n_bins)
        st, oh = oracle.histogram(vals, flags, lo, hi, n_bins)
        assert st == 0
        np.testing.assert_array_equal(as_np(hist).astype(np.uint32), oh)
    unit_flags = flags[::8].copy()
    hist = pace.staleness_histogram(to_dev(o["unit_score"]), to_dev(unit_flags), lo, hi, n_bins)
    _, oh = oracle.histogram(o["unit_score"], unit_flags, lo, hi, n_bins)
    np.testing.assert_array_equal(as_np(hist).astype(np.uint32), oh)


@pytest.mark.parametrize("capacity,batch,min_obs", [(512, 40, 32), (64, 0, 8), (4096, 100, 32)])
def test_quantile_admission_over_steps(capacity, batch, min_obs):
    """Five consecutive trainer steps, each on a fresh pool; both sides carry their own window."""
    gw = pace.ScoreWindow(capacity, DEV)
    ow = oracle.Window(capacity)
    for step in range(5):
        pool = workloads.make_pool("math7b", seed=7000 + step, n_traj=[512, 768, 384, 640, 512][step])
        o = oracle_score(pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
                         pool.trainer_version, pool.window, group_size=8)
        U = pool.n_traj // 8
        _, _, r_hat, _ = oracle.budget(pool.n_traj, pool.n_target, 0.5, 0.9, 0.1 * step, U)
        r_eff = min(r_hat, 0.9)
        status = pace.new_status(DEV)
        dec, kap = pace.quantile_admit(to_dev(o["unit_score"]), r_eff, batch, gw,
                                       min_obs=min_obs, status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        st, odec, okap = oracle.quantile_admit(o["unit_score"], r_eff, batch, ow, min_obs=min_obs)
        assert st == 0
        assert float(kap.item()) == okap, step
        np.testing.assert_array_equal(as_np(dec), odec)
        state = as_np(gw.state)
        assert (int(state[0]), int(state[1])) == (ow.count, ow.head)
        np.testing.assert_array_equal(as_np(gw.values)[:ow.count], ow.values[:ow.count])


def test_quantile_admission_large_candidate_list():
    pool = workloads.make_pool("sweep", n_traj=131072 * 8 // 8)
    o = oracle_score(pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
                     pool.trainer_version, pool.window, group_size=8)
    gw, ow = pace.ScoreWindow(512, DEV), oracle.Window(512)
    for r, batch in [(0.0, 0), (0.5, 5000), (0.25, 0)]:
        dec, kap = pace.quantile_admit(to_dev(o["unit_score"]), r, batch, gw)
        torch.cuda.synchronize()
        _, odec, okap = oracle.quantile_admit(o["unit_score"], r, batch, ow)
        assert float(kap.item()) == okap
        np.testing.assert_array_equal(as_np(dec), odec)
