"""Pins of the oracle's pool scoring (Eqs. 1-2, 7-10) to facts fixed outside it.

* a hand-worked pool with exact rational answers (tests/golden/hand_pool.json);
* the Lemma 1 identity sum_t (j - v_t) = sum_t (c - v_t) + T (j - c), exact in
  integers, on random pools;
* closed forms of phi_gamma (gamma = 1 is the identity, endpoints, the median);
* the ECDF against a sort + binary search of a library routine.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_pool.json")


def _hand():
    with open(GOLDEN) as f:
        return json.load(f)


def _pool_arrays(h):
    tr = h["trajectories"]
    tags = np.concatenate([np.array(t["tags"], np.int32) for t in tr])
    lens = [len(t["tags"]) for t in tr]
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    c = np.array([t["c"] for t in tr], np.int32)
    s_pre = np.array([np.nan if t["s_pre"] is None else t["s_pre"] for t in tr], np.float32)
    window = np.array(h["window"], np.float32)
    return tags, offsets, c, s_pre, window


def _frac(p):
    return Fraction(p[0], p[1])


def _close_to_fraction(x, fr, ulps=4):
    """|x - fr| within a few ulp of fr (x is an fp64 result of a few roundings)."""
    exact = float(fr)
    tol = ulps * np.spacing(max(abs(exact), 1e-300))
    return abs(x - exact) <= tol


def test_hand_pool_staleness_and_lag():
    h = _hand()
    tags, offsets, c, _, _ = _pool_arrays(h)
    j = h["trainer_version"]
    st, gsum, tcount, kgen, kwait = oracle.staleness(tags, offsets, c, j)
    assert st == oracle.OK
    st2, lsum, tcount2, kbar = oracle.policy_lag(tags, offsets, j)
    assert st2 == oracle.OK
    for i, t in enumerate(h["trajectories"]):
        # K_gen and K_wait of the hand pool are dyadic rationals: exact in fp64.
        assert Fraction(kgen[i]) == _frac(t["kgen"]), i
        assert Fraction(kwait[i]) == _frac(t["kwait"]), i
        assert Fraction(kbar[i]) == _frac(t["kbar"]), i
        assert tcount[i] == len(t["tags"]) == tcount2[i]


@pytest.mark.parametrize("mode,key", [(oracle.MODE_EFF, "eff"), (oracle.MODE_RAW, "raw"),
                                      (oracle.MODE_GEN, "gen")])
def test_hand_pool_scores(mode, key):
    h = _hand()
    tags, offsets, c, s_pre, window = _pool_arrays(h)
    st, kgen, kwait, w, score, us = oracle.score_pool(
        tags, offsets, c, s_pre, h["trainer_version"], window, mode=mode, gamma=h["gamma"],
        min_obs=h["min_obs"], f_missing=h["f_missing"], group_size=1)
    assert st == oracle.OK
    for i, t in enumerate(h["trajectories"]):
        if t["q"] is not None:
            assert Fraction(oracle.ecdf(window, t["s_pre"])) == _frac(t["q"])
        assert _close_to_fraction(w[i], _frac(t["F"])), (i, w[i], t["F"])
        assert _close_to_fraction(score[i], _frac(t[key])), (i, score[i], t[key])
    np.testing.assert_array_equal(us, score)  # G = 1: unit score is the score


@pytest.mark.parametrize("case", range(5))
def test_hand_pool_budget_and_selection(case):
    h = _hand()
    bc = h["budget_cases"][case]
    G = bc["group_size"]
    n_units = bc["n_traj"] // G
    st, r, r_hat, k = oracle.budget(bc["n_traj"], bc["n_target"], bc["beta"], bc["r_max"],
                                    bc["r_hat_prev"], n_units)
    assert st == oracle.OK
    assert _close_to_fraction(r, _frac(bc["r"]))
    assert _close_to_fraction(r_hat, _frac(bc["r_hat"]))
    assert k == bc["k"]
    if "rejected" not in bc:
        return
    tags, offsets, c, s_pre, window = _pool_arrays(h)
    modes = {"eff": oracle.MODE_EFF, "raw": oracle.MODE_RAW, "gen": oracle.MODE_GEN}
    for key, expect in bc["rejected"].items():
        st, *_, us = oracle.score_pool(tags, offsets, c, s_pre, h["trainer_version"], window,
                                       mode=modes[key], gamma=h["gamma"], min_obs=h["min_obs"],
                                       f_missing=h["f_missing"], group_size=G)
        assert st == oracle.OK
        if "unit_eff" in bc and key == "eff":
            for u, fr in enumerate(bc["unit_eff"]):
                assert _close_to_fraction(us[u], _frac(fr)), (u, us[u])
        st, acc, rej, flag = oracle.select(us, G, k)
        assert st == oracle.OK
        assert rej.tolist() == expect
        assert sorted(acc.tolist() + rej.tolist()) == list(range(bc["n_traj"]))
        assert acc.tolist() == sorted(acc.tolist())
        assert flag.tolist() == [0 if i in expect else 1 for i in range(bc["n_traj"])]


def _random_pool(rng, n, j, max_len=40, tool_frac=0.0):
    lens = rng.integers(0, max_len + 1, size=n)
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    c = rng.integers(0, j + 1, size=n).astype(np.int32)
    tags = np.empty(offsets[-1], np.int32)
    for i in range(n):
        seg = rng.integers(0, c[i] + 1, size=lens[i])
        seg = np.sort(seg)  # versions never decrease within a rollout
        tool = rng.random(lens[i]) < tool_frac
        seg[tool] = -1
        tags[offsets[i]:offsets[i + 1]] = seg
    return tags, offsets, c


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_lemma1_identity_exact(seed):
    """Lemma 1: sum (j - v_t) = sum (c - v_t) + T (j - c), exactly, and both parts >= 0."""
    rng = np.random.default_rng(seed)
    j = 50
    tags, offsets, c = _random_pool(rng, 200, j, tool_frac=0.2)
    st, gsum, tcount, kgen, kwait = oracle.staleness(tags, offsets, c, j)
    assert st == oracle.OK
    st, lsum, tcount2, kbar = oracle.policy_lag(tags, offsets, j)
    assert st == oracle.OK
    np.testing.assert_array_equal(tcount, tcount2)
    np.testing.assert_array_equal(lsum, gsum + tcount * (j - c.astype(np.int64)))
    assert (kgen >= 0).all() and (kwait >= 0).all()
    nz = tcount > 0
    np.testing.assert_allclose(kbar[nz], (kgen + kwait)[nz], rtol=1e-15, atol=0)
    # tool tokens (tag -1) are not counted
    for i in range(5):
        seg = tags[offsets[i]:offsets[i + 1]]
        assert tcount[i] == int((seg != -1).sum())


def test_zero_staleness_when_all_tags_current():
    j = 17
    lens = np.array([5, 1, 9, 0, 3])
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tags = np.full(offsets[-1], j, np.int32)
    c = np.full(5, j, np.int32)
    s_pre = np.array([0.1, np.nan, 0.7, 0.2, np.nan], np.float32)
    window = np.linspace(0.05, 0.95, 64).astype(np.float32)
    for mode in (oracle.MODE_EFF, oracle.MODE_RAW, oracle.MODE_GEN):
        st, kgen, kwait, w, score, us = oracle.score_pool(tags, offsets, c, s_pre, j, window,
                                                          mode=mode, group_size=5)
        assert st == oracle.OK
        assert (kgen == 0).all() and (kwait == 0).all() and (score == 0).all() and (us == 0).all()


def test_sharpen_closed_forms():
    for q in [0.0, 0.125, 0.3, 0.5, 0.77, 1.0]:
        assert oracle.sharpen(q, 1) == q  # gamma = 1 recovers the linear map
    for g in [1, 2, 3, 4, 8]:
        assert oracle.sharpen(0.0, g) == 0.0
        assert oracle.sharpen(1.0, g) == 1.0
        assert oracle.sharpen(0.5, g) == 0.5
    # gamma = 2 closed form: q^2 / (q^2 + (1-q)^2), exact rationals for dyadic q
    for num in range(0, 9):
        q = Fraction(num, 8)
        expect = q ** 2 / (q ** 2 + (1 - q) ** 2)
        assert _close_to_fraction(oracle.sharpen(float(q), 2), expect, ulps=2)
    # monotone and symmetric about the median
    qs = np.linspace(0, 1, 101)
    f = np.array([oracle.sharpen(q, 4) for q in qs])
    assert (np.diff(f) >= 0).all()
    np.testing.assert_allclose(f + f[::-1], 1.0, atol=1e-15)


def test_ecdf_matches_sorted_search():
    rng = np.random.default_rng(7)
    window = rng.random(512).astype(np.float32)
    window[10] = window[11]  # duplicates
    srt = np.sort(window)
    probes = np.concatenate([window[:50], rng.random(50).astype(np.float32),
                             np.array([-1.0, 0.0, 1.0, 2.0], np.float32)])
    for s in probes:
        expect = np.searchsorted(srt, s, side="right") / window.size
        assert oracle.ecdf(window, s) == expect


def test_window_below_min_obs_falls_back_to_raw_weight():
    h = _hand()
    tags, offsets, c, s_pre, window = _pool_arrays(h)
    st, kgen, kwait, w, score, _ = oracle.score_pool(tags, offsets, c, s_pre, 10, window,
                                                     mode=oracle.MODE_EFF, min_obs=32,
                                                     group_size=1)
    assert st == oracle.OK
    assert (w == 1.0).all()
    np.testing.assert_array_equal(score, kwait + kgen)


def test_missing_prefix_score_uses_f_missing():
    h = _hand()
    tags, offsets, c, s_pre, window = _pool_arrays(h)
    st, kgen, kwait, w, score, _ = oracle.score_pool(tags, offsets, c, s_pre, 10, window,
                                                     min_obs=1, f_missing=0.25, group_size=1)
    assert st == oracle.OK
    assert w[0] == w[2] == w[3] == 0.25


def test_errors():
    h = _hand()
    tags, offsets, c, s_pre, window = _pool_arrays(h)
    bad = tags.copy()
    bad[0] = 11  # v_t > c
    assert oracle.score_pool(bad, offsets, c, s_pre, 10, window, group_size=1)[0] == \
        oracle.ERR_VERSION_ORDER
    assert oracle.score_pool(tags, offsets, c, s_pre, 9, window, group_size=1)[0] == \
        oracle.ERR_VERSION_ORDER  # c > j
    bad = tags.copy()
    bad[3] = -2
    assert oracle.score_pool(bad, offsets, c, s_pre, 10, window, group_size=1)[0] == \
        oracle.ERR_INVALID_ARG
    wn = window.copy()
    wn[2] = np.nan
    assert oracle.score_pool(tags, offsets, c, s_pre, 10, wn, group_size=1)[0] == \
        oracle.ERR_NAN_INPUT
    assert oracle.score_pool(tags, offsets, c, s_pre, 10, window, group_size=4)[0] == \
        oracle.ERR_INVALID_ARG  # 6 trajectories are not whole groups of 4


def test_stale_k_admission_on_hand_pool():
    h = _hand()
    tags, offsets, c, _, _ = _pool_arrays(h)
    kbars = [_frac(t["kbar"]) for t in h["trajectories"]]  # 0, 5/2, 4, 1, 9/2, 5/4
    for k in (0.0, 1.0, 1.25, 2.5, 4.0, 4.5, 10.0):
        st, kbar, adm = oracle.stale_k(tags, offsets, 10, k)
        assert st == oracle.OK
        for i, kb in enumerate(kbars):
            assert Fraction(kbar[i]) == kb
            assert adm[i] == (1 if kb <= Fraction(k) else 0), (k, i)  # kbar == k admitted


def test_histogram_hand_counts():
    vals = np.array([-1.0, 0.0, 0.49, 0.5, 0.99, 1.0, 1.5, 7.0])
    flags = np.array([0, 1, 1, 0, 1, 0, 1, 1], np.uint8)
    st, h = oracle.histogram(vals, flags, 0.0, 1.0, 2)
    assert st == oracle.OK
    # bins [0, .5) and [.5, 1); below lo -> bin 0, at or above hi -> bin 1
    assert h[0].tolist() == [1, 2]  # rejected: -1.0 | 0.5, 1.0
    assert h[1].tolist() == [2, 3]  # accepted: 0.0, 0.49 | 0.99, 1.5, 7.0
    assert h.sum() == vals.size
    st, h = oracle.histogram(np.array([np.nan]), None, 0.0, 1.0, 4)
    assert st == oracle.ERR_NAN_INPUT
