"""Pins of the oracle's budget (Eqs. 3-4 + cap) and top-k rejection.

* the budget against exact rational arithmetic (fractions.Fraction) over a
  sweep of pool sizes, including the pairs where a plain fp64 floor lands one
  below the surplus (e.g. N = 47, N_tar = 35);
* the selection against brute-force enumeration of every k-subset on tiny pools
  with heavy ties: the rejected set is the subset whose members, listed by
  (score descending, id ascending), form the lexicographically greatest
  sequence.
"""
import itertools
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle


def _exact_k(n, n_tar, beta, r_hat_prev, r_max, units):
    r = Fraction(max(n - n_tar, 0), max(n, 1))
    r = min(max(r, Fraction(0)), Fraction(1))
    r_hat = Fraction(beta) * Fraction(r_hat_prev) + (1 - Fraction(beta)) * r
    r_eff = min(r_hat, Fraction(r_max))
    return min(math.floor(r_eff * units), units)


def test_budget_zero_at_or_below_target():
    for n in range(0, 200, 7):
        for n_tar in range(n, n + 50, 5):
            st, r, r_hat, k = oracle.budget(n, n_tar, 0.0, 0.9, 0.0, max(n // 8, 1))
            assert st == oracle.OK and r == 0.0 and r_hat == 0.0 and k == 0


def test_budget_regression_47_35():
    # (47 - 35) / 47 * 47 is 11.999999999999998 in fp64; the surplus is 12.
    assert math.floor(((47 - 35) / 47) * 47) == 11
    assert oracle.budget(47, 35, 0.0, 0.9, 0.0, 47)[3] == 12


def test_budget_matches_rational_sweep():
    rng = np.random.default_rng(3)
    mism = 0
    for n in list(range(1, 400)) + list(rng.integers(400, 2_000_000, size=300)):
        n = int(n)
        for n_tar in {0, n // 4, n // 2, (3 * n) // 4, n - 1, int(rng.integers(0, n + 1))}:
            for g in (1, 8, 12):
                units = max(n // g, 1)
                st, r, r_hat, k = oracle.budget(n, n_tar, 0.0, 0.9, 0.0, units)
                assert st == oracle.OK
                # the r_max cap is stated as the real number 0.9; its fp64 value
                # is a hair above, which never moves a floor for U <= 2^21.
                expect = _exact_k(n, n_tar, 0, 0, Fraction(9, 10), units)
                mism += k != expect
    assert mism == 0


def test_budget_ema_against_rationals():
    # beta and r_hat_prev as exact binary fractions, so the rational answer is
    # the one the paper's formula defines for the fp64 inputs.
    for beta in (0.0, 0.25, 0.5, 0.75, 0.875):
        for r_prev in (0.0, 0.125, 0.5, 0.625):
            for n, n_tar in ((64, 48), (512, 384), (480, 192), (1000, 999), (7, 1)):
                units = n // 1
                st, r, r_hat, k = oracle.budget(n, n_tar, beta, 0.9, r_prev, units)
                assert st == oracle.OK
                exact = _exact_k(n, n_tar, Fraction(beta), Fraction(r_prev), Fraction(9, 10),
                                 units)
                assert k == exact, (beta, r_prev, n, n_tar, k, exact)


def test_budget_rejects_bad_parameters():
    assert oracle.budget(10, 5, 1.0, 0.9, 0.0, 10)[0] == oracle.ERR_INVALID_ARG  # beta < 1
    assert oracle.budget(10, 5, -0.1, 0.9, 0.0, 10)[0] == oracle.ERR_INVALID_ARG
    assert oracle.budget(10, 5, 0.0, 1.5, 0.0, 10)[0] == oracle.ERR_INVALID_ARG


def _brute_force_rejected(scores, k):
    best, best_key = None, None
    for sub in itertools.combinations(range(len(scores)), k):
        key = sorted(((-scores[u], u) for u in sub))
        # lexicographically greatest sequence of (score desc, id asc) ==
        # lexicographically smallest sequence of (-score, id)
        if best_key is None or key < best_key:
            best, best_key = sub, key
    return sorted(best)


@pytest.mark.parametrize("seed", range(6))
def test_select_matches_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    for _ in range(40):
        u = int(rng.integers(1, 11))
        scores = rng.integers(0, 4, size=u).astype(np.float64) / 2.0  # many ties
        if rng.random() < 0.5:
            scores += rng.random(u) * 1e-3 * (rng.random(u) < 0.5)
        g = int(rng.choice([1, 2, 3]))
        for k in range(0, u + 1):
            st, acc, rej, flag = oracle.select(scores, g, k)
            assert st == oracle.OK
            units = _brute_force_rejected(list(scores), k)
            expect = [uu * g + i for uu in units for i in range(g)]
            assert rej.tolist() == expect
            assert acc.tolist() == [i for i in range(u * g) if i not in set(expect)]


def test_select_errors():
    assert oracle.select(np.array([1.0, np.nan]), 1, 1)[0] == oracle.ERR_NAN_INPUT


def test_quantile_admit_hand_worked():
    # window {1..8}, r = 1/4: type-1 quantile at 3/4 -> 6th smallest = 6; reject scores > 6
    w = oracle.Window(8)
    st, dec, kappa = oracle.quantile_admit(np.arange(1, 9, dtype=np.float64), 0.0, 0, w,
                                           min_obs=100)
    assert st == 0 and kappa == math.inf and (dec == 1).all()  # below min_obs: no threshold
    assert w.count == 8 and w.head == 0
    st, dec, kappa = oracle.quantile_admit([7.0, 2.0, 6.0, 9.0, 1.0, 3.0], 0.25, 3, w, min_obs=4)
    assert st == 0 and kappa == 6.0
    # draw: 7 rejected, 2 kept, 6 kept (ties at kappa kept), 9 rejected, 1 kept -> 3 kept, stop
    assert dec.tolist() == [0, 1, 1, 0, 1, 2]
    # the five drawn scores replaced the five oldest window slots
    assert w.count == 8 and w.head == 5
    assert sorted(w.values.tolist()) == sorted([6.0, 7.0, 8.0, 7.0, 2.0, 6.0, 9.0, 1.0])


def test_quantile_admit_matches_numpy_inverted_cdf():
    rng = np.random.default_rng(8)
    for _ in range(200):
        n = int(rng.integers(1, 600))
        vals = np.round(rng.random(n) * 20, 1)
        # dyadic r: (1 - r) * n is exact in fp64, so numpy's quantile and the
        # rule agree without the 1e-9 nudge
        r = float(rng.choice([0.0, 0.125, 0.25, 0.5, 0.75, 0.875, 1.0]))
        w = oracle.Window(1024)
        w.values[:n] = vals
        w.count, w.head = n, n % 1024
        st, dec, kappa = oracle.quantile_admit(np.zeros(0), r, 0, w, min_obs=1)
        assert st == 0
        p = 1.0 - r
        expect = np.quantile(vals, max(p, 1e-12), method="inverted_cdf")
        assert kappa == expect, (n, r)


def test_quantile_admit_rank_is_the_real_number_rank():
    # r = 1/3 over 189 values: (1 - r) n is 126 as a real number but 126.00000000000001
    # in fp64; the rule takes the 126th smallest (reading: the nudge), not the 127th.
    vals = np.arange(1, 190, dtype=np.float64)
    w = oracle.Window(256)
    w.values[:189] = vals
    w.count, w.head = 189, 189
    st, _, kappa = oracle.quantile_admit(np.zeros(0), 1 / 3, 0, w, min_obs=1)
    assert st == 0 and kappa == 126.0
