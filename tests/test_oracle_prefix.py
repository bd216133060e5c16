"""Pins of the oracle's Prefix Forgetting Score (Eq. 6) and its collection
rules (at least 32 eligible tokens; only the first 1,024 / 2,048 scored)."""
import math

import numpy as np

import oracle


def test_hand_worked_prefixes():
    # prefix 0: 4 eligible rows, |d| = 0.5, 0.1, 0.3, 0.1 -> mean 0.25
    # prefix 1: rows 4..9 with rows 5 and 7 masked out: |d| = 1, 2, 3, 4 -> 2.5
    lp = np.array([-1.0, -2.0, -0.5, -3.0, -1.0, 9.0, -2.0, 9.0, -3.0, -4.0])
    bl = np.array([-1.5, -1.9, -0.8, -2.9, 0.0, 0.0, 0.0, 0.0, 0.0, 0.0])
    mask = np.array([1, 1, 1, 1, 1, 0, 1, 0, 1, 1], np.uint8)
    st, s = oracle.prefix_score(lp, bl, [0, 4, 10], mask=mask, min_tokens=1, cap_tokens=100)
    assert st == 0
    assert abs(s[0] - 0.25) < 1e-15 and abs(s[1] - 2.5) < 1e-15


def test_zero_and_constant_drift():
    rng = np.random.default_rng(0)
    so = np.array([0, 40, 100, 1300], np.int64)
    lp = -rng.random(so[-1]) * 8
    st, s = oracle.prefix_score(lp, lp, so)
    assert st == 0 and (s == 0).all()
    st, s = oracle.prefix_score(lp, lp + 0.375, so)
    assert np.allclose(s, 0.375, rtol=0, atol=1e-12)  # |delta| for a constant shift
    st, s = oracle.prefix_score(lp, lp - 0.375, so)
    assert np.allclose(s, 0.375, rtol=0, atol=1e-12)


def test_min_tokens_boundary_and_cap():
    so = np.array([0, 31, 63, 2063], np.int64)  # 31, 32 and 2000 eligible rows
    lp = np.zeros(so[-1])
    bl = np.ones(so[-1])
    bl[63 + 1024:] = 100.0  # beyond the cap: must not count
    st, s = oracle.prefix_score(lp, bl, so, min_tokens=32, cap_tokens=1024)
    assert st == 0
    assert math.isnan(s[0]) and s[1] == 1.0 and s[2] == 1.0
    st, s = oracle.prefix_score(lp, bl, so, min_tokens=32, cap_tokens=2048)
    assert abs(s[2] - (1024 + 976 * 100.0) / 2000) < 1e-12
    # ineligible rows neither count toward the minimum nor the cap
    mask = np.ones(so[-1], np.uint8)
    mask[31:33] = 0
    st, s = oracle.prefix_score(lp, bl, so, mask=mask, min_tokens=32, cap_tokens=1024)
    assert math.isnan(s[1])
