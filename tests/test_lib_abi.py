"""The C-ABI library builds, loads without a GPU and exports every symbol that
include/*.h declares; its host-only budget function matches the oracle bit for
bit; host-side argument checks return before touching the device."""
import ctypes
import glob
import os
import re

import numpy as np
import pytest

import oracle
from paper_2609_36830_gb300 import build as pace_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def pace():
    pace_build.build()
    from paper_2609_36830_gb300 import pace as p
    p.lib()
    return p


def _declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        txt = open(h).read()
        names.update(re.findall(r"PACE_API\s+[\w\s\*]+?\b(pace_\w+)\s*\(", txt))
    return names


def test_every_declared_symbol_is_exported(pace):
    declared = _declared_symbols()
    assert len(declared) >= 16
    L = ctypes.CDLL(pace.LIB_PATH)
    for name in sorted(declared):
        assert hasattr(L, name), name
    # the binding declares a signature for each of them
    assert declared == set(pace.SIGNATURES)


def test_status_strings_and_defaults(pace):
    assert pace.status_string(0) == "PACE_OK"
    assert pace.status_string(2) == "PACE_ERR_VERSION_ORDER"
    assert pace.status_string(99) == "PACE_ERR_UNKNOWN"
    assert pace.lib().pace_version() == 300  # 0.3.0: sharded selection, PaceLossArgs.partial
    sp = pace.PaceScoreParams()
    pace.lib().pace_score_params_default(ctypes.byref(sp))
    assert (sp.mode, sp.gamma, sp.min_obs, sp.group_size, sp.f_missing) == (0, 4, 32, 8, 1.0)
    bp = pace.PaceBudgetParams()
    pace.lib().pace_budget_params_default(ctypes.byref(bp))
    assert (bp.beta, bp.r_max, bp.r_hat_prev) == (0.0, 0.9, 0.0)
    lp = pace.PaceLossParams()
    pace.lib().pace_loss_params_default(ctypes.byref(lp))
    assert lp.eps_low == np.float32(0.2) and lp.eps_high == np.float32(0.28)
    assert lp.dual_clip == 10.0 and lp.agg == 0 and lp.std_unbiased == 1


def test_budget_matches_oracle_bitwise(pace):
    rng = np.random.default_rng(11)
    cases = [(47, 35, 0.0, 0.9, 0.0, 47), (64, 48, 0.0, 0.9, 0.0, 8), (6, 4, 0.5, 0.9, 0.2, 6),
             (100, 0, 0.0, 0.9, 0.0, 100), (10, 20, 0.3, 0.9, 0.5, 10)]
    for _ in range(3000):
        n = int(rng.integers(0, 3_000_000))
        g = int(rng.choice([1, 8, 12, 16]))
        cases.append((n, int(rng.integers(0, n + 2)), float(rng.choice([0.0, 0.3, 0.9, 0.99])),
                      float(rng.choice([0.9, 0.5, 1.0])), float(rng.random()), max(n // g, 0)))
    for n, nt, beta, rmax, prev, u in cases:
        st, r, rh, k = oracle.budget(n, nt, beta, rmax, prev, u)
        assert st == 0
        r2, rh2, k2 = pace.budget(n, u, pace.budget_params(nt, beta, rmax, prev))
        assert (r2, rh2, k2) == (r, rh, k), (n, nt, beta, rmax, prev, u)


def test_budget_rejects_bad_parameters(pace):
    with pytest.raises(pace.PaceError):
        pace.budget(10, 10, pace.budget_params(5, beta=1.0))
    with pytest.raises(pace.PaceError):
        pace.budget(10, 10, pace.budget_params(5, r_max=1.5))


def test_host_argument_checks_return_before_launch(pace):
    L = pace.lib()
    fake = ctypes.c_void_p(0x1000)
    p = pace.score_params(group_size=8)
    # 12 trajectories are not whole groups of 8
    st = L.pace_score_pool(fake, fake, fake, fake, 12, 100, 5, None, 0, ctypes.byref(p), None,
                           None, None, fake, None, fake, 1 << 20, None, None)
    assert st == pace.ERR_INVALID_ARG
    p = pace.score_params(gamma=0)
    st = L.pace_score_pool(fake, fake, fake, fake, 8, 100, 5, None, 0, ctypes.byref(p), None,
                           None, None, fake, None, fake, 1 << 20, None, None)
    assert st == pace.ERR_INVALID_ARG
    p = pace.score_params()
    st = L.pace_score_pool(fake, fake, fake, fake, 8, 100, 5, fake, 5000, ctypes.byref(p), None,
                           None, None, fake, None, fake, 1 << 20, None, None)
    assert st == pace.ERR_UNSUPPORTED_SHAPE  # window longer than 4096
    st = L.pace_select_k(fake, 10, 1, 11, fake, fake, None, fake, 1 << 20, None, None)
    assert st == pace.ERR_INVALID_ARG  # k > U
    b = pace.PaceBatch(fake, None, None, 4, 100)
    st = L.pace_token_logprob(ctypes.byref(b), fake, fake, fake, 100, 1000, 1.0, fake, None,
                              None, fake, 1 << 20, None, None)
    assert st == pace.ERR_UNSUPPORTED_SHAPE  # hidden size not a multiple of 64
    st = L.pace_token_logprob(ctypes.byref(b), fake, fake, fake, 128, 1000, 0.0, fake, None,
                              None, fake, 1 << 20, None, None)
    assert st == pace.ERR_INVALID_ARG  # temperature must be > 0
    # the LM head reads the rows in the loss by index: no copy of the hidden rows
    # in the workspace, so its size does not depend on the hidden size
    ws = L.pace_token_logprob_workspace_size(1000, 10, 128, 1000)
    assert 1000 * 4 < ws < 1000 * 128 * 2
    assert L.pace_token_logprob_workspace_size(1000, 10, 16384, 1000) == ws
    assert L.pace_score_pool_workspace_size(1000, 512) >= 16 * 1000


def test_lmhead_split_control_range(pace):
    L = pace.lib()
    for bad in (-1, 9, 1 << 20):
        assert L.pace_set_lmhead_splits(bad) == pace.ERR_INVALID_ARG
    for good in (0, 1, 2, 4, 8):
        assert L.pace_set_lmhead_splits(good) == pace.OK
    assert L.pace_set_lmhead_splits(0) == pace.OK  # back to the automatic choice


def test_score_fusion_control_range(pace):
    L = pace.lib()
    assert L.pace_set_score_fused_min_traj(-1) == pace.ERR_INVALID_ARG
    for good in (0, 1, 1 << 18, 1 << 62):
        assert L.pace_set_score_fused_min_traj(good) == pace.OK
    assert L.pace_score_fused_min_traj_default() == 1 << 18
    pace.set_score_fused_min_traj()


def test_shard_selection_argument_checks_return_before_launch(pace):
    """The sharded rejection's calls refuse bad arguments on the host, before any launch."""
    L = pace.lib()
    fake = ctypes.c_void_p(0x1000)
    ws = ctypes.c_void_p(0x100000)  # 256-byte aligned, never dereferenced here
    n = 1 << 20
    assert L.pace_select_shard_workspace_size(100) > 0
    assert L.pace_select_shard_workspace_size(-1) == 0
    # pass out of range, a negative k, a missing histogram, no previous histogram after pass 0
    assert L.pace_select_shard_pass(fake, 100, 6, 3, fake, fake, ws, n, None, None) == \
        pace.ERR_INVALID_ARG
    assert L.pace_select_shard_pass(fake, 100, 0, -1, None, fake, ws, n, None, None) == \
        pace.ERR_INVALID_ARG
    assert L.pace_select_shard_pass(fake, 100, 0, 3, None, None, ws, n, None, None) == \
        pace.ERR_INVALID_ARG
    assert L.pace_select_shard_pass(fake, 100, 2, 3, None, fake, ws, n, None, None) == \
        pace.ERR_INVALID_ARG
    # workspace missing, unaligned or too small
    assert L.pace_select_shard_pass(fake, 100, 0, 3, None, fake, None, n, None, None) == \
        pace.ERR_WORKSPACE
    assert L.pace_select_shard_pass(fake, 100, 0, 3, None, fake, ctypes.c_void_p(0x100008), n,
                                    None, None) == pace.ERR_WORKSPACE
    assert L.pace_select_shard_pass(fake, 100, 0, 3, None, fake, ws, 8, None, None) == \
        pace.ERR_WORKSPACE
    # ties: missing output; write: ids past int32, missing tie count, bad group size
    assert L.pace_select_shard_ties(fake, 100, fake, None, ws, n, None, None) == \
        pace.ERR_INVALID_ARG
    assert L.pace_select_shard_write(fake, 100, 8, 3, fake, (1 << 31) - 100, fake, fake, fake,
                                     None, ws, n, None, None) == pace.ERR_INVALID_ARG
    assert L.pace_select_shard_write(fake, 100, 8, 3, None, 0, fake, fake, fake, None, ws, n,
                                     None, None) == pace.ERR_INVALID_ARG
    assert L.pace_select_shard_write(fake, 100, 0, 3, fake, 0, fake, fake, fake, None, ws, n,
                                     None, None) == pace.ERR_INVALID_ARG
    assert L.pace_loss_from_partial(None, fake, None) == pace.ERR_INVALID_ARG
    assert L.pace_div_selftest(None, None, -1, None, None, None, None, None) == \
        pace.ERR_INVALID_ARG
