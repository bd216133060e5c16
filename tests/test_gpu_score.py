"""Pool scoring on the GPU vs the oracle: fp64 bits must be identical
(K_gen, K_wait, F, score, unit score) on every workload, mode and edge case."""
import ctypes
import json
import os

import numpy as np
import pytest
import torch

from pace_cases import (DEV, as_np, assert_bits_equal, gpu_score, oracle_score,
                        pool_score_case, to_dev)
from paper_2609_36830_gb300 import pace, workloads

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_pool.json")


@pytest.fixture(autouse=True, params=["own_launch", "in_reduction"])
def finalisation(request):
    """Every test of this file runs on both finalisation paths: a launch of its
    own (the default below 2^18 trajectories) and inside the tag reduction's
    cooperative launch (the default from 2^18), whatever the pool's size."""
    pace.set_score_fused_min_traj(1 << 62 if request.param == "own_launch" else 0)
    yield request.param
    pace.set_score_fused_min_traj()


def _check(g, o, what):
    for k in ("kgen", "kwait", "weight", "score", "unit_score"):
        assert_bits_equal(g[k], o[k], f"{what}:{k}")


@pytest.mark.parametrize("mode", ["eff", "raw", "gen"])
def test_hand_pool(mode):
    h = json.load(open(GOLDEN))
    tr = h["trajectories"]
    tags = np.concatenate([np.array(t["tags"], np.int32) for t in tr])
    offsets = np.concatenate([[0], np.cumsum([len(t["tags"]) for t in tr])]).astype(np.int64)
    c = np.array([t["c"] for t in tr], np.int32)
    s_pre = np.array([np.nan if t["s_pre"] is None else t["s_pre"] for t in tr], np.float32)
    window = np.array(h["window"], np.float32)
    for G in (1, 2, 3, 6):
        g = gpu_score(tags, offsets, c, s_pre, 10, window, mode=mode, min_obs=1, group_size=G)
        o = oracle_score(tags, offsets, c, s_pre, 10, window, mode=mode, min_obs=1, group_size=G)
        _check(g, o, f"hand G={G}")


@pytest.mark.parametrize("name,n", [("tiny", None), ("math7b", 384), ("math7b", 512),
                                    ("math7b", 768), ("multiturn", 256), ("multiturn", 480),
                                    ("moe", None), ("sweep", 1024), ("sweep", 16384)])
@pytest.mark.parametrize("mode", ["eff", "raw", "gen"])
def test_workloads(name, n, mode):
    pool = workloads.make_pool(name, n_traj=n)
    g, o = pool_score_case(pool, mode=mode)
    _check(g, o, f"{name}/{n}/{mode}")


def test_group_sizes_and_gammas():
    pool = workloads.make_pool("math7b", n_traj=768)
    for G in (1, 12, 16, 96, 256, 768):
        for gamma in (1, 2, 4, 7):
            args = (pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
                    pool.trainer_version, pool.window)
            g = gpu_score(*args, group_size=G, gamma=gamma)
            o = oracle_score(*args, group_size=G, gamma=gamma)
            _check(g, o, f"G={G} gamma={gamma}")
    # the largest group the library takes (one group per 1024-thread block)
    pool = workloads.make_pool("moe")
    args = (pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
            pool.trainer_version, pool.window)
    _check(gpu_score(*args, group_size=1024), oracle_score(*args, group_size=1024), "G=1024")


def test_sweep_128k_full_and_1m_sampled():
    # 128k pool (~0.44 G tags) checked in full
    pool = workloads.make_pool("sweep", n_traj=131072, device=DEV)
    tags_h = pool.tags.cpu().numpy()
    args = (pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
            pool.trainer_version, pool.window)
    g = gpu_score(*args, group_size=8)
    o = oracle_score(tags_h, *args[1:], group_size=8)
    _check(g, o, "sweep128k")
    del pool, tags_h
    torch.cuda.empty_cache()
    # 1M pool (~3.4 G tags): the launch the benchmark times; the oracle scores a
    # seeded sample of whole groups from their own tags.
    pool = workloads.make_pool("sweep", n_traj=1048576, device=DEV)
    off = pool.meta["offsets_host"]
    g = gpu_score(pool.tags, off, pool.c_version, pool.s_pre, pool.trainer_version, pool.window,
                  group_size=8)
    rng = np.random.default_rng(5)
    units = np.sort(rng.choice(1048576 // 8, size=256, replace=False))
    ids = (units[:, None] * 8 + np.arange(8)[None, :]).ravel()
    seg = [pool.tags[off[i]:off[i + 1]].cpu().numpy() for i in ids]
    sub_off = np.concatenate([[0], np.cumsum([s.size for s in seg])]).astype(np.int64)
    o = oracle_score(np.concatenate(seg), sub_off, pool.c_version[ids], pool.s_pre[ids],
                     pool.trainer_version, pool.window, group_size=8)
    for k in ("kgen", "kwait", "weight", "score"):
        assert_bits_equal(g[k][ids], o[k], f"sweep1m:{k}")
    assert_bits_equal(g["unit_score"][units], o["unit_score"], "sweep1m:unit")
    # identities over the whole pool: score = K_wait + F K_gen, all finite, >= 0
    assert np.isfinite(g["score"]).all() and (g["score"] >= 0).all()
    np.testing.assert_array_equal(g["score"], g["kwait"] + g["weight"] * g["kgen"])


def _mk_fast(lens, rng, j=50):
    """_mk without tool tags, vectorised for large pools: tags of trajectory i
    uniform in [0, c_i], sorted within the trajectory."""
    lens = np.asarray(lens, np.int64)
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    n = lens.size
    c = rng.integers(0, j + 1, size=n).astype(np.int32)
    owner = np.repeat(np.arange(n), lens)
    tags = np.floor(rng.random(owner.size) * (c[owner].astype(np.float64) + 1)).astype(np.int32)
    tags = tags[np.lexsort((tags, owner))]
    s_pre = np.where(rng.random(n) < 0.5, rng.random(n), np.nan).astype(np.float32)
    window = rng.random(100).astype(np.float32)
    return tags, offsets, c, s_pre, j, window


def _mk(lens, rng, j=50, tool=0.0):
    offsets = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    n = len(lens)
    c = rng.integers(0, j + 1, size=n).astype(np.int32)
    tags = np.empty(int(offsets[-1]), np.int32)
    for i in range(n):
        t = np.sort(rng.integers(0, c[i] + 1, size=lens[i])).astype(np.int32)
        t[rng.random(lens[i]) < tool] = -1
        tags[offsets[i]:offsets[i + 1]] = t
    s_pre = np.where(rng.random(n) < 0.5, rng.random(n), np.nan).astype(np.float32)
    window = rng.random(100).astype(np.float32)
    return tags, offsets, c, s_pre, j, window


@pytest.mark.parametrize("case", ["empty_traj", "ragged", "one_long", "tiny_many", "all_tool",
                                  "single", "huge_versions", "mixed_versions", "warp_aligned"])
def test_edge_cases(case):
    """Pool shapes and tag ranges that take every path of the tag reduction: empty
    trajectories, boundaries at and off batch edges, tool tags, and versions at and
    above 2^26 (no 32-bit partial sums), alone and mixed with small ones."""
    rng = np.random.default_rng(sum(map(ord, case)))
    if case == "empty_traj":
        lens = [0, 5, 0, 0, 130, 0, 1, 0]
    elif case == "ragged":
        lens = list(rng.integers(1, 3000, size=64))
        lens[-1] = 1027
    elif case == "one_long":
        lens = [3, 5_000_003, 17, 0, 1, 2, 9, 100]
    elif case == "tiny_many":
        lens = list(rng.integers(0, 4, size=40000))
    elif case == "all_tool":
        lens = [10, 20, 30, 40]
    elif case in ("huge_versions", "mixed_versions"):
        lens = list(rng.integers(1, 5000, size=64))
    elif case == "warp_aligned":
        # trajectories of whole 512-tag batches, so every trajectory boundary is a
        # batch edge, where warp ranges begin and end too (many coincide), with
        # empty trajectories on the boundaries: each case of which warp writes a
        # trajectory's slot and which warp's head slot continues it
        lens = []
        for i in range(48):
            lens += [2048 * (1 + i % 3)] + [0] * (i % 2) + [512 * (1 + i % 5)] + [0] * (i % 3)
    else:
        lens = [1]
    lens = list(lens)
    while len(lens) % 4:
        lens.append(int(rng.integers(0, 9)))
    tool = 1.0 if case == "all_tool" else 0.2
    j = 2_000_000_000 if case in ("huge_versions", "mixed_versions") else 50
    tags, offsets, c, s_pre, j, window = _mk(lens, rng, j=j, tool=tool)
    if case == "huge_versions":  # every policy tag at or above 2^26
        pol = tags >= 0
        c = np.maximum(c, (1 << 26) + 1000).astype(np.int32)
        tags[pol] = np.minimum(tags[pol] + (1 << 26), np.repeat(c, lens)[pol]).astype(np.int32)
    elif case == "mixed_versions":  # alternate trajectories small (< 2^26) and large
        small = np.repeat(np.arange(len(lens)) % 2 == 0, lens)
        tags[small & (tags >= 0)] %= 1 << 20
        c = np.where(np.arange(len(lens)) % 2 == 0, np.minimum(c, 1 << 20), c).astype(np.int32)
    for G in (1, 4):
        g = gpu_score(tags, offsets, c, s_pre, j, window, group_size=G, min_obs=10)
        o = oracle_score(tags, offsets, c, s_pre, j, window, group_size=G, min_obs=10)
        _check(g, o, f"{case}/G={G}")


def test_window_below_min_obs_and_no_window():
    pool = workloads.make_pool("tiny")
    args = (pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
            pool.trainer_version)
    g = gpu_score(*args, pool.window[:20], min_obs=32)
    o = oracle_score(*args, pool.window[:20], min_obs=32)
    _check(g, o, "short window")
    assert (g["weight"] == 1.0).all()
    g = gpu_score(*args, None, min_obs=0)
    o = oracle_score(*args, np.zeros(0, np.float32), min_obs=0)
    _check(g, o, "no window")


@pytest.mark.parametrize("n_traj", [256, 32768])  # direct count / sorted window + F table
@pytest.mark.parametrize("wlen", [1, 7, 32, 512, 513, 1000, 4096])
@pytest.mark.parametrize("gamma", [1, 2, 4, 7])
def test_window_shapes_and_ties(n_traj, wlen, gamma):
    """The ECDF count of Eq. 9 against windows of every size up to the 4096
    maximum, heavy ties, +0 and -0, +inf, and s exactly on window values; F of
    Eq. 10 for several gamma; on a small pool (counted directly) and a large one
    (sorted window and a table of F).  Bits must match the oracle."""
    rng = np.random.default_rng(wlen * 10 + gamma)
    window = (np.round(rng.random(wlen) * 8) / 8).astype(np.float32)  # ties
    window[rng.random(wlen) < 0.05] = -0.0
    window[rng.random(wlen) < 0.02] = np.inf
    lens = rng.integers(1, 40, size=n_traj)
    tags, offsets, c, s_pre, j, _ = _mk_fast(lens, rng)
    pick = rng.random(len(lens))
    s_pre = np.where(pick < 0.4, rng.choice(window, size=len(lens)),  # exactly on window values
                     np.where(pick < 0.5, np.float32(0.0),
                              np.where(pick < 0.55, np.float32(np.inf),
                                       np.where(pick < 0.6, np.nan,
                                                rng.random(len(lens)) * 1.2 - 0.1)))).astype(
        np.float32)
    for mode in ("eff", "gen"):
        g = gpu_score(tags, offsets, c, s_pre, j, window, mode=mode, gamma=gamma, min_obs=1,
                      group_size=4)
        o = oracle_score(tags, offsets, c, s_pre, j, window, mode=mode, gamma=gamma, min_obs=1,
                         group_size=4)
        _check(g, o, f"w{wlen}/g{gamma}/{mode}")


@pytest.mark.parametrize("n_traj,n_tok,wlen", [(64, 0, 512), (8192, 0, 4096), (8192, 1500, 4096),
                                                (16384, 70000, 512)])
def test_short_streams(n_traj, n_tok, wlen):
    """Pools whose tag stream is empty or a block or two long: the finalisation
    runs in the tag reduction's launch, so its one or few stream blocks score every
    group; on the table path (8,192 trajectories and more) those few blocks also run
    every window-preparation task (the sort and up to 129 slices of the F table)."""
    rng = np.random.default_rng(n_traj + n_tok + wlen)
    lens = np.zeros(n_traj, np.int64)
    if n_tok:
        lens[:] = np.bincount(rng.integers(0, n_traj, size=n_tok), minlength=n_traj)
    tags, offsets, c, s_pre, j, _ = _mk_fast(lens, rng)
    window = rng.random(wlen).astype(np.float32)
    for G in (1, 8, min(256, n_traj)):
        g = gpu_score(tags, offsets, c, s_pre, j, window, group_size=G, min_obs=1)
        o = oracle_score(tags, offsets, c, s_pre, j, window, group_size=G, min_obs=1)
        _check(g, o, f"{n_traj}/{n_tok}/G={G}")


def test_empty_pool():
    out = gpu_score(np.zeros(0, np.int32), np.zeros(1, np.int64), np.zeros(0, np.int32),
                    np.zeros(0, np.float32), 5, np.ones(4, np.float32), group_size=1)
    assert out["score"].size == 0


@pytest.mark.parametrize("what,code", [("v_gt_c", pace.ERR_VERSION_ORDER),
                                       ("c_gt_j", pace.ERR_VERSION_ORDER),
                                       ("tag_below_sentinel", pace.ERR_INVALID_ARG),
                                       ("nan_window", pace.ERR_NAN_INPUT),
                                       ("bad_offsets", pace.ERR_INVALID_ARG)])
def test_device_side_errors(what, code):
    pool = workloads.make_pool("tiny")
    tags = pool.tags.copy()
    off = pool.meta["offsets_host"].copy()
    c = pool.c_version.copy()
    w = pool.window.copy()
    j = pool.trainer_version
    if what == "v_gt_c":
        tags[off[3] + 1] = c[3] + 1
    elif what == "c_gt_j":
        c[5] = j + 1
    elif what == "tag_below_sentinel":
        tags[7] = -3
    elif what == "nan_window":
        w[100] = np.nan
    else:
        off[10] = off[11] + 1  # not non-decreasing
    gpu_score(tags, off, c, pool.s_pre, j, w, expect_status=code)


def _div_selftest(S, T):
    L = pace.lib()
    n = S.size
    dS, dT = to_dev(S.astype(np.int64)), to_dev(T.astype(np.uint32).view(np.int32))
    outs = [torch.empty(n, dtype=torch.float64, device=DEV) for _ in range(4)]
    st = L.pace_div_selftest(ctypes.c_void_p(dS.data_ptr()), ctypes.c_void_p(dT.data_ptr()), n,
                             *[ctypes.c_void_p(o.data_ptr()) for o in outs], None)
    assert st == pace.OK
    torch.cuda.synchronize()
    return [as_np(o) for o in outs]


def test_integer_quotient_matches_the_fp64_pipe_bit_for_bit():
    """K_gen = S / T and K_wait = (double)x are built on the integer pipe (GB300's
    fp64 pipe bounds the finalisation).  They must equal __ddiv_rn(__ll2double_rn(S), T)
    and __ll2double_rn(x) bit for bit - and numpy's float64(S) / float64(T) on the
    host, the oracle's arithmetic - over all magnitudes and the rounding edge cases."""
    rng = np.random.default_rng(99)
    n = 1 << 20
    bits_s = rng.integers(0, 64, size=n)
    S = (rng.integers(0, 1 << 62, size=n, dtype=np.int64) >> (62 - np.minimum(bits_s, 62)))
    S = np.where(bits_s == 63, rng.integers(-(1 << 62), 1 << 62, size=n, dtype=np.int64) * 2 + 1,
                 S)
    S = np.where(rng.random(n) < 0.5, -S, S)
    bits_t = rng.integers(0, 33, size=n)
    T = (rng.integers(1, 1 << 32, size=n, dtype=np.int64) >> (32 - bits_t)).clip(1, (1 << 32) - 1)
    edge_s = [0, 1, -1, 7, (1 << 53) - 1, 1 << 53, (1 << 53) + 1, (1 << 53) + 3, (1 << 54) + 2,
              (1 << 54) + 6, -(1 << 53) - 1, (1 << 62) + (1 << 9), (1 << 63) - 1, -(1 << 63),
              -((1 << 63) - 1), 3 * 5 * 7 * 11 * 13 * (1 << 20), 123456789012345]
    edge_t = [1, 2, 3, 7, (1 << 31), (1 << 32) - 1, 65535, 3 * 5 * 7]
    es, et = np.meshgrid(np.array(edge_s, dtype=np.int64), np.array(edge_t, dtype=np.int64))
    S = np.concatenate([S, es.ravel(), np.arange(-5000, 5000, dtype=np.int64) * 37])
    T = np.concatenate([T, et.ravel(), np.full(10000, 37, np.int64)])
    q_int, q_fp64, c_int, c_fp64 = _div_selftest(S, T)
    np.testing.assert_array_equal(q_int.view(np.uint64), q_fp64.view(np.uint64))
    np.testing.assert_array_equal(c_int.view(np.uint64), c_fp64.view(np.uint64))
    host = S.astype(np.float64) / T.astype(np.float64)
    np.testing.assert_array_equal(q_int.view(np.uint64), host.view(np.uint64))
    np.testing.assert_array_equal(c_int.view(np.uint64), S.astype(np.float64).view(np.uint64))
