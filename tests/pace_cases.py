"""Shared helpers of the GPU parity tests: upload pools, run the library
through the binding, run the oracle on the same inputs."""
import numpy as np
import torch

import oracle
from paper_2609_36830_gb300 import pace, workloads

DEV = "cuda"
MODES = {"eff": pace.SCORE_EFF, "raw": pace.SCORE_RAW, "gen": pace.SCORE_GEN}


def to_dev(a, dtype=None):
    if isinstance(a, torch.Tensor):
        return a.to(DEV)
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.to(dtype)
    return t.to(DEV)


def bf16_dev(bits):
    """uint16 bf16 bit patterns (numpy) -> a bf16 CUDA tensor holding the same bits."""
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(DEV).view(torch.bfloat16)


def as_np(t):
    return t.detach().cpu().numpy() if isinstance(t, torch.Tensor) else np.asarray(t)


def gpu_score(tags, offsets, c, s_pre, j, window, mode="eff", gamma=4, min_obs=32,
              f_missing=1.0, group_size=8, expect_status=0):
    status = pace.new_status(DEV)
    out = pace.score_pool(to_dev(tags), to_dev(offsets), to_dev(c), to_dev(s_pre), j,
                          to_dev(window) if window is not None and len(window) else None,
                          pace.score_params(MODES[mode], gamma, min_obs, group_size, f_missing),
                          status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == expect_status, pace.status_string(int(status.item()))
    return {k: as_np(v) for k, v in out.items()}


def oracle_score(tags, offsets, c, s_pre, j, window, mode="eff", gamma=4, min_obs=32,
                 f_missing=1.0, group_size=8):
    st, kg, kw, w, sc, us = oracle.score_pool(as_np(tags), as_np(offsets), c, s_pre, j,
                                              window if window is not None else np.zeros(0,
                                                                                        np.float32),
                                              mode=MODES[mode], gamma=gamma, min_obs=min_obs,
                                              f_missing=f_missing, group_size=group_size)
    assert st == 0
    return {"kgen": kg, "kwait": kw, "weight": w, "score": sc, "unit_score": us}


def assert_bits_equal(a, b, what):
    a = np.ascontiguousarray(a, np.float64)
    b = np.ascontiguousarray(b, np.float64)
    assert a.shape == b.shape, what
    diff = np.nonzero(a.view(np.uint64) != b.view(np.uint64))[0]
    assert diff.size == 0, f"{what}: {diff.size} mismatches, first {diff[:5]}: " \
                           f"{a[diff[:5]]} vs {b[diff[:5]]}"


def pool_score_case(pool, mode="eff", **kw):
    args = (pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
            pool.trainer_version, pool.window)
    g = gpu_score(*args, mode=mode, group_size=pool.group_size, **kw)
    o = oracle_score(*args, mode=mode, group_size=pool.group_size, **kw)
    return g, o
