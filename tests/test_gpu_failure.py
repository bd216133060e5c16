"""Failure detection without a GPU fault: a bounded wait on an mbarrier that
nothing completes gives up after its limit and reports PACE_ERR_TIMEOUT through
the device status word; the context stays usable and later work is correct."""
import ctypes
import time

import numpy as np
import pytest
import torch

from pace_cases import DEV, assert_bits_equal, gpu_score, oracle_score
from paper_2609_36830_gb300 import pace, workloads

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives():
    status = pace.new_status(DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    t0 = time.perf_counter()
    st = pace.lib().pace_wait_timeout_selftest(20_000_000, ctypes.c_void_p(status.data_ptr()),
                                               stream)  # 20 ms
    assert st == pace.OK
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert int(status.item()) == pace.ERR_TIMEOUT
    assert elapsed < 5.0
    # the context is still healthy: a full scoring call afterwards is bit-exact
    pool = workloads.make_pool("tiny")
    args = (pool.tags, pool.meta["offsets_host"], pool.c_version, pool.s_pre,
            pool.trainer_version, pool.window)
    g = gpu_score(*args)
    o = oracle_score(*args)
    assert_bits_equal(g["score"], o["score"], "after timeout")


def test_selftest_rejects_bad_arguments():
    L = pace.lib()
    assert L.pace_wait_timeout_selftest(1000, None, None) == pace.ERR_INVALID_ARG
    fake = ctypes.c_void_p(0x1000)
    assert L.pace_wait_timeout_selftest(0, fake, None) == pace.ERR_INVALID_ARG
    assert L.pace_wait_timeout_selftest(3_000_000_000, fake, None) == pace.ERR_INVALID_ARG
