"""pace_select_k_noalloc: the selection entry point for callers that cannot
allocate device memory (for example a plugin inside a framework whose memory
pool owns all device memory).  Its scratch is a fixed 128 KB array inside the
library, so it must give exactly the ids of pace_select_k, which uses a
caller-provided workspace, and of the CPU oracle's top-k, and keep doing so on
back-to-back calls that reuse the shared array.  This file is collected last on
purpose."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2609_36830_gb300 import pace

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _outputs(n):
    return (torch.full((n,), -7, dtype=torch.int32, device=DEV),
            torch.full((n,), -7, dtype=torch.int32, device=DEV),
            torch.full((n,), 9, dtype=torch.uint8, device=DEV))


def _call_noalloc(scores, G, k):
    L = pace.lib()
    n = scores.numel() * G
    acc, rej, flags = _outputs(n)
    status = pace.new_status(DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = L.pace_select_k_noalloc(ctypes.c_void_p(scores.data_ptr()), scores.numel(), G, k,
                                 ctypes.c_void_p(acc.data_ptr()), ctypes.c_void_p(rej.data_ptr()),
                                 ctypes.c_void_p(flags.data_ptr()),
                                 ctypes.c_void_p(status.data_ptr()), stream)
    assert st == pace.OK, pace.status_string(st)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return acc.cpu().numpy(), rej.cpu().numpy(), flags.cpu().numpy()


def _call_workspace(scores, G, k):
    L = pace.lib()
    n = scores.numel() * G
    acc, rej, flags = _outputs(n)
    ws = pace.workspace(L.pace_select_workspace_size(scores.numel()), DEV)
    status = pace.new_status(DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = L.pace_select_k(ctypes.c_void_p(scores.data_ptr()), scores.numel(), G, k,
                         ctypes.c_void_p(acc.data_ptr()), ctypes.c_void_p(rej.data_ptr()),
                         ctypes.c_void_p(flags.data_ptr()), ctypes.c_void_p(ws.data_ptr()),
                         ws.numel(), ctypes.c_void_p(status.data_ptr()), stream)
    assert st == pace.OK, pace.status_string(st)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return acc.cpu().numpy(), rej.cpu().numpy(), flags.cpu().numpy()


@pytest.mark.parametrize("U,G", [(100, 8), (5000, 1), (131072, 8), (1 << 20, 1)])
def test_noalloc_matches_workspace_entry_point_twice(U, G):
    rng = np.random.default_rng(U)
    for call in range(2):  # the second call reuses the shared scratch array
        s = torch.from_numpy(rng.integers(0, 50, size=U).astype(np.float64) / 8.0).to(DEV)
        k = int(rng.integers(1, U))
        a = _call_noalloc(s, G, k)
        b = _call_workspace(s, G, k)
        for x, y in zip(a, b):
            np.testing.assert_array_equal(x, y)
        # and the oracle's (score desc, id asc) top-k on the same scores
        st, acc, rej, flag = oracle.select(s.cpu().numpy(), G, k)
        assert st == 0
        np.testing.assert_array_equal(a[0][: acc.size], acc)
        np.testing.assert_array_equal(a[1][: rej.size], rej)
        np.testing.assert_array_equal(a[2], flag)
        assert a[1][: k * G].size == k * G and (a[1][: k * G] >= 0).all()


def test_noalloc_rejects_pools_above_the_limit():
    L = pace.lib()
    st = L.pace_select_k_noalloc(ctypes.c_void_p(0x1000), (1 << 20) + 1, 1, 1,
                                 ctypes.c_void_p(0x1000), None, None, None, None)
    assert st == pace.ERR_UNSUPPORTED_SHAPE
