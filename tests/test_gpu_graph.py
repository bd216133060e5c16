"""Every call of the path is stream-ordered with no host synchronisation, so it can
be captured in a CUDA graph: replaying the graph must reproduce the eager results
bit for bit (pool scoring + selection on both selection paths, and a whole step)."""
import math

import numpy as np
import pytest
import torch

from pace_cases import DEV
from paper_2609_36830_gb300 import pace, step, workloads

pytestmark = pytest.mark.gpu


def _capture(fn):
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        fn()  # warm-up outside the capture (one-time attribute set-up)
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g


@pytest.fixture(params=["own_launch", "in_reduction"])
def finalisation(request):
    """Both finalisation paths of pace_score_pool, the second a cooperative launch."""
    pace.set_score_fused_min_traj(1 << 62 if request.param == "own_launch" else 0)
    yield request.param
    pace.set_score_fused_min_traj()


@pytest.mark.parametrize("n_traj", [1024, 16384])  # 128 units: one-block rank; 2048: radix
def test_scoring_and_selection_replay(n_traj, finalisation):
    pool = workloads.make_pool("sweep", n_traj=n_traj, device=DEV)
    n = pool.n_traj
    c = torch.from_numpy(pool.c_version).to(DEV)
    sp = torch.from_numpy(pool.s_pre).to(DEV)
    win = torch.from_numpy(pool.window).to(DEV)
    params = pace.score_params(group_size=8)
    out = {k: torch.empty(n, dtype=torch.float64, device=DEV)
           for k in ("kgen", "kwait", "weight", "score")}
    out["unit_score"] = torch.empty(n // 8, dtype=torch.float64, device=DEV)
    L = pace.lib()
    ws = pace.workspace(L.pace_score_pool_workspace_size(n, win.numel()), DEV)
    sel = {"accepted": torch.empty(n, dtype=torch.int32, device=DEV),
           "rejected": torch.empty(n, dtype=torch.int32, device=DEV),
           "flags": torch.empty(n, dtype=torch.uint8, device=DEV)}
    ws_sel = pace.workspace(L.pace_select_workspace_size(n // 8), DEV)
    status = pace.new_status(DEV)
    bp = pace.budget_params(pool.n_target)

    def one():
        pace.score_pool(pool.tags, pool.offsets, c, sp, pool.trainer_version, win, params,
                        out=out, ws=ws, status=status)
        pace.select(out["unit_score"], 8, bp, out=sel, ws=ws_sel, status=status)

    one()
    _, k_units, _, _, _ = pace.select(out["unit_score"], 8, bp, out=sel, ws=ws_sel,
                                      status=status)
    torch.cuda.synchronize()
    # the id lists fill only their first (U - k) G and k G entries
    used = {"accepted": (n // 8 - k_units) * 8, "rejected": k_units * 8}
    ref = {k: v[:used.get(k, v.numel())].clone()
           for k, v in list(out.items()) + list(sel.items())}
    g = _capture(one)
    for buf in list(out.values()) + list(sel.values()):
        buf.fill_(0)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    for k, v in list(out.items()) + list(sel.items()):
        assert torch.equal(v[:used.get(k, v.numel())], ref[k]), k


def test_tiny_step_replay():
    pool = workloads.make_pool("tiny")
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, pool.seed + 11)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), pool.seed + 12)
    behav = workloads.behaviour_logprob(rw, pool.trainer_version, workloads.uniform_center(V),
                                        pool.seed)
    x = step.build_inputs(pool, rw, hidden, w, behav)
    st = step.PaceStep(x, loss_params=pace.loss_params(eps_low=0.2, eps_high=0.2))
    st.run()
    torch.cuda.synchronize()
    lp_ref, loss_ref = st.logprob.clone(), st.loss.clone()
    flags_ref = st.sel_out["flags"].clone()
    g = st.capture()
    st.logprob.fill_(0)
    st.loss.fill_(0)
    st.sel_out["flags"].fill_(0)
    g.replay()
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    assert torch.equal(st.sel_out["flags"], flags_ref)
    assert torch.equal(st.logprob, lp_ref)
    assert float(st.loss.item()) == float(loss_ref.item())
    assert np.isfinite(float(st.loss.item()))


def test_capture_refuses_a_moving_budget():
    pool = workloads.make_pool("tiny")
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, 1)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), 2)
    behav = workloads.behaviour_logprob(rw, pool.trainer_version, workloads.uniform_center(V), 3)
    st = step.PaceStep(step.build_inputs(pool, rw, hidden, w, behav), beta=0.5)
    with pytest.raises(ValueError):
        st.capture()
