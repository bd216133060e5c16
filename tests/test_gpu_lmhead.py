"""Fused LM-head log-probs on the GPU vs the oracle's fp64 log-softmax.

Tolerance |lp_gpu - lp_oracle| <= 5e-3 (absolute) per row, on every row of
small shapes (ragged row blocks, partial vocabulary tiles, compacted and
uncompacted paths), on the tiny workload in full, and on seeded row samples
of the 7B-shaped, multi-turn and MoE-shaped heads at full size."""
import math

import numpy as np
import pytest
import torch

import oracle
from pace_cases import DEV, as_np, bf16_dev, to_dev
from paper_2609_36830_gb300 import pace, workloads

pytestmark = pytest.mark.gpu
TOL = 5e-3


def _bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _run(hidden, w, targets, seq_offsets=None, seq_accepted=None, mask=None, temperature=1.0,
         expect_status=0):
    n_rows = hidden.shape[0]
    if seq_offsets is None:
        seq_offsets = torch.tensor([0, n_rows], dtype=torch.int64, device=DEV)
    b = pace.make_batch(seq_offsets, n_rows, seq_accepted=seq_accepted, mask=mask)
    lse = torch.empty(n_rows, dtype=torch.float32, device=DEV)
    status = pace.new_status(DEV)
    lp = pace.token_logprob(b, hidden, w, targets, temperature, lse=lse, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == expect_status, pace.status_string(int(status.item()))
    return as_np(lp), as_np(lse)


@pytest.mark.parametrize("rows,H,V", [(1, 64, 256), (5, 64, 300), (127, 128, 1000),
                                      (128, 64, 256), (129, 192, 513), (300, 256, 2048),
                                      (1000, 512, 4099), (2048, 1024, 8192),
                                      (300, 8192, 1000), (260, 16384, 700)])
@pytest.mark.parametrize("masked", [False, True])
def test_small_shapes_all_rows(rows, H, V, masked):
    rng = np.random.default_rng(rows * 7 + H + V)
    hb = workloads.bf16_normal_host((rows, H), 1.0, rows + H)
    wb = workloads.bf16_normal_host((V, H), 1.0 / math.sqrt(H) * 2.0, V + H)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    hidden = bf16_dev(hb)
    w = bf16_dev(wb)
    mask = None
    if masked:
        m = (rng.random(rows) < 0.6).astype(np.uint8)
        mask = to_dev(m)
    lp, lse = _run(hidden, w, to_dev(y), mask=mask)
    st, olp, olse = oracle.token_logprob(hb, wb, y)
    assert st == 0
    sel = np.ones(rows, bool) if mask is None else as_np(mask).astype(bool)
    err = np.abs(lp[sel] - olp[sel])
    assert err.max(initial=0) <= TOL, err.max()
    assert np.abs(lse[sel] - olse[sel]).max(initial=0) <= TOL
    assert (lp[~sel] == 0).all() and (lse[~sel] == 0).all()


@pytest.mark.parametrize("rows,H,V,max_run", [(3000, 256, 2048, 300), (2500, 128, 1000, 9),
                                              (100, 64, 700, 40), (7, 64, 256, 3)])
def test_masks_of_runs(rows, H, V, max_run):
    """Rows in the loss as runs of random length (the shape prompt masks and
    rejected groups give): the LM head loads each run of consecutive rows as
    boxes of 2^j rows, or gathers a block of scattered rows, and every row in
    the loss must still match the oracle."""
    rng = np.random.default_rng(rows + max_run)
    m = np.zeros(rows, np.uint8)
    pos = 0
    while pos < rows:
        n = int(rng.integers(1, max_run + 1))
        m[pos:pos + n] = rng.random() < 0.7
        pos += n
    hb = workloads.bf16_normal_host((rows, H), 1.0, rows + 5 * H)
    wb = workloads.bf16_normal_host((V, H), 1.0 / math.sqrt(H) * 2.0, V + 3 * H)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    lp, lse = _run(bf16_dev(hb), bf16_dev(wb), to_dev(y), mask=to_dev(m))
    st, olp, olse = oracle.token_logprob(hb, wb, y)
    assert st == 0
    sel = m.astype(bool)
    assert np.abs(lp[sel] - olp[sel]).max(initial=0) <= TOL
    assert np.abs(lse[sel] - olse[sel]).max(initial=0) <= TOL
    assert (lp[~sel] == 0).all() and (lse[~sel] == 0).all()


def test_vocab_smaller_than_one_tile():
    rng = np.random.default_rng(1)
    rows, H, V = 200, 64, 100
    hb = workloads.bf16_normal_host((rows, H), 1.0, 3)
    wb = workloads.bf16_normal_host((V, H), 0.125, 4)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    lp, _ = _run(bf16_dev(hb), bf16_dev(wb), to_dev(y))
    st, olp, _ = oracle.token_logprob(hb, wb, y)
    assert np.abs(lp - olp).max() <= TOL


def test_temperature():
    rng = np.random.default_rng(2)
    rows, H, V = 333, 128, 3000
    hb = workloads.bf16_normal_host((rows, H), 1.0, 5)
    wb = workloads.bf16_normal_host((V, H), 0.09, 6)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    for tau in (0.7, 1.3):
        lp, _ = _run(bf16_dev(hb), bf16_dev(wb),
                     to_dev(y), temperature=tau)
        st, olp, _ = oracle.token_logprob(hb, wb, y, temperature=float(np.float32(tau)))
        assert np.abs(lp - olp).max() <= TOL


def test_zero_weights_give_uniform():
    rows, H, V = 130, 64, 1000
    hb = workloads.bf16_normal_host((rows, H), 1.0, 7)
    w = torch.zeros(V, H, dtype=torch.bfloat16, device=DEV)
    y = torch.randint(0, V, (rows,), dtype=torch.int32, device=DEV)
    lp, _ = _run(bf16_dev(hb), w, y)
    assert np.abs(lp + math.log(V)).max() <= 1e-5


def test_bad_target_reported():
    rows, H, V = 140, 64, 512
    hb = workloads.bf16_normal_host((rows, H), 1.0, 8)
    wb = workloads.bf16_normal_host((V, H), 0.125, 9)
    y = np.zeros(rows, np.int32)
    y[17] = V
    lp, _ = _run(bf16_dev(hb), bf16_dev(wb), to_dev(y),
                 expect_status=pace.ERR_INVALID_ARG)
    assert math.isnan(lp[17]) and np.isfinite(np.delete(lp, 17)).all()


def _tiny_case():
    pool = workloads.make_pool("tiny")
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hb = workloads.bf16_normal_host((rw.n_rows, H), 1.0, pool.seed + 1)
    wb = workloads.bf16_normal_host((V, H), 1.0 / math.sqrt(H), pool.seed + 2)
    return pool, rw, hb, wb


@pytest.mark.parametrize("agg", [pace.AGG_TOKEN_MEAN, pace.AGG_SEQ_MEAN_TOKEN_MEAN])
def test_tiny_workload_full_with_fused_loss(agg):
    pool, rw, hb, wb = _tiny_case()
    st, olp, _ = oracle.token_logprob(hb, wb, rw.targets)
    assert st == 0
    # behaviour = current + N(0, 0.05 * staleness), current from the oracle
    behav = workloads.behaviour_logprob(rw, pool.trainer_version, olp, pool.seed)
    rng = np.random.default_rng(3)
    acc = (rng.random(pool.n_traj) < 0.75).astype(np.uint8)
    eps_l, eps_h = np.float32(pool.spec.eps_low), np.float32(pool.spec.eps_high)
    params = pace.loss_params(eps_low=eps_l, eps_high=eps_h, agg=agg)
    loss = torch.zeros(1, dtype=torch.float64, device=DEV)
    la = pace.make_loss_args(to_dev(behav), to_dev(pool.reward), pool.group_size, params, loss)
    b = pace.make_batch(to_dev(rw.row_offsets), rw.n_rows, seq_accepted=to_dev(acc),
                        mask=to_dev(rw.mask))
    status = pace.new_status(DEV)
    lp = pace.token_logprob(b, bf16_dev(hb), bf16_dev(wb),
                            to_dev(rw.targets), 1.0, loss=la, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    in_loss = np.repeat(acc, np.diff(rw.row_offsets)).astype(bool) & rw.mask.astype(bool)
    lp = as_np(lp)
    assert np.abs(lp[in_loss] - olp[in_loss]).max() <= TOL
    assert (lp[~in_loss] == 0).all()
    st, oadv = oracle.group_advantages(pool.reward, pool.group_size, seq_accepted=acc,
                                       eps=float(np.float32(1e-6)))
    st, oloss, _, _ = oracle.surrogate(olp, behav, rw.row_offsets, oadv, mask=rw.mask,
                                       seq_accepted=acc, eps_low=float(eps_l),
                                       eps_high=float(eps_h), agg=agg)
    gl = float(loss.item())
    assert abs(gl - oloss) <= 1e-3 * abs(oloss), (gl, oloss)


@pytest.mark.parametrize("name", ["math7b", "multiturn", "moe"])
def test_full_size_heads_sampled_rows(name):
    """Full-size heads in the benchmark's launch configuration (all pool rows,
    accepted flags and loss mask applied by the library's compaction); the
    oracle recomputes a seeded sample of the rows in the loss."""
    pool = workloads.make_pool(name)
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, pool.seed + 11)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), pool.seed + 12)
    rng = np.random.default_rng(pool.seed)
    acc = np.repeat((rng.random(pool.n_traj // 8) < 0.75).astype(np.uint8), 8)
    b = pace.make_batch(to_dev(rw.row_offsets), rw.n_rows, seq_accepted=to_dev(acc),
                        mask=to_dev(rw.mask))
    status = pace.new_status(DEV)
    lp = pace.token_logprob(b, hidden, w, to_dev(rw.targets), 1.0, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    lp = as_np(lp)
    in_loss = np.repeat(acc, np.diff(rw.row_offsets)).astype(bool) & rw.mask.astype(bool)
    assert (lp[~in_loss] == 0).all() and np.isfinite(lp).all()
    cand = np.nonzero(in_loss)[0]
    sample = np.sort(rng.choice(cand, size=48, replace=False))
    sample = np.concatenate([sample, cand[:2], cand[-2:]])  # first and last rows of the loss
    hb = _bits(hidden[torch.from_numpy(sample).to(DEV)])
    wb = _bits(w)
    st, olp, _ = oracle.token_logprob(hb, wb, rw.targets[sample])
    assert st == 0
    err = np.abs(lp[sample] - olp)
    assert err.max() <= TOL, err.max()


@pytest.mark.parametrize("case", ["no_rows", "all_masked", "none_accepted", "one_row"])
def test_degenerate_batches(case):
    H, V = 128, 640
    rng = np.random.default_rng(13)
    rows = {"no_rows": 0, "all_masked": 300, "none_accepted": 300, "one_row": 1}[case]
    hb = workloads.bf16_normal_host((max(rows, 1), H), 1.0, 5)[:rows]
    wb = workloads.bf16_normal_host((V, H), 0.1, 6)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    so = np.array([0, rows // 2, rows], np.int64)
    mask = np.zeros(rows, np.uint8) if case == "all_masked" else np.ones(rows, np.uint8)
    acc = np.zeros(2, np.uint8) if case == "none_accepted" else np.ones(2, np.uint8)
    hidden = bf16_dev(hb) if rows else torch.empty(0, H, dtype=torch.bfloat16, device=DEV)
    b = pace.make_batch(to_dev(so), rows, seq_accepted=to_dev(acc), mask=to_dev(mask))
    loss = torch.full((1,), 5.0, dtype=torch.float64, device=DEV)
    la = pace.make_loss_args(to_dev(np.zeros(max(rows, 1), np.float32)),
                             to_dev(np.ones(2, np.float32)), 2, pace.loss_params(), loss)
    status = pace.new_status(DEV)
    lp = pace.token_logprob(b, hidden, bf16_dev(wb), to_dev(y), 1.0, loss=la, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    lp = as_np(lp)
    if case == "one_row":
        st, olp, _ = oracle.token_logprob(hb, wb, y)
        assert abs(lp[0] - olp[0]) <= TOL
    else:
        assert (lp == 0).all()
        assert float(loss.item()) == 0.0


def test_vocabulary_split_counts_agree():
    """Every split count of the LM head gives the same log-probabilities up to the
    merge's rounding order (40,000 rows: 157 row pairs, so every preferred count
    from 2 up gives each resident cluster at least four items)."""
    H, V, rows = 3584, 152064, 40000
    hidden = workloads.bf16_normal_device((rows, H), 1.0, 31)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), 32)
    y = torch.randint(0, V, (rows,), dtype=torch.int32, device=DEV,
                      generator=torch.Generator(device=DEV).manual_seed(5))
    so = to_dev(np.array([0, rows], np.int64))
    b = pace.make_batch(so, rows)
    out = {}
    try:
        for s in (0, 2, 3, 4, 6, 8):
            pace.set_lmhead_splits(s)
            status = pace.new_status(DEV)
            lp = torch.empty(rows, dtype=torch.float32, device=DEV)
            pace.token_logprob(b, hidden, w, y, 1.0, logprob=lp, status=status)
            torch.cuda.synchronize()
            assert int(status.item()) == 0
            out[s] = lp
    finally:
        pace.set_lmhead_splits(0)
    for s, lp in out.items():
        assert float((lp - out[0]).abs().max()) <= 2e-5, s


@pytest.mark.parametrize("scale", [8.0, 40.0])
def test_large_logits(scale):
    """Logits of tens (sharply peaked softmax): the online log-sum-exp keeps a running
    maximum, so nothing overflows and lp still matches the oracle's two-pass fp64 LSE
    within the same 5e-3."""
    rows, H, V = 300, 256, 2048
    rng = np.random.default_rng(int(scale))
    hb = workloads.bf16_normal_host((rows, H), scale, 9)
    wb = workloads.bf16_normal_host((V, H), 1.0 / math.sqrt(H), 10)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    lp, lse = _run(bf16_dev(hb), bf16_dev(wb), to_dev(y))
    st, olp, olse = oracle.token_logprob(hb, wb, y)
    assert st == 0
    assert np.isfinite(lp).all() and np.isfinite(lse).all()
    assert np.abs(lp - olp).max() <= TOL, np.abs(lp - olp).max()
    assert np.abs(lse - olse).max() <= TOL, np.abs(lse - olse).max()


def test_concurrent_launches_on_two_streams():
    """Two LM-head calls at once on two streams, each sized to fill the GPU: the second
    launch's clusters are not all resident until the first's retire, so its round barrier
    (a bounded wait on the other clusters' progress) times out and proceeds on the resident
    ones.  Both results must equal the same calls run one after the other, with no
    timeout reported."""
    rows, H, V = 100000, 1024, 8192  # ~20 rounds of items per launch
    hb = workloads.bf16_normal_host((rows, H), 1.0, 31)
    wb = workloads.bf16_normal_host((V, H), 2.0 / math.sqrt(H), 32)
    y = np.random.default_rng(33).integers(0, V, size=rows).astype(np.int32)
    hidden, w, tg = bf16_dev(hb), bf16_dev(wb), to_dev(y)
    b = pace.make_batch(torch.tensor([0, rows], dtype=torch.int64, device=DEV), rows)
    ref = [_run(hidden, w, tg)[0] for _ in range(2)]
    outs, statuses = [], []
    streams = [torch.cuda.Stream(device=DEV) for _ in range(2)]
    ws = [pace.workspace(pace.token_logprob_workspace_size(rows, 1, H, V), DEV) for _ in range(2)]
    torch.cuda.synchronize()
    for s, w_s in zip(streams, ws):
        with torch.cuda.stream(s):
            st = pace.new_status(DEV)
            outs.append(pace.token_logprob(b, hidden, w, tg, 1.0, ws=w_s, status=st))
            statuses.append(st)
    torch.cuda.synchronize()
    assert all(int(st.item()) == 0 for st in statuses)
    for lp, r in zip(outs, ref):
        np.testing.assert_array_equal(as_np(lp), r)
