"""Backward of the surrogate and of the fused LM head on the GPU vs the oracle.

The surrogate derivative is compared row by row (fp32 vs fp64, relative 1e-5)
away from the clip kinks, where fp32 and fp64 may legitimately pick different
branches.  The LM-head gradients hold G = (g/tau)(onehot - softmax) in bf16
(8 significant bits, round to nearest even: a relative rounding of at most
2^-8 per element), and everything else is fp32.  So each element is compared
with the fp64 oracle against the bound that rounding allows:
    |dH_rk - dH*_rk| <= (2^-8 + 2^-10) * sum_v |G_rv| |W_vk|
    |dW_vk - dW*_vk| <= (2^-8 + 2^-10) * sum_r |G_rv| |h_rk|
(the sums from the oracle in fp64; 2^-10 covers the fp32 softmax, the fp32
accumulation and the forward's log-sum-exp).  A wrong tile, a mis-scattered row
or a sign error on a few columns fails it where a whole-matrix norm would not.
The Frobenius relative error (1e-2) stays as a summary check."""
import math

import numpy as np
import pytest
import torch

import oracle
from pace_cases import DEV, as_np, bf16_dev, to_dev
from paper_2609_36830_gb300 import pace, workloads

pytestmark = pytest.mark.gpu
REL = 1e-2
ELEM = 2.0 ** -8 + 2.0 ** -10


def _rel(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


def _check_elementwise(got, ref, mag, what):
    """|got - ref| <= ELEM * mag element by element (exact where mag is 0)."""
    err = np.abs(got.astype(np.float64) - ref)
    bad = err > ELEM * mag
    assert not bad.any(), (what, int(bad.sum()), np.argwhere(bad)[:5].tolist(),
                           float((err / np.maximum(mag, 1e-300)).max()))


@pytest.mark.parametrize("rows_spec", [("tiny", None), ("math7b", 512), ("multiturn", 480)])
@pytest.mark.parametrize("agg", [pace.AGG_TOKEN_MEAN, pace.AGG_SEQ_MEAN_TOKEN_MEAN])
def test_surrogate_backward_matches_oracle(rows_spec, agg):
    pool = workloads.make_pool(*rows_spec)
    rw = workloads.make_rows(pool)
    rng = np.random.default_rng(11)
    V = pool.spec.vocab
    lp = (workloads.uniform_center(V) + rng.standard_normal(rw.n_rows)).astype(np.float32)
    behav = workloads.behaviour_logprob(rw, pool.trainer_version, workloads.uniform_center(V), 5)
    acc = np.repeat((rng.random(pool.n_traj // 8) < 0.75).astype(np.uint8), 8)
    params = pace.loss_params(eps_low=pool.spec.eps_low, eps_high=pool.spec.eps_high, agg=agg)
    la = pace.make_loss_args(to_dev(behav), to_dev(pool.reward), 8, params,
                             torch.zeros(1, dtype=torch.float64, device=DEV))
    b = pace.make_batch(to_dev(rw.row_offsets), rw.n_rows, seq_accepted=to_dev(acc),
                        mask=to_dev(rw.mask))
    status = pace.new_status(DEV)
    g = pace.surrogate_backward(b, to_dev(lp), la, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    _, oadv = oracle.group_advantages(pool.reward, 8, seq_accepted=acc,
                                      eps=float(np.float32(1e-6)))
    eps_l, eps_h = float(np.float32(pool.spec.eps_low)), float(np.float32(pool.spec.eps_high))
    st, og = oracle.surrogate_grad(lp, behav, rw.row_offsets, oadv, mask=rw.mask,
                                   seq_accepted=acc, eps_low=eps_l, eps_high=eps_h, agg=agg)
    assert st == 0
    rho = np.exp(np.clip(lp.astype(np.float64) - behav, -20, 20))
    a_row = np.repeat(oadv, np.diff(rw.row_offsets))
    near = (np.abs(rho - (1 - eps_l)) < 1e-5) | (np.abs(rho - (1 + eps_h)) < 1e-5) | \
        (np.abs(rho - 10.0) < 1e-4)
    gg = as_np(g).astype(np.float64)
    ok = ~near
    assert np.abs(gg[ok] - og[ok]).max() <= 1e-5 * np.abs(og).max()
    assert (gg[og == 0] == 0).sum() >= (og == 0).sum() - near.sum()


@pytest.mark.parametrize("rows,H,V,masked", [(100, 64, 256, False), (300, 128, 1000, True),
                                             (1000, 256, 2048, False), (700, 192, 4099, True),
                                             (3000, 512, 2304, True), (600, 2048, 1000, True),
                                             (300, 4096, 520, False)])
def test_lmhead_backward_matches_oracle(rows, H, V, masked):
    rng = np.random.default_rng(rows + H + V)
    hb = workloads.bf16_normal_host((rows, H), 1.0, rows)
    wb = workloads.bf16_normal_host((V, H), 1.0 / math.sqrt(H) * 2, V)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    mask = (rng.random(rows) < 0.7).astype(np.uint8) if masked else np.ones(rows, np.uint8)
    g = (rng.standard_normal(rows) * mask).astype(np.float32)
    so = to_dev(np.array([0, rows], np.int64))
    b = pace.make_batch(so, rows, mask=to_dev(mask) if masked else None)
    hidden, w = bf16_dev(hb), bf16_dev(wb)
    lse = torch.empty(rows, dtype=torch.float32, device=DEV)
    status = pace.new_status(DEV)
    pace.token_logprob(b, hidden, w, to_dev(y), 1.0, lse=lse, status=status)
    dh, dw = pace.token_logprob_backward(b, hidden, w, to_dev(y), lse, to_dev(g), status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    st, odh, odw = oracle.lmhead_backward(hb, wb, y, g.astype(np.float64))
    assert st == 0
    st, mh, mw = oracle.lmhead_backward(hb, wb, y, g.astype(np.float64), magnitude=True)
    assert st == 0
    _check_elementwise(as_np(dh), odh, mh, "dH")
    _check_elementwise(as_np(dw), odw, mw, "dW")
    assert _rel(as_np(dh), odh) <= REL, _rel(as_np(dh), odh)
    assert _rel(as_np(dw), odw) <= REL, _rel(as_np(dw), odw)
    assert (as_np(dh)[mask == 0] == 0).all()


def test_full_size_backward_sampled_rows_and_identity():
    pool = workloads.make_pool("math7b")
    rw = workloads.make_rows(pool)
    H, V = pool.spec.hidden, pool.spec.vocab
    hidden = workloads.bf16_normal_device((rw.n_rows, H), 1.0, pool.seed + 11)
    w = workloads.bf16_normal_device((V, H), 1.0 / math.sqrt(H), pool.seed + 12)
    rng = np.random.default_rng(4)
    acc = np.repeat((rng.random(pool.n_traj // 8) < 0.75).astype(np.uint8), 8)
    in_loss = np.repeat(acc, np.diff(rw.row_offsets)).astype(bool) & rw.mask.astype(bool)
    g = (rng.standard_normal(rw.n_rows) * 1e-6 * in_loss).astype(np.float32)
    b = pace.make_batch(to_dev(rw.row_offsets), rw.n_rows, seq_accepted=to_dev(acc),
                        mask=to_dev(rw.mask))
    targets = to_dev(rw.targets)
    lse = torch.empty(rw.n_rows, dtype=torch.float32, device=DEV)
    status = pace.new_status(DEV)
    pace.token_logprob(b, hidden, w, targets, 1.0, lse=lse, status=status)
    dh, dw = pace.token_logprob_backward(b, hidden, w, targets, lse, to_dev(g), status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    dh_np = dh[torch.from_numpy(~in_loss).to(DEV)]
    assert float(dh_np.abs().max().item()) == 0.0
    sample = np.sort(rng.choice(np.nonzero(in_loss)[0], size=6, replace=False))
    hb = hidden[torch.from_numpy(sample).to(DEV)].view(torch.int16).cpu().numpy().view(np.uint16)
    wb = w.view(torch.int16).cpu().numpy().view(np.uint16)
    st, odh, _ = oracle.lmhead_backward(hb, wb, rw.targets[sample], g[sample].astype(np.float64),
                                        with_dw=False)
    assert st == 0
    st, mh, _ = oracle.lmhead_backward(hb, wb, rw.targets[sample], g[sample].astype(np.float64),
                                       with_dw=False, magnitude=True)
    assert st == 0
    got = dh[torch.from_numpy(sample).to(DEV)].cpu().numpy()
    _check_elementwise(got, odh, mh, "dH sampled rows")
    for i in range(len(sample)):
        assert _rel(got[i], odh[i]) <= REL
    # sum over the vocabulary of dW vanishes (sum_v G_rv = 0 for every row)
    col_sum = dw.double().sum(dim=0)
    assert float(col_sum.norm()) <= 1e-2 * float(dw.double().norm())
    assert torch.isfinite(dw).all()


@pytest.mark.parametrize("rows,frac", [(135000, 0.3), (135000, 0.98)])
def test_lmhead_backward_multi_chunk_trimmed(rows, frac):
    """More rows than four 32,768-row chunks, with the rows in the loss ending inside
    the first (frac 0.3: later chunks hold none) or inside the last chunk (0.98):
    the GEMMs cut their extent to the device-side count and dW must still be whole."""
    H, V = 64, 256
    rng = np.random.default_rng(int(frac * 100))
    hb = workloads.bf16_normal_host((rows, H), 1.0, 5)
    wb = workloads.bf16_normal_host((V, H), 2.0 / math.sqrt(H), 6)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    mask = (rng.random(rows) < frac).astype(np.uint8)
    g = (rng.standard_normal(rows) * mask).astype(np.float32)
    so = to_dev(np.array([0, rows], np.int64))
    b = pace.make_batch(so, rows, mask=to_dev(mask))
    hidden, w = bf16_dev(hb), bf16_dev(wb)
    lse = torch.empty(rows, dtype=torch.float32, device=DEV)
    status = pace.new_status(DEV)
    pace.token_logprob(b, hidden, w, to_dev(y), 1.0, lse=lse, status=status)
    dh, dw = pace.token_logprob_backward(b, hidden, w, to_dev(y), lse, to_dev(g), status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    st, odh, odw = oracle.lmhead_backward(hb, wb, y, g.astype(np.float64))
    assert st == 0
    st, mh, mw = oracle.lmhead_backward(hb, wb, y, g.astype(np.float64), magnitude=True)
    assert st == 0
    _check_elementwise(as_np(dh), odh, mh, "dH")
    _check_elementwise(as_np(dw), odw, mw, "dW")
    assert _rel(as_np(dh), odh) <= REL, _rel(as_np(dh), odh)
    assert _rel(as_np(dw), odw) <= REL, _rel(as_np(dw), odw)
    assert (as_np(dh)[mask == 0] == 0).all()
