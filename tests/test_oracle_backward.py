"""Pins of the oracle's backward pass: the surrogate derivative against central
finite differences of the oracle's own loss (a different computation: loss
values, not the analytic derivative) away from the clip kinks, and the LM-head
backward against fp64 autograd of a library (torch, CPU, test-only) plus the
vocabulary-sum-zero identity sum_v dW_v = 0."""
import math

import numpy as np
import pytest
import torch

import oracle


def _bits(x):
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy(), t.to(torch.float64).numpy()


@pytest.mark.parametrize("agg", [oracle.AGG_TOKEN_MEAN, oracle.AGG_SEQ_MEAN_TOKEN_MEAN])
def test_surrogate_grad_matches_finite_differences(agg):
    rng = np.random.default_rng(1)
    so = np.array([0, 7, 7, 19, 30], np.int64)
    n = so[-1]
    lp = -rng.random(n) * 6
    behav = lp + rng.normal(0, 0.4, n)
    mask = (rng.random(n) < 0.8).astype(np.uint8)
    adv = np.array([1.3, -0.7, -2.0, 0.4])
    st, g = oracle.surrogate_grad(lp, behav, so, adv, mask=mask, agg=agg)
    assert st == 0
    h = 1e-6
    for r in range(n):
        up, dn = lp.copy(), lp.copy()
        up[r] += h
        dn[r] -= h
        _, lu, _, _ = oracle.surrogate(up, behav, so, adv, mask=mask, agg=agg)
        _, ld, _, _ = oracle.surrogate(dn, behav, so, adv, mask=mask, agg=agg)
        fd = (lu - ld) / (2 * h)
        # skip rows within 2h of a kink (clip bound or dual-clip switch)
        rho = math.exp(lp[r] - behav[r])
        near = min(abs(rho - 0.8), abs(rho - 1.28)) < 1e-4
        if not near:
            assert abs(g[r] - fd) <= 1e-6 * max(1.0, abs(fd)), (r, g[r], fd)


def test_surrogate_grad_zero_in_clipped_regions():
    so = np.array([0, 1], np.int64)
    # A = 1, rho = 1.5 > 1 + eps_high: clipped term active, gradient 0
    st, g = oracle.surrogate_grad([math.log(1.5)], [0.0], so, [1.0])
    assert g[0] == 0.0
    # A = -1, rho = 20: dual clip active, gradient 0
    st, g = oracle.surrogate_grad([math.log(20.0)], [0.0], so, [-1.0])
    assert g[0] == 0.0
    # A = -1, rho = 1.1 inside the trust region: -A rho
    st, g = oracle.surrogate_grad([math.log(1.1)], [0.0], so, [-1.0])
    assert abs(g[0] - 1.1) < 1e-12


@pytest.mark.parametrize("rows,H,V,tau", [(6, 16, 37, 1.0), (9, 32, 70, 0.8)])
def test_lmhead_backward_matches_autograd(rows, H, V, tau):
    rng = np.random.default_rng(rows + V)
    hb, hf = _bits(rng.standard_normal((rows, H)))
    wb, wf = _bits(rng.standard_normal((V, H)) / math.sqrt(H) * 2)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    g = rng.standard_normal(rows)
    g[2] = 0.0
    st, dh, dw = oracle.lmhead_backward(hb, wb, y, g, temperature=tau, n_threads=3)
    assert st == 0
    h = torch.from_numpy(hf).requires_grad_(True)
    w = torch.from_numpy(wf).requires_grad_(True)
    lp = torch.log_softmax(h @ w.T / tau, dim=-1)[torch.arange(rows), torch.from_numpy(y).long()]
    (lp * torch.from_numpy(g)).sum().backward()
    np.testing.assert_allclose(dh, h.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dw, w.grad.numpy(), rtol=1e-10, atol=1e-12)
    assert np.abs(dw.sum(axis=0)).max() < 1e-12  # sum over the vocabulary is zero
    assert (dh[2] == 0).all()


@pytest.mark.parametrize("rows,H,V,tau", [(6, 16, 37, 1.0), (9, 32, 70, 0.8)])
def test_lmhead_backward_magnitude_matches_autograd(rows, H, V, tau):
    """The element-wise error scales sum_v |G_rv||W_vk| and sum_r |G_rv||h_rk|, with G
    the library's autograd gradient of the logits (a different route to G), and the
    triangle-inequality bound they put on dH and dW."""
    rng = np.random.default_rng(rows * V)
    hb, hf = _bits(rng.standard_normal((rows, H)))
    wb, wf = _bits(rng.standard_normal((V, H)) / math.sqrt(H) * 2)
    y = rng.integers(0, V, size=rows).astype(np.int32)
    g = rng.standard_normal(rows)
    g[1] = 0.0
    st, mh, mw = oracle.lmhead_backward(hb, wb, y, g, temperature=tau, n_threads=2,
                                        magnitude=True)
    assert st == 0
    z = torch.from_numpy(hf @ wf.T).requires_grad_(True)
    lp = torch.log_softmax(z / tau, dim=-1)[torch.arange(rows), torch.from_numpy(y).long()]
    (lp * torch.from_numpy(g)).sum().backward()
    G = np.abs(z.grad.numpy())
    np.testing.assert_allclose(mh, G @ np.abs(wf), rtol=1e-10, atol=1e-14)
    np.testing.assert_allclose(mw, G.T @ np.abs(hf), rtol=1e-10, atol=1e-14)
    _, dh, dw = oracle.lmhead_backward(hb, wb, y, g, temperature=tau, n_threads=2)
    assert (np.abs(dh) <= mh * (1 + 1e-12)).all() and (np.abs(dw) <= mw * (1 + 1e-12)).all()
    assert (mh[1] == 0).all()
