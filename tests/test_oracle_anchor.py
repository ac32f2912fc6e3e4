"""Pins of the forward-KL anchor (oracle/anchor.py) and of the combined objectives, CPU only."""

import numpy as np
import pytest
import scipy.stats
import torch

import oracle
from oracle.anchor import (MODE_KL, anchor_backward, anchor_forward, kl_divergence, objective_backward,
                           objective_forward)


def _logits(rng, *shape, scale=2.0):
    return rng.normal(0.0, scale, size=shape)


def test_kl_matches_torch_and_scipy():
    """Two independent library routines: torch's kl_div (pointwise p (log p - log q)) and
    scipy's relative entropy of probability vectors."""
    rng = np.random.default_rng(0)
    zp = _logits(rng, 5, 3, 17)
    zq = _logits(rng, 5, 3, 17)
    kl = kl_divergence(zp, zq)
    lp = torch.log_softmax(torch.from_numpy(zp), -1)
    lq = torch.log_softmax(torch.from_numpy(zq), -1)
    ref = torch.nn.functional.kl_div(lq, lp, reduction="none", log_target=True).sum(-1).numpy()
    np.testing.assert_allclose(kl, ref, rtol=1e-13, atol=1e-15)
    p = np.exp(lp.numpy())
    q = np.exp(lq.numpy())
    for idx in np.ndindex(5, 3):
        assert abs(kl[idx] - scipy.stats.entropy(p[idx], q[idx])) < 1e-13


def test_kl_special_cases():
    rng = np.random.default_rng(1)
    z = _logits(rng, 4, 9)
    assert np.all(np.abs(kl_divergence(z, z)) < 1e-15)                       # KL(p || p) = 0
    assert np.allclose(kl_divergence(z, z + 3.7), 0.0, atol=1e-14)           # logits shift freely
    w = _logits(rng, 4, 9)
    assert np.all(kl_divergence(z, w) > 0)                                    # Gibbs' inequality
    np.testing.assert_allclose(kl_divergence(z + 1.0, w - 2.0), kl_divergence(z, w), rtol=1e-12)
    # a target entry of probability 0 contributes nothing (0 log 0 = 0)
    zp = np.array([[0.0, 0.0, -np.inf]])
    zq = np.array([[0.0, 1.0, 2.0]])
    lq = zq - np.log(np.exp(zq).sum())
    assert abs(kl_divergence(zp, zq)[0] - (0.5 * (np.log(0.5) - lq[0, 0]) + 0.5 * (np.log(0.5) - lq[0, 1]))) < 1e-15
    # two-point distributions: the binary relative entropy
    a, b = 0.3, 0.8
    zp = np.log([[a, 1 - a]])
    zq = np.log([[b, 1 - b]])
    assert abs(kl_divergence(zp, zq)[0] - (a * np.log(a / b) + (1 - a) * np.log((1 - a) / (1 - b)))) < 1e-15


def test_kl_by_monte_carlo():
    """E_{x~p}[log p(x) - log q(x)] over 200000 draws, within 5 standard errors."""
    rng = np.random.default_rng(2)
    zp = _logits(rng, 30, scale=1.5)
    zq = zp + _logits(rng, 30, scale=0.7)
    lp = zp - np.log(np.exp(zp).sum())
    lq = zq - np.log(np.exp(zq).sum())
    x = rng.choice(30, size=200000, p=np.exp(lp))
    d = lp[x] - lq[x]
    assert abs(d.mean() - kl_divergence(zp, zq)) < 5 * d.std() / np.sqrt(d.size)


def test_anchor_is_the_mean_over_valid_positions():
    rng = np.random.default_rng(3)
    zp = _logits(rng, 2, 3, 6)
    zq = _logits(rng, 2, 3, 6)
    mask = np.array([[1, 0, 1], [0, 1, 0]], dtype=np.uint8)
    kl = kl_divergence(zp, zq)
    fw = anchor_forward(zp, zq, mask)
    assert fw["npos"] == 3
    assert abs(fw["loss"] - (kl[0, 0] + kl[0, 2] + kl[1, 1]) / 3) < 1e-15
    assert anchor_forward(zp, zq, np.zeros((2, 3)))["loss"] == 0.0
    assert np.all(anchor_backward(zp, zq, np.zeros((2, 3))) == 0.0)


def test_anchor_gradient_matches_torch_autograd():
    rng = np.random.default_rng(4)
    zp = _logits(rng, 3, 2, 11)
    zq = _logits(rng, 3, 2, 11)
    mask = np.array([[1, 1], [0, 1], [1, 0]], dtype=np.uint8)
    g = anchor_backward(zp, zq, mask, dloss=2.5)
    tq = torch.from_numpy(zq).requires_grad_(True)
    lp = torch.log_softmax(torch.from_numpy(zp), -1)
    per = torch.nn.functional.kl_div(torch.log_softmax(tq, -1), lp, reduction="none", log_target=True).sum(-1)
    m = torch.from_numpy(mask.astype(np.float64))
    (2.5 * (per * m).sum() / m.sum()).backward()
    np.testing.assert_allclose(g, tq.grad.numpy(), rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("mode,T", [(MODE_KL | 1, 1.0), (MODE_KL | 2, 0.8), (MODE_KL | 3, 1.0), (MODE_KL | 3, 1.5),
                                    (MODE_KL, 1.0)])
def test_objective_gradient_by_finite_differences(mode, T):
    rng = np.random.default_rng(5)
    N, K, V = 2, 3, 7
    while True:
        zp = _logits(rng, N, K, V, scale=1.5)
        zq = zp + _logits(rng, N, K, V, scale=1.0)
        pt = np.exp(oracle.log_softmax(zp, T))
        qt = np.exp(oracle.log_softmax(zq, T))
        if np.min(np.abs(pt - qt)) > 1e-3:
            break
    mask = np.array([[1, 1, 0], [1, 1, 1]], dtype=np.uint8)
    kw = dict(mode=mode, T=T, w_greedy=0.1, w_sampling=0.6, w_kl=1.0)
    g = objective_backward(zp, zq, mask, dloss=3.0, **kw)
    h = 1e-6
    for idx in np.ndindex(N, K, V):
        a = zq.copy(); a[idx] += h
        b = zq.copy(); b[idx] -= h
        fd = 3.0 * (objective_forward(zp, a, mask, **kw)["loss"] - objective_forward(zp, b, mask, **kw)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-7, (idx, fd, g[idx])


def test_objective_adds_the_terms_with_their_own_normalisers():
    rng = np.random.default_rng(6)
    zp = _logits(rng, 4, 3, 8)
    zq = _logits(rng, 4, 3, 8)
    mask = np.ones((4, 3), dtype=np.uint8)
    mask[1, 0] = 0        # window 1 leaves W; its later positions stay valid for the anchor
    mask[2, 2] = 0
    fw = objective_forward(zp, zq, mask, MODE_KL | 1, 1.0, 0.1, 0.0, 1.0)
    eal = oracle.loss_forward(zp, zq, mask, 1, 1.0, 0.1, 0.0)
    kl = kl_divergence(zp, zq)
    assert eal["nvalid"] == 3 and fw["npos"] == 10
    assert abs(fw["loss"] - (eal["loss"] + kl[mask.astype(bool)].sum() / 10)) < 1e-14


def test_sequence_objective_by_finite_differences():
    rng = np.random.default_rng(7)
    B, Tn, K, V = 1, 5, 3, 6
    zp = _logits(rng, B, Tn, V, scale=1.5)
    zq = zp + _logits(rng, B, Tn, V, scale=1.0)
    mask = np.ones((B, Tn), dtype=np.uint8)
    mask[0, 1] = 0
    kw = dict(mode=MODE_KL | 1, T=1.0, w_greedy=0.1, w_sampling=0.0, w_kl=1.0)
    g = oracle.seq_objective_backward(zp, zq, mask, K, dloss=2.0, **kw)
    h = 1e-6
    for idx in np.ndindex(B, Tn, V):
        a = zq.copy(); a[idx] += h
        b = zq.copy(); b[idx] -= h
        fd = 2.0 * (oracle.seq_objective_forward(zp, a, mask, K, **kw)["loss"]
                    - oracle.seq_objective_forward(zp, b, mask, K, **kw)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-7, (idx, fd, g[idx])
    fw = oracle.seq_objective_forward(zp, zq, mask, K, **kw)
    assert fw["npos"] == 4


# ---------------------------------------------------------------------- the L_TV baseline term

def test_total_variation_against_scipy_and_special_cases():
    import scipy.spatial.distance as ssd
    rng = np.random.default_rng(20)
    zp = _logits(rng, 3, 2, 12)
    zq = _logits(rng, 3, 2, 12)
    tv = oracle.total_variation(zp, zq, 0.7)
    pt = np.exp(oracle.log_softmax(zp, 0.7))
    qt = np.exp(oracle.log_softmax(zq, 0.7))
    for idx in np.ndindex(3, 2):
        assert abs(tv[idx] - 0.5 * ssd.cityblock(pt[idx], qt[idx])) < 1e-14
    np.testing.assert_allclose(tv, 1.0 - oracle.acceptance_sampling(zp, zq, 0.7), atol=1e-14)
    assert np.all(oracle.total_variation(zp, zp, 1.3) < 1e-15)
    a = np.array([[0.0, 0.0, -np.inf, -np.inf]])
    b = np.array([[-np.inf, -np.inf, 0.0, 1.0]])
    assert abs(oracle.total_variation(a, b, 1.0)[0] - 1.0) < 1e-15          # disjoint supports


def test_tv_term_averages_each_window_over_its_valid_positions():
    rng = np.random.default_rng(21)
    zp = _logits(rng, 3, 4, 9)
    zq = _logits(rng, 3, 4, 9)
    mask = np.ones((3, 4), dtype=np.uint8)
    mask[1, 2] = 0          # K_1 = 2
    mask[2, 0] = 0          # window 2 not in W
    fw = oracle.tv_forward(zp, zq, mask, 0.9)
    tv = oracle.total_variation(zp, zq, 0.9)
    want = (tv[0].mean() + tv[1, :2].mean()) / 2
    assert fw["nvalid"] == 2 and abs(fw["loss"] - want) < 1e-15


@pytest.mark.parametrize("mode,T", [(oracle.MODE_TV, 1.0), (oracle.MODE_KL | oracle.MODE_TV, 0.8),
                                    (oracle.MODE_TV | 3, 1.2)])
def test_tv_objective_by_finite_differences(mode, T):
    rng = np.random.default_rng(22)
    N, K, V = 2, 3, 6
    while True:
        zp = _logits(rng, N, K, V, scale=1.5)
        zq = zp + _logits(rng, N, K, V, scale=1.0)
        pt = np.exp(oracle.log_softmax(zp, T))
        qt = np.exp(oracle.log_softmax(zq, T))
        if np.min(np.abs(pt - qt)) > 1e-3:
            break
    mask = np.array([[1, 1, 0], [1, 1, 1]], dtype=np.uint8)
    kw = dict(mode=mode, T=T, w_greedy=0.2, w_sampling=0.5, w_kl=1.0, w_tv=0.1)
    g = objective_backward(zp, zq, mask, dloss=2.0, **kw)
    h = 1e-6
    for idx in np.ndindex(N, K, V):
        a = zq.copy(); a[idx] += h
        b = zq.copy(); b[idx] -= h
        fd = 2.0 * (objective_forward(zp, a, mask, **kw)["loss"] - objective_forward(zp, b, mask, **kw)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-7, (idx, fd, g[idx])
