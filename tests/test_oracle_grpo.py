"""Pins of the GRPO surrogate (oracle/grpo.py), CPU only."""

import math

import numpy as np
import pytest

from oracle.grpo import grpo_backward, grpo_forward, policy_log_ratio, trajectory_log_probs


def _two_token_logits(a):
    """V = 2 logits [a, 0]: for a > 0 the argmax is token 0 and log pi(0) = -log(1 + e^-a)."""
    return np.array([a, 0.0])


def test_log_prob_of_the_argmax_is_minus_log_sum_exp_from_the_max():
    rng = np.random.default_rng(0)
    z = rng.normal(0, 2, size=(3, 4, 50))
    S = np.argmax(z, axis=-1)
    lp = trajectory_log_probs(z, S)
    m = z.max(-1, keepdims=True)
    np.testing.assert_allclose(lp, -np.log(np.exp(z - m).sum(-1)), rtol=0, atol=1e-14)
    a = 1.3
    assert abs(trajectory_log_probs(_two_token_logits(a)[None, None], [[0]])[0, 0]
               + math.log1p(math.exp(-a))) < 1e-15


def test_log_ratio_is_the_mean_over_the_window_and_clipped_at_ten():
    zq = np.stack([_two_token_logits(a) for a in (1.0, 2.0, 0.5)])[None]       # [1][3][2]
    zr = np.stack([_two_token_logits(b) for b in (0.2, 3.0, 0.5)])[None]
    lr, raw, S = policy_log_ratio(zq, zr)
    want = np.mean([math.log1p(math.exp(-b)) - math.log1p(math.exp(-a))
                    for a, b in [(1.0, 0.2), (2.0, 3.0), (0.5, 0.5)]])
    assert S.tolist() == [[0, 0, 0]]
    assert abs(raw[0] - want) < 1e-15 and lr[0] == raw[0]
    zq = np.array([[[60.0, 0.0]]])
    zr = np.array([[[-40.0, 0.0]]])      # log pi_ref(S) = -40 (to 1e-17): raw log rho ~ 40
    lr, raw, _ = policy_log_ratio(zq, zr)
    assert raw[0] > 39.9 and lr[0] == 10.0
    # a uniform draft over 1e5 tokens (S = 0, log pi = -log 1e5) against a reference peaked on
    # token 0: raw log rho = -11.51 -> -10
    zq = np.zeros((1, 1, 100000))
    zr = np.zeros((1, 1, 100000))
    zr[0, 0, 0] = 50.0
    lr, raw, _ = policy_log_ratio(zq, zr)
    assert abs(raw[0] + math.log(1e5)) < 1e-9 and lr[0] == -10.0


def _pair_group(a_theta, b_ref, theta_correct=(True, False), ref_correct=(False, False)):
    """One group of two single-depth windows, V = 2: target argmax token 0 (logits [5, 0]).
    Window w: draft [+-a, 0] (token 0 iff correct), reference [+-b, 0]."""
    tgt = np.array([[[5.0, 0.0]], [[5.0, 0.0]]])
    dr = np.array([[[a if c else -a, 0.0]] for a, c in zip(a_theta, theta_correct)])
    rf = np.array([[[b if c else -b, 0.0]] for b, c in zip(b_ref, ref_correct)])
    return tgt, dr, rf


def test_ppo_clip_cases_by_hand():
    """R = tau^theta - tau^ref = [1, 0] -> A = [+c, -c] with c = 0.5 / (0.5 + 1e-6).  The draft
    puts its argmax on token 0 or 1; log pi(S) for V = 2 has the logistic closed form."""
    c = 0.5 / (0.5 + 1e-6)
    # window 0 (A > 0): draft [3, 0] -> S = 0, pi(0) = 1/(1+e^-3); ref [-1, 0], pi_ref(0) = 1/(1+e^1)
    # window 1 (A < 0): draft [-2, 0] -> S = 1, pi(1) = 1/(1+e^-2); ref [-0.3, 0], pi_ref(1) = 1/(1+e^-0.3)
    tgt, dr, rf = _pair_group((3.0, 2.0), (1.0, 0.3))
    rho0 = (1 + math.exp(1.0)) / (1 + math.exp(-3.0))         # ~ 3.54 > 1.2, A > 0: clipped branch
    rho1 = (1 + math.exp(-0.3)) / (1 + math.exp(-2.0))        # ~ 1.49 > 1.2, A < 0: unclipped
    fw = grpo_forward(tgt, dr, rf, 1, 2, eps_clip=0.2, rho_min=0.0, rho_max=10.0)
    np.testing.assert_allclose(fw["reward"]["R"], [1.0, 0.0])
    np.testing.assert_allclose(fw["advantage_window"], [c, -c], rtol=1e-15)
    np.testing.assert_allclose(fw["rho"], [rho0, rho1], rtol=1e-14)
    want = -0.5 * (1.2 * c + rho1 * (-c))
    assert abs(fw["loss"] - want) < 1e-14
    g = grpo_backward(tgt, dr, rf, 1, 2, eps_clip=0.2, rho_min=0.0, rho_max=10.0)
    assert np.all(g[0] == 0.0)                                  # clipped: no gradient
    # window 1: coef = -(1/2) * A * rho / K, direction (onehot(S=1) - pi)
    pi = np.array([math.exp(-2.0), 1.0]) / (1 + math.exp(-2.0))
    np.testing.assert_allclose(g[1, 0], -0.5 * (-c) * rho1 * (np.array([0.0, 1.0]) - pi), rtol=1e-13)


def test_rho_clip_stops_the_gradient():
    tgt, dr, rf = _pair_group((3.0, 2.0), (1.0, 0.3))
    fw = grpo_forward(tgt, dr, rf, 1, 2, eps_clip=0.2, rho_min=0.0, rho_max=1.4)
    assert fw["rho"][1] == 1.4
    g = grpo_backward(tgt, dr, rf, 1, 2, eps_clip=0.2, rho_min=0.0, rho_max=1.4)
    assert np.all(g == 0.0)


def test_identical_policies_give_rho_one_and_zero_loss():
    """pi_theta = pi_ref: rho = 1 everywhere, the surrogate is A, and an unclipped group's
    advantages have mean 0, so every group loss is 0."""
    rng = np.random.default_rng(1)
    tgt = rng.normal(0, 2, size=(8, 3, 20))
    dr = tgt + rng.normal(0, 1.5, size=tgt.shape)
    fw = grpo_forward(tgt, dr, dr, 2, 2, adv_clip=100.0)
    np.testing.assert_allclose(fw["rho"], 1.0, rtol=0, atol=1e-15)
    assert np.all(np.abs(fw["group_loss"]) < 1e-15)


@pytest.mark.parametrize("wpr,rpg,eps", [(1, 4, 0.2), (2, 2, 0.3), (1, 2, 0.05)])
def test_gradient_by_finite_differences(wpr, rpg, eps):
    """Inputs with a clear argmax (margin >= 1) so the trajectory and tau stay fixed under a
    1e-6 step, and rho away from every clip boundary."""
    rng = np.random.default_rng(7 + wpr)
    N, K, V = 8, 3, 6
    for _ in range(200):
        tgt = rng.normal(0, 2, size=(N, K, V))
        dr = rng.normal(0, 1, size=(N, K, V))
        # a planted argmax 3 above the rest, on the target's token for about half the rows
        S = np.where(rng.random((N, K)) < 0.6, np.argmax(tgt, -1), rng.integers(0, V, (N, K)))
        np.put_along_axis(dr, S[..., None], np.max(dr, -1, keepdims=True) + 3.0, axis=-1)
        rf = dr + rng.normal(0, 0.4, size=(N, K, V))
        # the reference moves its argmax on about 40% of the rows, so tau^ref differs
        Sr = np.where(rng.random((N, K)) < 0.4, rng.integers(0, V, (N, K)), S)
        np.put_along_axis(rf, Sr[..., None], np.max(rf, -1, keepdims=True) + 1.5, axis=-1)
        fw = grpo_forward(tgt, dr, rf, wpr, rpg, eps_clip=eps, rho_min=0.0, rho_max=10.0)
        if np.min(np.abs(fw["rho"] - (1 + eps))) > 1e-3 and np.min(np.abs(fw["rho"] - (1 - eps))) > 1e-3 \
                and np.any(fw["advantage_window"] != 0):
            break
    else:
        raise AssertionError("no admissible input in 200 draws")
    g = grpo_backward(tgt, dr, rf, wpr, rpg, eps_clip=eps, dloss=2.0)
    h = 1e-6
    for idx in np.ndindex(N, K, V):
        a = dr.copy(); a[idx] += h
        b = dr.copy(); b[idx] -= h
        fd = 2.0 * (grpo_forward(tgt, a, rf, wpr, rpg, eps_clip=eps)["loss"]
                    - grpo_forward(tgt, b, rf, wpr, rpg, eps_clip=eps)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-8, (idx, fd, g[idx])
    assert np.any(g != 0)


def test_a_slice_with_the_batch_advantages_gives_its_rows():
    """The full-size GPU test checks sampled windows against the oracle run on those windows
    alone, given the whole batch's advantages and N: their gradient rows are unchanged."""
    rng = np.random.default_rng(11)
    N, K, V = 8, 2, 5
    tgt = rng.normal(0, 2, size=(N, K, V))
    dr = tgt + rng.normal(0, 1.5, size=(N, K, V))
    rf = tgt + rng.normal(0, 1.5, size=(N, K, V))
    full = grpo_forward(tgt, dr, rf, 1, 4)
    g = grpo_backward(tgt, dr, rf, 1, 4, dloss=3.0)
    sel = [1, 5, 6]
    fs = grpo_forward(tgt[sel], dr[sel], rf[sel], 1, 4, advantage_window=full["advantage_window"][sel],
                      n_windows_total=N)
    gs = grpo_backward(tgt[sel], dr[sel], rf[sel], 1, 4, dloss=3.0,
                       advantage_window=full["advantage_window"][sel], n_windows_total=N)
    np.testing.assert_allclose(gs, g[sel], rtol=0, atol=1e-16)
    np.testing.assert_allclose(fs["rho"], full["rho"][sel], rtol=0, atol=0)
    assert abs(fs["loss"] - (-np.sum(full["surrogate"][sel]) / N)) < 1e-16


def test_sequence_grpo_gradient_by_finite_differences():
    """Overlapping windows sliced from one sequence pass (Sec. 3.4): the per-position gradient
    adds every covering window's row; checked against central differences of the loss."""
    from oracle.sequence import seq_grpo_backward, seq_grpo_forward
    rng = np.random.default_rng(17)
    B, T, K, V = 2, 9, 3, 5
    for _ in range(200):
        tgt = rng.normal(0, 2, size=(B, T, V))
        dr = rng.normal(0, 1, size=(B, T, V))
        S = np.where(rng.random((B, T)) < 0.6, np.argmax(tgt, -1), rng.integers(0, V, (B, T)))
        np.put_along_axis(dr, S[..., None], np.max(dr, -1, keepdims=True) + 3.0, axis=-1)
        rf = dr + rng.normal(0, 0.4, size=(B, T, V))
        Sr = np.where(rng.random((B, T)) < 0.4, rng.integers(0, V, (B, T)), S)
        np.put_along_axis(rf, Sr[..., None], np.max(rf, -1, keepdims=True) + 1.5, axis=-1)
        starts = [0, 1, 2, 4, 9 + 0, 9 + 3, 9 + 5, 9 + 6]          # two groups of four, overlapping
        kw = dict(windows_per_rollout=1, rollouts_per_group=4, eps_clip=0.25)
        fw = seq_grpo_forward(tgt, dr, rf, starts, K, **kw)
        if np.min(np.abs(fw["rho"] - 1.25)) > 1e-3 and np.min(np.abs(fw["rho"] - 0.75)) > 1e-3 \
                and np.any(fw["advantage_window"] != 0):
            break
    else:
        raise AssertionError("no admissible input")
    g = seq_grpo_backward(tgt, dr, rf, starts, K, dloss=2.0, **kw)
    h = 1e-6
    for idx in np.ndindex(B, T, V):
        a = dr.copy(); a[idx] += h
        b = dr.copy(); b[idx] -= h
        fd = 2.0 * (seq_grpo_forward(tgt, a, rf, starts, K, **kw)["loss"]
                    - seq_grpo_forward(tgt, b, rf, starts, K, **kw)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-8, (idx, fd, g[idx])
    assert np.all(g[0, 7:] == 0) and np.any(g != 0)        # positions 7, 8 of sequence 0 are in no window
