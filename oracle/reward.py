"""GRPO-stage acceptance reward and advantages, float64 (test infrastructure only).

Sec. 3.4 of the paper: greedy draft trajectories of the current and reference
drafts, the simulated accepted length tau under greedy verification against the
target's argmax tokens, the debiased reward R = tau^theta - tau^ref, and the
clipped group-normalised advantage (Eq. advantage).  The sampling-verification
variant accepts the drafted token with probability min(1, p~/q~) using a
counter-based uniform per (window, depth).
"""

from __future__ import annotations

import numpy as np

from .losses import argmax_lowest, as_f64, log_softmax
from .philox import gumbel_uniforms, uniform01

REWARD_GREEDY = 1
REWARD_SAMPLING = 2
REWARD_SAMPLED_DRAFT = 6   # sampling verification with the drafted token sampled from q~


def greedy_trajectory(z) -> np.ndarray:
    """S_k = argmax_v z_k(v) for each window and depth k (Sec. 3.4, greedy draft trajectory)."""
    return argmax_lowest(as_f64(z))


def simulated_accept_length(accept: np.ndarray) -> np.ndarray:
    """tau = sum_{k=1}^{gamma} prod_{j=1}^{k} 1[draft token j accepted] (Sec. 3.4).

    ``accept`` is [N][gamma] of 0/1; the product form counts the accepted tokens
    before the first rejection.
    """
    N, gamma = accept.shape
    tau = np.zeros(N, dtype=np.int64)
    for n in range(N):
        total = 0
        for k in range(1, gamma + 1):
            prod = 1
            for j in range(k):
                prod *= int(accept[n, j])
            total += prod
        tau[n] = total
    return tau


def sampled_trajectory(draft, T: float, seed: int, row_offset: int = 0) -> np.ndarray:
    """S_k ~ q~_k drawn by the Gumbel-max method: S_k = argmax_v (z_k(v)/T + G_v) with
    G_v = -log(-log U_v), U_v the counter-based uniforms of gumbel_uniforms for (window
    row_offset + n, depth k); lowest index on ties.  (Sec. 2.3: under sampling verification the
    draft samples its token from q~.)"""
    zq = as_f64(draft)
    N, K, V = zq.shape
    S = np.zeros((N, K), dtype=np.int64)
    for n in range(N):
        for k in range(K):
            U = gumbel_uniforms(seed, row_offset + n, k, V)
            S[n, k] = int(np.argmax(zq[n, k] / T - np.log(-np.log(U))))
    return S


def sampling_accepts_at(target, draft, T: float, u: np.ndarray, S: np.ndarray):
    """Acceptance of given drafted tokens S under sampling verification: u < min(1, p~(S)/q~(S))."""
    lp = np.take_along_axis(log_softmax(as_f64(target), T), S[..., None], axis=-1)[..., 0]
    lq = np.take_along_axis(log_softmax(as_f64(draft), T), S[..., None], axis=-1)[..., 0]
    thr = np.minimum(1.0, np.exp(lp - lq))
    return (u < thr).astype(np.int64), thr


def sampling_accepts(target, draft, T: float, u: np.ndarray):
    """Per-position acceptance of the greedy-drafted token under sampling verification.

    The drafted token y = argmax z_q (the trajectory S of Sec. 3.4) is admitted with
    probability min(1, p~(y)/q~(y)) (Sec. 2.3); with the uniform u it is accepted iff
    u < min(1, p~(y)/q~(y)).  Returns (accept [N][K] of 0/1, threshold [N][K]).
    """
    zp = as_f64(target)
    zq = as_f64(draft)
    y = argmax_lowest(zq)
    lp = np.take_along_axis(log_softmax(zp, T), y[..., None], axis=-1)[..., 0]
    lq = np.take_along_axis(log_softmax(zq, T), y[..., None], axis=-1)[..., 0]
    thr = np.minimum(1.0, np.exp(lp - lq))
    return (u < thr).astype(np.int64), thr


def debiased_reward(tau_theta: np.ndarray, tau_ref=None) -> np.ndarray:
    """R = tau^theta - tau^ref, Eq. debiased_reward; without a reference draft R = tau^theta."""
    tau_theta = np.asarray(tau_theta, dtype=np.float64)
    if tau_ref is None:
        return tau_theta
    return tau_theta - np.asarray(tau_ref, dtype=np.float64)


def rollout_lengths(R: np.ndarray, windows_per_rollout: int) -> np.ndarray:
    """Accepted length of a rollout: the mean reward over its consecutive windows."""
    R = np.asarray(R, dtype=np.float64)
    n_roll = R.shape[0] // windows_per_rollout
    out = np.zeros(n_roll, dtype=np.float64)
    for r in range(n_roll):
        out[r] = np.mean(R[r * windows_per_rollout:(r + 1) * windows_per_rollout])
    return out


def group_advantages(x: np.ndarray, group_size: int, clip: float, eps: float = 1e-6) -> np.ndarray:
    """Eq. advantage: A = clip((x - mean_g) / (std_g + eps), -C_A, C_A) within each group.

    std is the population standard deviation of the group; eps = 1e-6 as in the
    paper; groups are consecutive blocks of ``group_size`` samples.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros_like(x)
    for g0 in range(0, x.shape[0], group_size):
        grp = x[g0:g0 + group_size]
        mu = np.mean(grp)
        sd = np.sqrt(np.mean((grp - mu) ** 2))
        out[g0:g0 + group_size] = np.clip((grp - mu) / (sd + eps), -clip, clip)
    return out


def accept_reward(target, draft, ref_draft=None, mode: int = REWARD_GREEDY, T: float = 1.0,
                  seed: int = 0, row_offset: int = 0, windows_per_rollout: int = 1,
                  rollouts_per_group: int = 1, adv_clip: float = 5.0):
    """The reward pipeline of Sec. 3.4 for N windows of [K][V] logits.

    Greedy: accepted iff S_k = x*_k (draft argmax equals target argmax).
    Sampling: accepted iff u(seed, row_offset + n, k) < min(1, p~(S_k)/q~(S_k)), with S_k the
    draft's argmax, or (REWARD_SAMPLED_DRAFT) S_k sampled from q~ by sampled_trajectory; the
    reference draft's tokens are drawn with the same uniforms.
    The reference draft, when given, is verified the same way with the same
    uniforms.  Returns tau, R, rollout lengths, advantages and (for sampling) the
    acceptance thresholds of both drafts, so a comparison can set aside draws that
    sit on the threshold.
    """
    zp = as_f64(target)
    N, K, V = zp.shape
    xstar = argmax_lowest(zp)
    u = None
    if mode in (REWARD_SAMPLING, REWARD_SAMPLED_DRAFT):
        n_idx = np.arange(N, dtype=np.uint64)[:, None] + np.uint64(row_offset)
        k_idx = np.arange(K, dtype=np.uint64)[None, :]
        u = uniform01(seed, n_idx, k_idx)

    def verify(z):
        if mode == REWARD_GREEDY:
            return (greedy_trajectory(z) == xstar).astype(np.int64), None
        if mode == REWARD_SAMPLED_DRAFT:
            return sampling_accepts_at(zp, z, T, u, sampled_trajectory(z, T, seed, row_offset))
        return sampling_accepts(zp, z, T, u)

    acc, thr = verify(draft)
    tau = simulated_accept_length(acc)
    tau_ref, thr_ref = None, None
    if ref_draft is not None:
        acc_ref, thr_ref = verify(ref_draft)
        tau_ref = simulated_accept_length(acc_ref)
    R = debiased_reward(tau, tau_ref)
    rl = rollout_lengths(R, windows_per_rollout)
    adv = group_advantages(rl, rollouts_per_group, adv_clip)
    return dict(tau=tau, tau_ref=tau_ref, R=R, rollout_len=rl, advantage=adv, u=u,
                thr=thr, thr_ref=thr_ref, accept=acc)
