"""The GRPO surrogate loss of Sec. 3.4, float64 (test infrastructure only).

For each window t of gamma = K positions:
  * the draft's greedy trajectory S_k = argmax z_theta,k (Sec. 3.4) and the reward and
    advantage of accept_reward (simulated greedy verification, R = tau^theta - tau^ref,
    group-standardised and clipped, Eq. advantage), with gradients stopped;
  * the log policy ratio along that trajectory, a per-token geometric mean
        log rho_t = (1/gamma) sum_k [log pi_theta(S_k) - log pi_ref(S_k)],
    with pi = softmax of the logits at T = 1, clipped to [-10, 10], and
    rho_t = exp(log rho_t) clipped to [rho_min, rho_max];
  * the PPO-style clipped surrogate min(rho_t A_t, clip(rho_t, 1 - eps, 1 + eps) A_t).
The group loss is minus the mean surrogate over the group's windows and L_GRPO is the mean
over groups.

Readings: the paper gives no values for rho_min, rho_max and eps_clip (arguments here).  When
a rollout holds several windows (windows_per_rollout > 1, a generalisation; the paper's
samples are single windows), every window of the rollout takes the rollout's advantage and a
group's mean runs over its windows.

Gradient (the argmax trajectory is piecewise constant and held fixed; R and A are stopped):
  d log pi(S_k)/dz_k,u = delta_{u,S_k} - pi_k(u)   (log-softmax Jacobian),
  d log rho_t/dz_k,u   = (1/gamma)(delta_{u,S_k} - pi_k(u)) inside the [-10, 10] clip, else 0,
  d rho_t / d log rho_t = rho_t inside [rho_min, rho_max], else 0,
  d surrogate / d rho  = A when the unclipped term is the minimum, i.e. when
                         (A >= 0 and rho <= 1 + eps) or (A < 0 and rho >= 1 - eps); else 0.
Clip boundaries count as inside.
"""

from __future__ import annotations

import numpy as np

from .losses import as_f64, log_softmax
from .reward import REWARD_GREEDY, accept_reward, greedy_trajectory

LOG_RHO_CLIP = 10.0   # Sec. 3.4 clips log rho to [-10, 10] before exponentiating


def trajectory_log_probs(z, S) -> np.ndarray:
    """log pi(S_k) = log softmax(z_k)(S_k) at T = 1, [N][K]."""
    lz = log_softmax(as_f64(z), 1.0)
    return np.take_along_axis(lz, np.asarray(S)[..., None], axis=-1)[..., 0]


def policy_log_ratio(draft, ref_draft, log_rho_clip: float = LOG_RHO_CLIP):
    """(clipped log rho [N], raw log rho [N], trajectory S [N][K])."""
    S = greedy_trajectory(draft)
    K = S.shape[1]
    raw = np.sum(trajectory_log_probs(draft, S) - trajectory_log_probs(ref_draft, S), axis=1) / K
    return np.clip(raw, -log_rho_clip, log_rho_clip), raw, S


def grpo_forward(target, draft, ref_draft, windows_per_rollout: int = 1, rollouts_per_group: int = 1,
                 adv_clip: float = 5.0, eps_clip: float = 0.2, rho_min: float = 0.0,
                 rho_max: float = 10.0, log_rho_clip: float = LOG_RHO_CLIP,
                 advantage_window=None, n_windows_total=None):
    """``advantage_window`` and ``n_windows_total`` stand in for the advantages and N of a larger
    batch when only some of its windows are passed in (then the loss is those windows' share)."""
    zq = as_f64(draft)
    N = zq.shape[0]
    rw = None
    if advantage_window is None:
        rw = accept_reward(target, draft, ref_draft, REWARD_GREEDY, windows_per_rollout=windows_per_rollout,
                           rollouts_per_group=rollouts_per_group, adv_clip=adv_clip)
        A = np.repeat(rw["advantage"], windows_per_rollout)       # per window
    else:
        A = np.asarray(advantage_window, dtype=np.float64)
    log_rho, raw, S = policy_log_ratio(draft, ref_draft, log_rho_clip)
    rho_exp = np.exp(log_rho)
    rho = np.clip(rho_exp, rho_min, rho_max)
    surrogate = np.minimum(rho * A, np.clip(rho, 1.0 - eps_clip, 1.0 + eps_clip) * A)
    m = windows_per_rollout * rollouts_per_group
    if n_windows_total is None:
        G = N // m
        group_loss = np.array([-np.mean(surrogate[g * m:(g + 1) * m]) for g in range(G)])
        loss = float(np.mean(group_loss)) if G > 0 else 0.0
    else:   # equal groups: the mean of group means is the mean over all windows
        group_loss = None
        loss = float(-np.sum(surrogate) / n_windows_total)
    return dict(loss=loss, group_loss=group_loss, log_rho=log_rho, log_rho_raw=raw, rho=rho,
                rho_exp=rho_exp, advantage_window=A, surrogate=surrogate, S=S, reward=rw)


def grpo_backward(target, draft, ref_draft, windows_per_rollout: int = 1, rollouts_per_group: int = 1,
                  adv_clip: float = 5.0, eps_clip: float = 0.2, rho_min: float = 0.0,
                  rho_max: float = 10.0, log_rho_clip: float = LOG_RHO_CLIP,
                  dloss: float = 1.0, advantage_window=None, n_windows_total=None) -> np.ndarray:
    """dloss * dL_GRPO/dz_theta, [N][K][V] (see the module docstring)."""
    zq = as_f64(draft)
    N, K, V = zq.shape
    fw = grpo_forward(target, draft, ref_draft, windows_per_rollout, rollouts_per_group, adv_clip,
                      eps_clip, rho_min, rho_max, log_rho_clip, advantage_window, n_windows_total)
    m = windows_per_rollout * rollouts_per_group
    n_all = N if n_windows_total is None else int(n_windows_total)
    G = n_all // m
    grad = np.zeros((N, K, V))
    if G == 0:
        return grad
    pi = np.exp(log_softmax(zq, 1.0))
    for t in range(N):
        A = fw["advantage_window"][t]
        rho = fw["rho"][t]
        unclipped = (A >= 0 and rho <= 1.0 + eps_clip) or (A < 0 and rho >= 1.0 - eps_clip)
        d_surr = A if unclipped else 0.0
        inside_rho = rho_min <= fw["rho_exp"][t] <= rho_max
        inside_log = -log_rho_clip <= fw["log_rho_raw"][t] <= log_rho_clip
        d_rho = fw["rho_exp"][t] if (inside_rho and inside_log) else 0.0
        coef = dloss * (-1.0 / (G * m)) * d_surr * d_rho / K
        for k in range(K):
            onehot = np.zeros(V)
            onehot[fw["S"][t, k]] = 1.0
            grad[t, k] = coef * (onehot - pi[t, k])
    return grad
