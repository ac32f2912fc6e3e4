"""The forward-KL anchor of the combined objectives, float64 (test infrastructure only).

Sec. 4.1: the greedy-regime draft is trained on L_KL + 0.1 L_EAL.  The anchor L_KL is a
forward KL from the target to the draft, one per token position:
KL(p_t || q_t) = sum_v p_t(v) (log p_t(v) - log q_t(v)).  The anchor uses the model
distributions themselves (T = 1): the temperature of Sec. 4.1 is stated for p~ and q~,
which only the acceptance terms use.

Readings (the paper says no more than that the KL is taken per token position):
  * the anchor is the mean of the per-position KL over the valid positions (mask 1),
    independent of any window; with none it is 0;
  * its weight w_kl enters the objective as  L = w_kl L_KL + w_g L_EAL + w_s L_WTV,
    each term with its own normaliser (|positions| for the anchor, |W| for the others).

The gradient with respect to the draft logits follows from the draft's log-softmax
Jacobian d log q(v)/dz_u = delta_uv - q(u):
  d KL / dz_u = -sum_v p(v) (delta_uv - q(u)) = q(u) - p(u).
"""

from __future__ import annotations

import numpy as np

from .losses import as_f64, log_softmax, loss_backward, loss_forward

MODE_KL = 4  # the anchor term; combines with MODE_GREEDY / MODE_SAMPLING as a bit


def kl_divergence(target, draft) -> np.ndarray:
    """KL(p || q) of every row of [..., V] logits, natural log, T = 1."""
    lp = log_softmax(as_f64(target), 1.0)
    lq = log_softmax(as_f64(draft), 1.0)
    p = np.exp(lp)
    # 0 log 0 = 0: a target entry of probability 0 contributes nothing
    pos = p > 0.0
    terms = np.zeros_like(p)
    terms[pos] = p[pos] * (lp[pos] - lq[pos])
    return np.sum(terms, axis=-1)


def valid_positions(mask, shape) -> np.ndarray:
    """Boolean validity of every row (position) of logits whose leading shape is ``shape``."""
    if mask is None:
        return np.ones(shape, dtype=bool)
    return np.asarray(mask).astype(bool).reshape(shape)


def anchor_forward(target, draft, mask=None, n_positions_total=None):
    """L_KL = mean KL over the valid positions.  ``n_positions_total`` replaces the count
    when only part of a larger batch is passed in."""
    zp = as_f64(target)
    kl = kl_divergence(zp, draft)
    valid = valid_positions(mask, zp.shape[:-1])
    npos = int(valid.sum()) if n_positions_total is None else int(n_positions_total)
    loss = float(np.sum(np.where(valid, kl, 0.0)) / npos) if npos > 0 else 0.0
    return dict(loss=loss, kl=kl, npos=npos, valid=valid)


def anchor_backward(target, draft, mask=None, dloss: float = 1.0, n_positions_total=None) -> np.ndarray:
    """dloss * dL_KL/dz_q: (q - p) dloss / |positions| on valid rows, zero elsewhere."""
    zp = as_f64(target)
    zq = as_f64(draft)
    fw = anchor_forward(zp, zq, mask, n_positions_total)
    if fw["npos"] == 0:
        return np.zeros_like(zq)
    p = np.exp(log_softmax(zp, 1.0))
    q = np.exp(log_softmax(zq, 1.0))
    return np.where(fw["valid"][..., None], (q - p) * (dloss / fw["npos"]), 0.0)


def objective_forward(target, draft, mask=None, mode: int = MODE_KL | 1, T: float = 1.0,
                      w_greedy: float = 1.0, w_sampling: float = 1.0, w_kl: float = 1.0,
                      n_windows_total=None, n_positions_total=None, w_tv: float = 1.0):
    """w_kl L_KL + w_g L_EAL + w_s L_WTV + w_tv L_TV over [N][K][V] windows (terms selected by
    ``mode``)."""
    fw = loss_forward(target, draft, mask, mode & 3, T, w_greedy, w_sampling, n_windows_total)
    if mode & MODE_KL:
        an = anchor_forward(target, draft, mask, n_positions_total)
        fw["loss"] += w_kl * an["loss"]
        fw["kl"] = an["kl"]
        fw["npos"] = an["npos"]
    if mode & MODE_TV:
        tv = tv_forward(target, draft, mask, T, n_windows_total)
        fw["loss"] += w_tv * tv["loss"]
        fw["tv"] = tv["tv"]
        fw["nvalid"] = tv["nvalid"]
    return fw


def objective_backward(target, draft, mask=None, mode: int = MODE_KL | 1, T: float = 1.0,
                       w_greedy: float = 1.0, w_sampling: float = 1.0, w_kl: float = 1.0,
                       dloss: float = 1.0, n_windows_total=None, n_positions_total=None,
                       w_tv: float = 1.0) -> np.ndarray:
    """dloss * d(objective)/dz_q, [N][K][V]."""
    g = loss_backward(target, draft, mask, mode & 3, T, w_greedy, w_sampling, dloss, n_windows_total)
    if mode & MODE_KL:
        g = g + anchor_backward(target, draft, mask, dloss * w_kl, n_positions_total)
    if mode & MODE_TV:
        g = g + tv_backward(target, draft, mask, T, dloss * w_tv, n_windows_total)
    return g


# ---------------------------------------------------------------------------------------
# The L_TV baseline's auxiliary term (Sec. 4.1): the per-position total variation distance
# averaged across the window, L_aux(t) = (1/gamma) sum_j TV(p~_{t+j}, q~_{t+j}), with
# TV = (1/2) sum_v |p~(v) - q~(v)|.  Readings: a masked window averages over its K_n valid
# leading positions (1/K_n; = 1/gamma without a mask), windows not in W add nothing, and
# L_TV is the mean over W:  L_TV = (1/|W|) sum_{n in W} (1/K_n) sum_{j < K_n} TV_{n,j}.
# Gradient: TV = 1 - sum_v min(p~, q~) (Sec. 3.3), so dTV/dz_u = -d a^sample/dz_u with the
# subgradient of losses.loss_backward (the min follows the frozen p~ at a tie).

MODE_TV = 16  # the L_TV auxiliary term, a mode bit


def total_variation(target, draft, T: float) -> np.ndarray:
    """TV(p~, q~) of every row, from its definition (1/2) sum_v |p~(v) - q~(v)|."""
    pt = np.exp(log_softmax(as_f64(target), T))
    qt = np.exp(log_softmax(as_f64(draft), T))
    return 0.5 * np.sum(np.abs(pt - qt), axis=-1)


def tv_forward(target, draft, mask=None, T: float = 1.0, n_windows_total=None):
    from .losses import leading_valid_depths
    zp = as_f64(target)
    N, K, _ = zp.shape
    kn = leading_valid_depths(mask, N, K)
    tv = total_variation(zp, draft, T)
    per = np.zeros(N)
    for n in range(N):
        if kn[n] >= 1:
            per[n] = np.sum(tv[n, :kn[n]]) / kn[n]
    nvalid = int(np.sum(kn >= 1)) if n_windows_total is None else int(n_windows_total)
    loss = float(np.sum(per) / nvalid) if nvalid > 0 else 0.0
    return dict(loss=loss, tv=tv, per_window=per, kn=kn, nvalid=nvalid)


def tv_backward(target, draft, mask=None, T: float = 1.0, dloss: float = 1.0, n_windows_total=None) -> np.ndarray:
    """dloss * dL_TV/dz_q, [N][K][V]."""
    zp = as_f64(target)
    zq = as_f64(draft)
    fw = tv_forward(zp, zq, mask, T, n_windows_total)
    grad = np.zeros_like(zq)
    if fw["nvalid"] == 0:
        return grad
    lp = log_softmax(zp, T)
    lq = log_softmax(zq, T)
    qt = np.exp(lq)
    c = (lq < lp).astype(np.float64)
    qlt = np.sum(c * qt, axis=-1, keepdims=True)
    da_s = (1.0 / T) * qt * (c - qlt)          # d a^sample / dz_u, as in losses.loss_backward
    N, K, _ = zq.shape
    for n in range(N):
        for j in range(int(fw["kn"][n])):
            grad[n, j] = -dloss / (fw["nvalid"] * fw["kn"][n]) * da_s[n, j]
    return grad
