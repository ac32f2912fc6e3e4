"""EAL / WTV losses over whole sequences with sliding windows, float64 (test infrastructure only).

Sec. 3.3 (Fig. wtv and its description): the draft and the target each run once over a
sequence, every position t gets its acceptance a_t, and a window of size gamma starts at
every position and slides by one; the loss accumulates -E[L_t] over all window starts W.
The paper does not say what happens at the end of a sequence.  Two readings are offered:
by default a window that runs past the end, or into an invalid position, is truncated there
(the same reading as for masked windows of the windowed layout) and a start belongs to W iff
its own position is valid; with ``full_windows`` only windows whose gamma positions are all
valid and inside the sequence belong to W (for an unmasked sequence of length T, the starts
0 .. T - gamma).

The sequence loss is the windowed loss of losses.py applied to the gathered windows; its
gradient with respect to a position's draft logits is the sum of the gradients of the rows
that position contributes to (one per window that contains it).
"""

from __future__ import annotations

import numpy as np

from .losses import MODE_BOTH, as_f64, leading_valid_depths, loss_backward, loss_forward


def gather_windows(target, draft, mask, K: int, full_windows: bool = False):
    """[B][T][V] logits -> [B*T][K][V] windows (window n = b*T + t covers positions t..t+K-1)
    and their [B*T][K] validity (position valid and inside the sequence; with ``full_windows``
    every depth of a window with fewer than K leading valid positions is invalid)."""
    zp = as_f64(target)
    zq = as_f64(draft)
    B, T, V = zp.shape
    valid = np.ones((B, T), dtype=bool) if mask is None else np.asarray(mask).astype(bool).reshape(B, T)
    wp = np.zeros((B * T, K, V))
    wq = np.zeros((B * T, K, V))
    wm = np.zeros((B * T, K), dtype=np.uint8)
    src = np.full((B * T, K), -1, dtype=np.int64)  # flat position index of each window row
    for b in range(B):
        for t in range(T):
            n = b * T + t
            for j in range(K):
                p = t + j
                if p < T:
                    wp[n, j] = zp[b, p]
                    wq[n, j] = zq[b, p]
                    wm[n, j] = 1 if valid[b, p] else 0
                    src[n, j] = b * T + p
    if full_windows:
        wm[leading_valid_depths(wm, B * T, K) < K] = 0
    return wp, wq, wm, src


def _window_ids(xstar, src):
    """[B][T] token ids -> the [B*T][K] ids of every window row (0 outside the sequence)."""
    flat = np.asarray(xstar, dtype=np.int64).reshape(-1)
    return np.where(src >= 0, flat[np.maximum(src, 0)], 0)


def seq_loss_forward(target, draft, mask, K: int, mode: int = MODE_BOTH, T: float = 1.0,
                     w_greedy: float = 1.0, w_sampling: float = 1.0, n_windows_total=None,
                     full_windows: bool = False, xstar=None):
    """The loss over every sliding window of every sequence (see the module docstring).
    ``n_windows_total`` replaces |W| when the sequences given are a slice of a larger batch;
    ``xstar`` ([B][T] token ids) replaces the target's argmax (greedy term only)."""
    if xstar is not None:
        target = np.zeros(as_f64(draft).shape)   # not read: the ids define x*
    wp, wq, wm, src = gather_windows(target, draft, mask, K, full_windows)
    ids = None if xstar is None else _window_ids(xstar, src)
    return loss_forward(None if ids is not None else wp, wq, wm, mode, T, w_greedy, w_sampling,
                        n_windows_total, ids)


def seq_loss_backward(target, draft, mask, K: int, mode: int = MODE_BOTH, T: float = 1.0,
                      w_greedy: float = 1.0, w_sampling: float = 1.0, dloss: float = 1.0,
                      n_windows_total=None, full_windows: bool = False, xstar=None) -> np.ndarray:
    """dloss * dL/dz_q per position, [B][T][V]: the window rows' gradients added back to the
    positions they were gathered from (|W| replaced by ``n_windows_total`` when given)."""
    zq = as_f64(draft)
    B, Tn, V = zq.shape
    if xstar is not None:
        target = np.zeros(zq.shape)
    wp, wq, wm, src = gather_windows(target, draft, mask, K, full_windows)
    ids = None if xstar is None else _window_ids(xstar, src)
    g = loss_backward(None if ids is not None else wp, wq, wm, mode, T, w_greedy, w_sampling, dloss,
                      n_windows_total, ids)
    out = np.zeros((B * Tn, V))
    for n in range(B * Tn):
        for j in range(K):
            if src[n, j] >= 0:
                out[src[n, j]] += g[n, j]
    return out.reshape(B, Tn, V)


def seq_objective_forward(target, draft, mask, K: int, mode: int = 5, T: float = 1.0,
                          w_greedy: float = 1.0, w_sampling: float = 1.0, w_kl: float = 1.0,
                          n_windows_total=None, n_positions_total=None, full_windows: bool = False,
                          w_tv: float = 1.0):
    """w_kl L_KL + w_g L_EAL + w_s L_WTV over whole sequences: the window terms as in
    seq_loss_forward, the anchor once per valid position (anchor.py)."""
    from .anchor import MODE_KL, MODE_TV, anchor_forward, tv_forward
    fw = seq_loss_forward(target, draft, mask, K, mode & 3, T, w_greedy, w_sampling, n_windows_total,
                          full_windows)
    if mode & MODE_KL:
        an = anchor_forward(target, draft, mask, n_positions_total)
        fw["loss"] += w_kl * an["loss"]
        fw["kl"] = an["kl"]
        fw["npos"] = an["npos"]
    if mode & MODE_TV:   # the L_TV term over the same sliding windows
        wp, wq, wm, _ = gather_windows(target, draft, mask, K, full_windows)
        tv = tv_forward(wp, wq, wm, T, n_windows_total)
        fw["loss"] += w_tv * tv["loss"]
        fw["nvalid"] = tv["nvalid"]
    return fw


def seq_objective_backward(target, draft, mask, K: int, mode: int = 5, T: float = 1.0,
                           w_greedy: float = 1.0, w_sampling: float = 1.0, w_kl: float = 1.0,
                           dloss: float = 1.0, n_windows_total=None, n_positions_total=None,
                           full_windows: bool = False, w_tv: float = 1.0) -> np.ndarray:
    """dloss * d(objective)/dz_q per position, [B][T][V]."""
    from .anchor import MODE_KL, MODE_TV, anchor_backward, tv_backward
    g = seq_loss_backward(target, draft, mask, K, mode & 3, T, w_greedy, w_sampling, dloss,
                          n_windows_total, full_windows)
    if mode & MODE_KL:
        g = g + anchor_backward(target, draft, mask, dloss * w_kl, n_positions_total)
    if mode & MODE_TV:   # window rows' gradients added back to their positions
        B, Tn, V = as_f64(draft).shape
        wp, wq, wm, src = gather_windows(target, draft, mask, K, full_windows)
        gw = tv_backward(wp, wq, wm, T, dloss * w_tv, n_windows_total)
        out = np.zeros((B * Tn, V))
        for n in range(B * Tn):
            for j in range(K):
                if src[n, j] >= 0:
                    out[src[n, j]] += gw[n, j]
        g = g + out.reshape(B, Tn, V)
    return g


# ---------------------------------------------------------------------------------------
# The GRPO stage over sequences (Sec. 3.4): the three forward passes run once per sequence
# and the window samples are sliced from them.  Windows are given by their start positions
# (flat index b*T + t, each window inside its sequence); the surrogate is grpo.py's over the
# sliced windows, and a position's gradient row adds the rows of every window that covers it.

def slice_windows(x, starts, K: int):
    """[B][T][V] -> the [N][K][V] windows starting at the given flat positions."""
    z = as_f64(x)
    B, T, V = z.shape
    flat = z.reshape(B * T, V)
    starts = np.asarray(starts, dtype=np.int64)
    for s in starts:
        if s < 0 or s % T + K > T:
            raise ValueError("a window must lie inside its sequence")
    return np.stack([flat[s:s + K] for s in starts]) if len(starts) else np.zeros((0, K, V))


def seq_grpo_forward(target, draft, ref, starts, K: int, **grpo_kw):
    from .grpo import grpo_forward
    return grpo_forward(slice_windows(target, starts, K), slice_windows(draft, starts, K),
                        slice_windows(ref, starts, K), **grpo_kw)


def seq_grpo_backward(target, draft, ref, starts, K: int, dloss: float = 1.0, **grpo_kw) -> np.ndarray:
    """dloss * dL_GRPO/dz_theta per position, [B][T][V]."""
    from .grpo import grpo_backward
    zq = as_f64(draft)
    B, T, V = zq.shape
    g = grpo_backward(slice_windows(target, starts, K), slice_windows(draft, starts, K),
                      slice_windows(ref, starts, K), dloss=dloss, **grpo_kw)
    out = np.zeros((B * T, V))
    for n, s in enumerate(np.asarray(starts, dtype=np.int64)):
        for k in range(K):
            out[s + k] += g[n, k]
    return out.reshape(B, T, V)
