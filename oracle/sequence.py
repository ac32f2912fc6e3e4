"""EAL / WTV losses over whole sequences with sliding windows, float64 (test infrastructure only).

Sec. 3.3 (Fig. wtv and its description): the draft and the target each run once over a
sequence, every position t gets its acceptance a_t, and a window of size gamma starts at
every position and slides by one; the loss accumulates -E[L_t] over all window starts W.
Windows that run past the end of a sequence, or into an invalid position, are truncated
there (the same reading as for masked windows of the windowed layout), and a start belongs
to W iff its own position is valid.

The sequence loss is the windowed loss of losses.py applied to the gathered windows; its
gradient with respect to a position's draft logits is the sum of the gradients of the rows
that position contributes to (one per window that contains it).
"""

from __future__ import annotations

import numpy as np

from .losses import MODE_BOTH, as_f64, loss_backward, loss_forward


def gather_windows(target, draft, mask, K: int):
    """[B][T][V] logits -> [B*T][K][V] windows (window n = b*T + t covers positions t..t+K-1)
    and their [B*T][K] validity (position valid and inside the sequence)."""
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
    return wp, wq, wm, src


def seq_loss_forward(target, draft, mask, K: int, mode: int = MODE_BOTH, T: float = 1.0,
                     w_greedy: float = 1.0, w_sampling: float = 1.0):
    """The loss over every sliding window of every sequence (see the module docstring)."""
    wp, wq, wm, _ = gather_windows(target, draft, mask, K)
    return loss_forward(wp, wq, wm, mode, T, w_greedy, w_sampling)


def seq_loss_backward(target, draft, mask, K: int, mode: int = MODE_BOTH, T: float = 1.0,
                      w_greedy: float = 1.0, w_sampling: float = 1.0, dloss: float = 1.0) -> np.ndarray:
    """dloss * dL/dz_q per position, [B][T][V]: the window rows' gradients added back to the
    positions they were gathered from."""
    zq = as_f64(draft)
    B, Tn, V = zq.shape
    wp, wq, wm, src = gather_windows(target, draft, mask, K)
    g = loss_backward(wp, wq, wm, mode, T, w_greedy, w_sampling, dloss)
    out = np.zeros((B * Tn, V))
    for n in range(B * Tn):
        for j in range(K):
            if src[n, j] >= 0:
                out[src[n, j]] += g[n, j]
    return out.reshape(B, Tn, V)
