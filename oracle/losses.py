"""EAL / WTV losses and their draft-logit gradient, in float64 (test infrastructure only).

Notation follows the paper (Sec. 2.3): ``p`` is the frozen target, ``q`` the draft,
``z_p`` / ``z_q`` their logits, ``T`` the sampling temperature, ``gamma`` (= K) the
speculative window size.  Logit tensors are [N windows][K depths][V]; depth j of
window n is the position t + j of the window starting at t.
"""

from __future__ import annotations

import numpy as np

MODE_GREEDY = 1     # EAL, greedy verification
MODE_SAMPLING = 2   # WTV, sampling verification
MODE_BOTH = 3       # w_g * L_EAL + w_s * L_WTV


def as_f64(x) -> np.ndarray:
    """Widen fp32 / bf16 logits to float64 exactly (bf16 -> fp32 -> fp64 loses nothing)."""
    if hasattr(x, "detach"):  # a torch tensor; bf16 has no numpy dtype
        return x.detach().to("cpu").double().numpy()
    return np.asarray(x, dtype=np.float64)


def log_softmax(z: np.ndarray, T: float = 1.0) -> np.ndarray:
    """log of the temperature-scaled distribution along the last axis.

    Sec. 2.3 (Preliminaries): p~(v) is proportional to exp(log p(v) / T).  Since
    log p(v) = z(v) - logsumexp(z), this is softmax(z / T), whose log is
    z/T - logsumexp(z/T).  The log-sum-exp is taken with the row maximum
    factored out.  Entries of -inf get probability 0.
    """
    s = z / T
    m = np.max(s, axis=-1, keepdims=True)
    return s - (m + np.log(np.sum(np.exp(s - m), axis=-1, keepdims=True)))


def argmax_lowest(z: np.ndarray) -> np.ndarray:
    """argmax over the vocabulary; the lowest index wins a tie (np.argmax keeps the first)."""
    return np.argmax(z, axis=-1)


def acceptance_greedy(zp: np.ndarray, zq: np.ndarray):
    """Greedy-verification acceptance, Eq. acc_greedy (Sec. 2.3).

    The target commits to x* = argmax_v p(v) and the drafted token is admitted only
    if it equals x*, so a^greedy = q(x*): the (unscaled, T = 1) draft probability of
    the target's choice.  Returns (a_greedy, x_star).
    """
    xstar = argmax_lowest(zp)
    lq1 = log_softmax(zq, 1.0)
    a = np.exp(np.take_along_axis(lq1, xstar[..., None], axis=-1)[..., 0])
    return a, xstar


def acceptance_sampling(zp: np.ndarray, zq: np.ndarray, T: float) -> np.ndarray:
    """Sampling-verification acceptance, Eq. acc_sample (Sec. 2.3) and Eq. rejection_rate.

    a^sample = E_{y ~ q~}[min(1, p~(y)/q~(y))] = sum_v min(p~(v), q~(v)) = 1 - TV(p~, q~),
    with both distributions temperature-scaled.
    """
    pt = np.exp(log_softmax(zp, T))
    qt = np.exp(log_softmax(zq, T))
    return np.sum(np.minimum(pt, qt), axis=-1)


def row_acceptances(zp: np.ndarray, zq: np.ndarray, T: float):
    """(a_greedy, a_sample, x_star) for every row of [..., V] logits."""
    a_g, xstar = acceptance_greedy(zp, zq)
    a_s = acceptance_sampling(zp, zq, T) if T > 0 else np.full(a_g.shape, np.nan)
    return a_g, a_s, xstar


def leading_valid_depths(mask, N: int, K: int) -> np.ndarray:
    """K_n: how many leading depths of window n are valid positions.

    The paper defines the window over valid positions only (Sec. 3.1, the set W of
    window starts).  Reading used here: a window stops at its first invalid
    position, and it belongs to W iff its first position is valid (K_n >= 1).
    ``mask`` is [N][K] with 1 = valid, or None for all valid.
    """
    if mask is None:
        return np.full(N, K, dtype=np.int64)
    m = np.asarray(mask).astype(bool).reshape(N, K)
    kn = np.zeros(N, dtype=np.int64)
    for n in range(N):
        k = 0
        while k < K and m[n, k]:
            k += 1
        kn[n] = k
    return kn


def expected_length(a: np.ndarray, kn: np.ndarray) -> np.ndarray:
    """Expected accepted length of each window, Eq. eal_generic / eal_compact (Sec. 3.1-3.2).

    E[L_t] = sum_{k=1}^{gamma} prod_{j=0}^{k-1} a_{t+j}, with gamma = K_n for a
    window truncated at its first invalid position.  ``a`` is [N][K].
    """
    N = a.shape[0]
    out = np.zeros(N, dtype=np.float64)
    for n in range(N):
        total = 0.0
        for k in range(1, int(kn[n]) + 1):
            prod = 1.0
            for j in range(k):
                prod *= a[n, j]
            total += prod
        out[n] = total
    return out


def expected_length_partials(a: np.ndarray, kn: np.ndarray) -> np.ndarray:
    """d E[L_t] / d a_{t+j} for every window and depth, from Eq. eal_generic.

    Term k of the sum contains a_{t+j} iff j <= k-1, and its derivative is the same
    product with that factor left out:
    dE/da_j = sum_{k=j+1}^{gamma} prod_{i<k, i != j} a_i  (zero for j >= gamma).
    """
    N, K = a.shape
    out = np.zeros((N, K), dtype=np.float64)
    for n in range(N):
        g = int(kn[n])
        for j in range(g):
            total = 0.0
            for k in range(j + 1, g + 1):
                prod = 1.0
                for i in range(k):
                    if i != j:
                        prod *= a[n, i]
                total += prod
            out[n, j] = total
    return out


def _weights(mode: int, w_greedy: float, w_sampling: float):
    wg = w_greedy if mode & MODE_GREEDY else 0.0
    ws = w_sampling if mode & MODE_SAMPLING else 0.0
    return wg, ws


def loss_forward(target, draft, mask=None, mode: int = MODE_BOTH, T: float = 1.0,
                 w_greedy: float = 1.0, w_sampling: float = 1.0, n_windows_total=None, xstar=None):
    """The EAL and WTV losses, Eq. loss_eal (Sec. 3.2) and Eq. loss_tv (Sec. 3.3).

    L_EAL = -(1/|W|) sum_t sum_k prod_{j<k} a^greedy_{t+j}
    L_WTV = -(1/|W|) sum_t sum_k prod_{j<k} (1 - TV(p~_{t+j}, q~_{t+j}))
    L     = w_greedy L_EAL + w_sampling L_WTV  (only the terms ``mode`` selects)

    ``target`` and ``draft`` are [N][K][V] logits.  |W| is the number of windows
    whose first position is valid; with none the loss is 0.  ``n_windows_total``
    overrides |W| when only some windows of a larger batch are passed in.
    Returns a dict with the loss, the per-window expected lengths and the
    per-position acceptances.

    ``xstar`` ([N][K] token ids) gives the target's tokens directly (Sec. 3.2: for greedy
    target-generated data x* is the ground-truth token); the target logits are then not
    needed (``target`` may be None) and only the greedy term is defined.
    """
    zq = as_f64(draft)
    if xstar is not None:
        if mode & MODE_SAMPLING:
            raise ValueError("token ids define the greedy term only")
        zp = None
        N, K, V = zq.shape
    else:
        zp = as_f64(target)
        N, K, V = zp.shape
    kn = leading_valid_depths(mask, N, K)
    nvalid = int(np.sum(kn >= 1)) if n_windows_total is None else int(n_windows_total)
    wg, ws = _weights(mode, w_greedy, w_sampling)
    if xstar is None:
        a_g, xstar = acceptance_greedy(zp, zq)
    else:
        xstar = np.asarray(xstar, dtype=np.int64).reshape(N, K)
        a_g = np.exp(np.take_along_axis(log_softmax(zq, 1.0), xstar[..., None], axis=-1)[..., 0])
    eal_g = expected_length(a_g, kn) if mode & MODE_GREEDY else np.zeros(N)
    if mode & MODE_SAMPLING:
        a_s = acceptance_sampling(zp, zq, T)
        eal_s = expected_length(a_s, kn)
    else:
        a_s = np.full((N, K), np.nan)
        eal_s = np.zeros(N)
    if nvalid == 0:
        loss = 0.0
    else:
        loss = -(wg * np.sum(eal_g) + ws * np.sum(eal_s)) / nvalid
    return dict(loss=float(loss), eal_g=eal_g, eal_s=eal_s, nvalid=nvalid, kn=kn,
                a_g=a_g, a_s=a_s, xstar=xstar)


def loss_backward(target, draft, mask=None, mode: int = MODE_BOTH, T: float = 1.0,
                  w_greedy: float = 1.0, w_sampling: float = 1.0, dloss: float = 1.0,
                  n_windows_total=None, xstar=None) -> np.ndarray:
    """dloss * dL/dz_q for every draft logit, [N][K][V] float64.

    The target is frozen (Sec. 3.2, 3.3): only the draft logits get a gradient.
    Chain rule through the window sum and the per-position acceptances:

    dL/dz_q[n,j,u] = -(dloss/|W|) * ( w_g dE^g_n/da^g_{n,j} * da^g_{n,j}/dz_u
                                     + w_s dE^s_n/da^s_{n,j} * da^s_{n,j}/dz_u )

    with the softmax Jacobian dq~_v/dz_u = (1/T) q~_v (delta_uv - q~_u):
      a^g = q(x*)            -> da^g/dz_u = a^g (delta_{u,x*} - q(u))           (T = 1)
      a^s = sum_v min(p~,q~) -> da^s/dz_u = sum_v c_v dq~_v/dz_u
                                           = (1/T) q~_u (c_u - sum_v c_v q~_v),
    where c_v = 1 if q~_v < p~_v else 0.  TV is piecewise linear in q~ (Sec. 3.3);
    at a tie q~_v = p~_v the min is taken to follow the frozen p~, so c_v = 0 there.
    The comparison is made on log-probabilities.
    """
    zq = as_f64(draft)
    N, K, V = zq.shape
    fw = loss_forward(target, draft, mask, mode, T, w_greedy, w_sampling, n_windows_total, xstar)
    nvalid, kn = fw["nvalid"], fw["kn"]
    grad = np.zeros((N, K, V), dtype=np.float64)
    if nvalid == 0:
        return grad
    wg, ws = _weights(mode, w_greedy, w_sampling)
    scale = -dloss / nvalid
    if mode & MODE_GREEDY:
        dEg = expected_length_partials(fw["a_g"], kn)                 # [N,K]
        q1 = np.exp(log_softmax(zq, 1.0))
        onehot = np.zeros_like(q1)
        np.put_along_axis(onehot, fw["xstar"][..., None], 1.0, axis=-1)
        da_g = fw["a_g"][..., None] * (onehot - q1)                   # [N,K,V]
        grad += scale * wg * dEg[..., None] * da_g
    if mode & MODE_SAMPLING:
        dEs = expected_length_partials(fw["a_s"], kn)
        lp = log_softmax(as_f64(target), T)
        lq = log_softmax(zq, T)
        qt = np.exp(lq)
        c = (lq < lp).astype(np.float64)
        qlt = np.sum(c * qt, axis=-1, keepdims=True)
        da_s = (1.0 / T) * qt * (c - qlt)
        grad += scale * ws * dEs[..., None] * da_s
    return grad
