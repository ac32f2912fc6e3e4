"""Pins of the sliding-window sequence loss (oracle/sequence.py), CPU only."""

from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle.sequence import gather_windows, seq_loss_backward, seq_loss_forward
from tests.spec_sim import expected_accepted_length_greedy, expected_accepted_length_sampling


def _rational_dist(rng, V, denom=10):
    w = rng.integers(1, denom, size=V)
    s = int(w.sum())
    return [Fraction(int(x), s) for x in w]


def test_every_window_equals_brute_force_verification():
    """Each window starting at t covers positions t..t+K-1 of the sequence (truncated at its end)
    and its E[L] equals enumerated speculative verification over exactly those positions."""
    rng = np.random.default_rng(0)
    Tn, K, V = 5, 3, 3
    p = [_rational_dist(rng, V) for _ in range(Tn)]
    q = [_rational_dist(rng, V) for _ in range(Tn)]
    zp = np.log(np.array([[[float(x) for x in r] for r in p]]))
    zq = np.log(np.array([[[float(x) for x in r] for r in q]]))
    fw = seq_loss_forward(zp, zq, None, K, oracle.MODE_BOTH, 1.0, 1.0, 1.0)
    pstar = [max(range(V), key=lambda v: (r[v], -v)) for r in p]
    total = 0.0
    for t in range(Tn):
        span = range(t, min(t + K, Tn))
        es = expected_accepted_length_sampling([p[i] for i in span], [q[i] for i in span])
        eg = expected_accepted_length_greedy([pstar[i] for i in span], [q[i] for i in span])
        assert abs(fw["eal_s"][t] - float(es)) < 1e-13
        assert abs(fw["eal_g"][t] - float(eg)) < 1e-13
        total += float(es) + float(eg)
    assert fw["nvalid"] == Tn
    assert abs(fw["loss"] + total / Tn) < 1e-13


def test_invalid_positions_end_windows_and_start_none():
    rng = np.random.default_rng(1)
    B, Tn, K, V = 2, 6, 3, 4
    zp = rng.normal(size=(B, Tn, V))
    zq = rng.normal(size=(B, Tn, V))
    mask = np.ones((B, Tn), dtype=np.uint8)
    mask[0, 2] = 0
    mask[1, 4:] = 0           # padding at the end of sequence 1
    fw = seq_loss_forward(zp, zq, mask, K)
    kn = fw["kn"].reshape(B, Tn)
    assert list(kn[0]) == [2, 1, 0, 3, 2, 1]
    assert list(kn[1]) == [3, 3, 2, 1, 0, 0]
    assert fw["nvalid"] == 9


def test_window_size_one_is_the_mean_acceptance():
    rng = np.random.default_rng(2)
    zp = rng.normal(size=(2, 7, 9))
    zq = rng.normal(size=(2, 7, 9))
    fw = seq_loss_forward(zp, zq, None, 1, oracle.MODE_SAMPLING, 0.8)
    a = oracle.acceptance_sampling(zp, zq, 0.8)
    assert abs(fw["loss"] + a.mean()) < 1e-14


@pytest.mark.parametrize("mode,T", [(oracle.MODE_BOTH, 1.0), (oracle.MODE_SAMPLING, 0.7), (oracle.MODE_GREEDY, 1.0)])
def test_sequence_gradient_by_finite_differences(mode, T):
    """Positions shared by up to K windows: the summed gradient against central differences."""
    rng = np.random.default_rng(3)
    B, Tn, K, V = 1, 5, 3, 6
    while True:
        zp = rng.normal(0, 1.5, size=(B, Tn, V))
        zq = zp + rng.normal(0, 1.0, size=(B, Tn, V))
        pt = np.exp(oracle.log_softmax(zp, T)); qt = np.exp(oracle.log_softmax(zq, T))
        if np.min(np.abs(pt - qt)) > 1e-3:
            break
    mask = np.ones((B, Tn), dtype=np.uint8)
    mask[0, 3] = 0
    kw = dict(mode=mode, T=T, w_greedy=0.4, w_sampling=0.6)
    g = seq_loss_backward(zp, zq, mask, K, dloss=3.0, **kw)
    h = 1e-6
    for idx in np.ndindex(B, Tn, V):
        a = zq.copy(); a[idx] += h
        b = zq.copy(); b[idx] -= h
        fd = 3.0 * (seq_loss_forward(zp, a, mask, K, **kw)["loss"] - seq_loss_forward(zp, b, mask, K, **kw)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-7, (idx, fd, g[idx])


def test_gathered_windows_point_back_to_their_positions():
    zp = np.arange(2 * 4 * 3, dtype=np.float64).reshape(2, 4, 3)
    wp, wq, wm, src = gather_windows(zp, zp, None, 3)
    assert src[5].tolist() == [5, 6, 7]          # sequence 1, t = 1
    assert src[7].tolist() == [7, -1, -1]         # last position of sequence 1
    assert wm[7].tolist() == [1, 0, 0]
    np.testing.assert_array_equal(wp[5, 1], zp[1, 2])


def test_slice_around_a_position_gives_its_gradient():
    """The full-size GPU tests check sampled positions against the oracle run on the positions
    t-K+1 .. t+K-1 only, with |W| of the whole batch: every window containing t lies inside."""
    rng = np.random.default_rng(4)
    B, Tn, K, V = 2, 12, 3, 5
    zp = rng.normal(size=(B, Tn, V))
    zq = zp + rng.normal(size=(B, Tn, V))
    mask = np.ones((B, Tn), dtype=np.uint8)
    mask[1, 7] = 0
    full = seq_loss_backward(zp, zq, mask, K, oracle.MODE_BOTH, 0.9, 0.3, 0.7, 2.0)
    fw = seq_loss_forward(zp, zq, mask, K, oracle.MODE_BOTH, 0.9, 0.3, 0.7)
    for b, t in [(0, 0), (0, 5), (1, 6), (1, 8), (1, 11)]:
        lo, hi = max(0, t - K + 1), min(Tn, t + K)
        g = seq_loss_backward(zp[b:b + 1, lo:hi], zq[b:b + 1, lo:hi], mask[b:b + 1, lo:hi], K,
                              oracle.MODE_BOTH, 0.9, 0.3, 0.7, 2.0, n_windows_total=fw["nvalid"])
        np.testing.assert_allclose(g[0, t - lo], full[b, t], rtol=0, atol=1e-15)


def test_full_windows_reading_keeps_only_complete_windows():
    """With full_windows, an unmasked sequence of length T has the windows starting at
    0 .. T-K only, each equal to brute-force verification over its K positions; a hole removes
    every window that would cover it."""
    rng = np.random.default_rng(5)
    Tn, K, V = 6, 3, 3
    p = [_rational_dist(rng, V) for _ in range(Tn)]
    q = [_rational_dist(rng, V) for _ in range(Tn)]
    zp = np.log(np.array([[[float(x) for x in r] for r in p]]))
    zq = np.log(np.array([[[float(x) for x in r] for r in q]]))
    fw = seq_loss_forward(zp, zq, None, K, oracle.MODE_SAMPLING, full_windows=True)
    assert fw["nvalid"] == Tn - K + 1
    total = 0.0
    for t in range(Tn):
        if t <= Tn - K:
            es = float(expected_accepted_length_sampling(p[t:t + K], q[t:t + K]))
            assert abs(fw["eal_s"][t] - es) < 1e-13
            total += es
        else:
            assert fw["eal_s"][t] == 0.0
    assert abs(fw["loss"] + total / (Tn - K + 1)) < 1e-13
    mask = np.ones((1, Tn), dtype=np.uint8)
    mask[0, 3] = 0
    fw = seq_loss_forward(zp, zq, mask, K, oracle.MODE_SAMPLING, full_windows=True)
    assert list(fw["kn"]) == [3, 0, 0, 0, 0, 0]
    g = seq_loss_backward(zp, zq, mask, K, oracle.MODE_SAMPLING, full_windows=True)
    assert np.all(g[0, 3:] == 0) and np.any(g[0, :3] != 0)


def test_sequence_tv_term_by_finite_differences():
    rng = np.random.default_rng(8)
    B, Tn, K, V = 1, 5, 3, 5
    while True:
        zp = rng.normal(0, 1.5, size=(B, Tn, V))
        zq = zp + rng.normal(0, 1.0, size=(B, Tn, V))
        pt = np.exp(oracle.log_softmax(zp, 0.9)); qt = np.exp(oracle.log_softmax(zq, 0.9))
        if np.min(np.abs(pt - qt)) > 1e-3:
            break
    mask = np.ones((B, Tn), dtype=np.uint8)
    mask[0, 3] = 0
    kw = dict(mode=oracle.MODE_KL | oracle.MODE_TV, T=0.9, w_greedy=0.0, w_sampling=0.0, w_kl=1.0, w_tv=0.1)
    g = oracle.seq_objective_backward(zp, zq, mask, K, dloss=2.0, **kw)
    h = 1e-6
    for idx in np.ndindex(B, Tn, V):
        a = zq.copy(); a[idx] += h
        b = zq.copy(); b[idx] -= h
        fd = 2.0 * (oracle.seq_objective_forward(zp, a, mask, K, **kw)["loss"]
                    - oracle.seq_objective_forward(zp, b, mask, K, **kw)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-7, (idx, fd, g[idx])


def test_sequence_token_ids_equal_a_peaked_target():
    rng = np.random.default_rng(9)
    B, Tn, K, V = 2, 6, 3, 8
    zq = rng.normal(0, 2, size=(B, Tn, V))
    ids = rng.integers(0, V, size=(B, Tn))
    zp = np.zeros((B, Tn, V))
    np.put_along_axis(zp, ids[..., None], 60.0, axis=-1)
    mask = np.ones((B, Tn), dtype=np.uint8)
    mask[1, 4] = 0
    a = seq_loss_forward(None, zq, mask, K, oracle.MODE_GREEDY, xstar=ids)
    b = seq_loss_forward(zp, zq, mask, K, oracle.MODE_GREEDY)
    assert abs(a["loss"] - b["loss"]) < 1e-15
    np.testing.assert_array_equal(seq_loss_backward(None, zq, mask, K, oracle.MODE_GREEDY, dloss=2.0, xstar=ids),
                                  seq_loss_backward(zp, zq, mask, K, oracle.MODE_GREEDY, dloss=2.0))
