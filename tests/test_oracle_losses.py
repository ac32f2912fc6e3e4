"""Pins of the oracle's loss arithmetic to what the paper and mathematics fix (CPU only)."""

import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle import MODE_BOTH, MODE_GREEDY, MODE_SAMPLING
from tests.spec_sim import (acceptance_by_rejection, expected_accepted_length_greedy,
                            expected_accepted_length_sampling)

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rational_dist(rng, V, denom=12):
    w = rng.integers(1, denom, size=V)
    s = int(w.sum())
    return [Fraction(int(x), s) for x in w]


def _scaled(dist, T_inv):
    """p~ proportional to p^(1/T) for integer 1/T, exactly."""
    w = [x ** T_inv for x in dist]
    s = sum(w)
    return [x / s for x in w]


# ---------------------------------------------------------------- log-softmax

def test_log_softmax_closed_forms():
    V = 37
    z = np.full((1, V), 3.25)
    np.testing.assert_allclose(oracle.log_softmax(z, 0.7), -math.log(V), rtol=0, atol=1e-15)
    # two tokens: log p(0) = -log(1 + e^{a/T})
    for a, T in [(2.0, 1.0), (-5.0, 0.5), (30.0, 2.0)]:
        lp = oracle.log_softmax(np.array([[0.0, a]]), T)
        assert abs(lp[0, 0] + math.log1p(math.exp(a / T))) < 1e-13
    # -inf entries get probability zero
    lp = oracle.log_softmax(np.array([[0.0, -np.inf, 0.0]]), 1.0)
    assert lp[0, 1] == -np.inf and abs(lp[0, 0] + math.log(2)) < 1e-15


def test_temperature_matches_power_of_probabilities():
    """Sec. 2.3: p~ is proportional to exp(log p / T), i.e. p^(1/T) normalised."""
    rng = np.random.default_rng(1)
    p = rng.dirichlet(np.ones(11))
    for T in [0.5, 1.0, 1.5]:
        expect = p ** (1 / T) / np.sum(p ** (1 / T))
        got = np.exp(oracle.log_softmax(np.log(p)[None] + 4.0, T))[0]
        np.testing.assert_allclose(got, expect, rtol=1e-12)


# ---------------------------------------------------------------- acceptances

def test_sampling_acceptance_equals_rejection_expectation_exactly():
    """Eq. acc_sample: E_{y~q~}[min(1,p~/q~)] = sum min(p~,q~), checked by enumeration."""
    rng = np.random.default_rng(2)
    for V in [2, 3, 5]:
        for T_inv in [1, 2]:
            p = _scaled(_rational_dist(rng, V), T_inv)
            q = _scaled(_rational_dist(rng, V), T_inv)
            exact = acceptance_by_rejection(p, q)
            # logits whose T-scaled softmax is p~ / q~: z = T log p~
            T = 1.0 / T_inv
            zp = T * np.log(np.array([[float(x) for x in p]]))
            zq = T * np.log(np.array([[float(x) for x in q]]))
            got = oracle.acceptance_sampling(zp, zq, T)[0]
            assert abs(got - float(exact)) < 1e-13
            # 1 - TV with TV = 1/2 sum |p~ - q~|
            tv = sum(abs(a - b) for a, b in zip(p, q)) / 2
            assert exact == 1 - tv


def test_sampling_acceptance_monte_carlo():
    """Rejection sampling with 1e6 draws reproduces a^sample within 5 sigma."""
    rng = np.random.default_rng(3)
    V = 60
    zp = rng.normal(0, 2, size=(1, V))
    zq = zp + rng.normal(0, 1, size=(1, V))
    T = 0.8
    a = oracle.acceptance_sampling(zp, zq, T)[0]
    pt = np.exp(oracle.log_softmax(zp, T))[0]
    qt = np.exp(oracle.log_softmax(zq, T))[0]
    n = 1_000_000
    y = rng.choice(V, size=n, p=qt / qt.sum())
    u = rng.random(n)
    acc = np.mean(u < pt[y] / qt[y])
    sigma = math.sqrt(a * (1 - a) / n)
    assert abs(acc - a) < 5 * sigma


def test_greedy_acceptance_is_draft_mass_on_target_argmax():
    rng = np.random.default_rng(4)
    zp = rng.normal(size=(3, 9))
    zq = rng.normal(size=(3, 9))
    a, xs = oracle.acceptance_greedy(zp, zq)
    for r in range(3):
        q = np.exp(zq[r]) / np.exp(zq[r]).sum()
        assert xs[r] == int(np.argmax(zp[r]))
        assert abs(a[r] - q[xs[r]]) < 1e-15


def test_argmax_ties_take_lowest_index():
    z = np.array([[1.0, 5.0, 2.0, 5.0, 5.0]])
    assert oracle.argmax_lowest(z)[0] == 1


# ---------------------------------------------------------------- window sum

def _eval_terms(terms, a):
    out = Fraction(0)
    for coef, pos, neg in terms:
        t = Fraction(coef)
        for j in pos:
            t *= a[j]
        for j in neg:
            t *= (1 - a[j])
        out += t
    return out


def test_gamma3_worked_example_golden():
    """The paper's gamma = 3 example: the full form equals the compact form, and the oracle."""
    with open(os.path.join(GOLDEN, "eal_gamma3_example.json")) as f:
        g = json.load(f)
    rng = np.random.default_rng(5)
    for _ in range(50):
        a = [Fraction(int(rng.integers(0, 97)), 96) for _ in range(g["gamma"])]
        full = _eval_terms(g["full_form"], a)
        compact = _eval_terms(g["compact_form"], a)
        assert full == compact
        got = oracle.expected_length(np.array([[float(x) for x in a]]), np.array([3]))[0]
        assert abs(got - float(full)) < 1e-15


def test_tail_sum_equals_distribution_mean():
    """Sec. 3.2: sum_l l P(L=l) from the explicit distribution of L equals Eq. eal_compact."""
    rng = np.random.default_rng(6)
    for K in range(1, 9):
        a = rng.random((20, K))
        got = oracle.expected_length(a, np.full(20, K))
        for n in range(20):
            mean = 0.0
            for ell in range(1, K):
                mean += ell * np.prod(a[n, :ell]) * (1 - a[n, ell])
            mean += K * np.prod(a[n, :K])
            assert abs(got[n] - mean) < 1e-14
            probs = [1 - a[n, 0]] + [np.prod(a[n, :ell]) * (1 - a[n, ell]) for ell in range(1, K)] \
                + [np.prod(a[n, :K])]
            assert abs(sum(probs) - 1.0) < 1e-14


def test_window_special_cases():
    assert oracle.expected_length(np.ones((1, 6)), np.array([6]))[0] == 6.0
    assert oracle.expected_length(np.zeros((1, 6)), np.array([6]))[0] == 0.0
    a = np.array([[0.3, 0.9, 0.9]])
    assert oracle.expected_length(a, np.array([1]))[0] == 0.3          # K = 1: E = a
    assert oracle.expected_length(a, np.array([0]))[0] == 0.0


def test_partials_by_finite_differences():
    rng = np.random.default_rng(7)
    for K in [1, 2, 5, 8]:
        a = rng.random((4, K))
        kn = rng.integers(0, K + 1, size=4)
        d = oracle.expected_length_partials(a, kn)
        h = 1e-6
        for n in range(4):
            for j in range(K):
                ap = a.copy(); ap[n, j] += h
                am = a.copy(); am[n, j] -= h
                fd = (oracle.expected_length(ap, kn)[n] - oracle.expected_length(am, kn)[n]) / (2 * h)
                assert abs(fd - d[n, j]) < 1e-8


# ---------------------------------------------------------------- losses vs brute force

@pytest.mark.parametrize("gamma", [1, 2, 3])
def test_wtv_window_equals_brute_force_verification(gamma):
    """E[L] of the WTV window (Eq. eal_tv) equals enumerated sampling verification, V = 3."""
    rng = np.random.default_rng(10 + gamma)
    for T_inv in [1, 2]:
        T = 1.0 / T_inv
        p = [_rational_dist(rng, 3) for _ in range(gamma)]
        q = [_rational_dist(rng, 3) for _ in range(gamma)]
        pt = [_scaled(x, T_inv) for x in p]
        qt = [_scaled(x, T_inv) for x in q]
        exact = expected_accepted_length_sampling(pt, qt)
        zp = np.log(np.array([[[float(x) for x in r] for r in p]]))
        zq = np.log(np.array([[[float(x) for x in r] for r in q]]))
        fw = oracle.loss_forward(zp, zq, None, MODE_SAMPLING, T)
        assert abs(fw["eal_s"][0] - float(exact)) < 1e-13
        assert abs(fw["loss"] + float(exact)) < 1e-13


@pytest.mark.parametrize("gamma", [1, 2, 3])
def test_eal_window_equals_brute_force_verification(gamma):
    """E[L] of the EAL window (Eq. loss_eal) equals enumerated greedy verification, V = 3."""
    rng = np.random.default_rng(20 + gamma)
    p = [_rational_dist(rng, 3, 50) for _ in range(gamma)]
    q = [_rational_dist(rng, 3) for _ in range(gamma)]
    pstar = [max(range(3), key=lambda v: (r[v], -v)) for r in p]
    exact = expected_accepted_length_greedy(pstar, q)
    zp = np.log(np.array([[[float(x) for x in r] for r in p]]))
    zq = np.log(np.array([[[float(x) for x in r] for r in q]]))
    fw = oracle.loss_forward(zp, zq, None, MODE_GREEDY, 1.0)
    assert abs(fw["eal_g"][0] - float(exact)) < 1e-13


def test_loss_normalises_by_valid_windows_and_truncates_at_mask():
    rng = np.random.default_rng(30)
    N, K, V = 5, 4, 6
    zp = rng.normal(size=(N, K, V))
    zq = rng.normal(size=(N, K, V))
    mask = np.ones((N, K), dtype=np.uint8)
    mask[1, 0] = 0           # window 1 not in W
    mask[2, 2] = 0           # window 2 truncated after 2 depths
    mask[3, 3] = 0
    fw = oracle.loss_forward(zp, zq, mask, MODE_BOTH, 1.0, 0.25, 0.75)
    assert fw["nvalid"] == 4
    assert list(fw["kn"]) == [4, 0, 2, 3, 4]
    a_g, _ = oracle.acceptance_greedy(zp, zq)
    a_s = oracle.acceptance_sampling(zp, zq, 1.0)
    tot = 0.0
    for n, g in enumerate([4, 0, 2, 3, 4]):
        for k in range(1, g + 1):
            tot += 0.25 * np.prod(a_g[n, :k]) + 0.75 * np.prod(a_s[n, :k])
    assert abs(fw["loss"] + tot / 4) < 1e-14


def test_no_valid_window_gives_zero_loss_and_gradient():
    rng = np.random.default_rng(31)
    zp = rng.normal(size=(3, 2, 5)); zq = rng.normal(size=(3, 2, 5))
    mask = np.zeros((3, 2), dtype=np.uint8); mask[:, 1] = 1
    assert oracle.loss_forward(zp, zq, mask)["loss"] == 0.0
    assert not np.any(oracle.loss_backward(zp, zq, mask))


def test_identical_rows_give_full_acceptance_and_zero_wtv_gradient():
    rng = np.random.default_rng(32)
    z = rng.normal(0, 3, size=(2, 5, 40))
    for T in [0.5, 1.0, 1.5]:
        fw = oracle.loss_forward(z, z, None, MODE_SAMPLING, T)
        np.testing.assert_allclose(fw["a_s"], 1.0, rtol=0, atol=1e-14)
        np.testing.assert_allclose(fw["eal_s"], 5.0, rtol=0, atol=1e-13)
        g = oracle.loss_backward(z, z, None, MODE_SAMPLING, T)
        assert not np.any(g)


def test_disjoint_supports_give_zero_acceptance_and_gradient():
    V = 10
    zp = np.full((1, 3, V), -np.inf); zq = np.full((1, 3, V), -np.inf)
    zp[..., :5] = np.random.default_rng(33).normal(size=(1, 3, 5))
    zq[..., 5:] = np.random.default_rng(34).normal(size=(1, 3, 5))
    fw = oracle.loss_forward(zp, zq, None, MODE_SAMPLING, 1.0)
    assert np.all(fw["a_s"] == 0.0) and fw["eal_s"][0] == 0.0
    assert not np.any(oracle.loss_backward(zp, zq, None, MODE_SAMPLING, 1.0))


def test_peaked_draft_on_target_argmax_gives_full_greedy_length():
    rng = np.random.default_rng(35)
    zp = rng.normal(size=(2, 6, 30))
    zq = rng.normal(size=(2, 6, 30))
    xs = np.argmax(zp, axis=-1)
    np.put_along_axis(zq, xs[..., None], 100.0, axis=-1)
    fw = oracle.loss_forward(zp, zq, None, MODE_GREEDY)
    np.testing.assert_allclose(fw["eal_g"], 6.0, rtol=0, atol=1e-12)


def test_shift_invariance_of_loss_and_gradient_sum():
    rng = np.random.default_rng(36)
    zp = rng.normal(size=(3, 4, 12)); zq = rng.normal(size=(3, 4, 12))
    base = oracle.loss_forward(zp, zq, None, MODE_BOTH, 1.3, 0.5, 0.5)["loss"]
    cp = rng.normal(size=(3, 4, 1)) * 10; cq = rng.normal(size=(3, 4, 1)) * 10
    moved = oracle.loss_forward(zp + cp, zq + cq, None, MODE_BOTH, 1.3, 0.5, 0.5)["loss"]
    assert abs(base - moved) < 1e-13
    g = oracle.loss_backward(zp, zq, None, MODE_BOTH, 1.3, 0.5, 0.5)
    np.testing.assert_allclose(g.sum(-1), 0.0, atol=1e-15)


def _well_separated(rng, N, K, V, T):
    while True:
        zp = rng.normal(0, 1.5, size=(N, K, V))
        zq = zp + rng.normal(0, 1.0, size=(N, K, V))
        pt = np.exp(oracle.log_softmax(zp, T)); qt = np.exp(oracle.log_softmax(zq, T))
        if np.min(np.abs(pt - qt)) > 1e-3:
            return zp, zq


@pytest.mark.parametrize("K", [1, 3, 5])
@pytest.mark.parametrize("mode,T", [(MODE_GREEDY, 1.0), (MODE_SAMPLING, 0.7),
                                    (MODE_SAMPLING, 1.0), (MODE_BOTH, 1.4)])
def test_gradient_matches_central_differences(K, mode, T):
    """The analytic draft-logit gradient against central differences of the loss, V = 8."""
    rng = np.random.default_rng(100 + K + 10 * mode)
    N, V = 2, 8
    zp, zq = _well_separated(rng, N, K, V, T)
    mask = np.ones((N, K), dtype=np.uint8)
    if K > 1:
        mask[1, K - 1] = 0
    kw = dict(mode=mode, T=T, w_greedy=0.3, w_sampling=0.7)
    g = oracle.loss_backward(zp, zq, mask, dloss=2.0, **kw)
    h = 1e-6
    for idx in np.ndindex(N, K, V):
        zplus = zq.copy(); zplus[idx] += h
        zminus = zq.copy(); zminus[idx] -= h
        fd = 2.0 * (oracle.loss_forward(zp, zplus, mask, **kw)["loss"]
                    - oracle.loss_forward(zp, zminus, mask, **kw)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-7, (idx, fd, g[idx])


# ------------------------------------------------------------------ target token ids

def test_token_ids_equal_a_target_peaked_on_them():
    """x* given as ids (Sec. 3.2: the ground-truth token of greedy target-generated data) is
    the same as target logits whose argmax is that id: a +60 peak on zero logits."""
    rng = np.random.default_rng(40)
    N, K, V = 3, 4, 11
    zq = rng.normal(0, 2, size=(N, K, V))
    ids = rng.integers(0, V, size=(N, K))
    zp = np.zeros((N, K, V))
    np.put_along_axis(zp, ids[..., None], 60.0, axis=-1)
    mask = np.ones((N, K), dtype=np.uint8)
    mask[1, 2] = 0
    a = oracle.loss_forward(None, zq, mask, oracle.MODE_GREEDY, 1.0, 0.7, 0.0, xstar=ids)
    b = oracle.loss_forward(zp, zq, mask, oracle.MODE_GREEDY, 1.0, 0.7, 0.0)
    assert abs(a["loss"] - b["loss"]) < 1e-15 and np.array_equal(a["xstar"], ids)
    ga = oracle.loss_backward(None, zq, mask, oracle.MODE_GREEDY, 1.0, 0.7, 0.0, 2.0, xstar=ids)
    gb = oracle.loss_backward(zp, zq, mask, oracle.MODE_GREEDY, 1.0, 0.7, 0.0, 2.0)
    np.testing.assert_array_equal(ga, gb)
    with pytest.raises(ValueError):
        oracle.loss_forward(None, zq, mask, oracle.MODE_BOTH, 1.0, xstar=ids)


def test_token_id_gradient_by_finite_differences():
    rng = np.random.default_rng(41)
    N, K, V = 2, 3, 7
    zq = rng.normal(0, 1.5, size=(N, K, V))
    ids = rng.integers(0, V, size=(N, K))
    g = oracle.loss_backward(None, zq, None, oracle.MODE_GREEDY, 1.0, 1.0, 0.0, 3.0, xstar=ids)
    h = 1e-6
    for idx in np.ndindex(N, K, V):
        a = zq.copy(); a[idx] += h
        b = zq.copy(); b[idx] -= h
        fd = 3.0 * (oracle.loss_forward(None, a, None, 1, 1.0, 1.0, 0.0, xstar=ids)["loss"]
                    - oracle.loss_forward(None, b, None, 1, 1.0, 1.0, 0.0, xstar=ids)["loss"]) / (2 * h)
        assert abs(fd - g[idx]) < 1e-8
