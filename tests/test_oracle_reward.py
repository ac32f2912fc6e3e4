"""Pins of the oracle's GRPO reward, advantages and Philox generator (CPU only)."""

import ctypes
import ctypes.util
import glob
import math
import os
from itertools import product

import numpy as np
import pytest

import oracle
from oracle.reward import REWARD_GREEDY, REWARD_SAMPLING


# ---------------------------------------------------------------- simulated accepted length

def test_tau_counts_matches_before_first_mismatch():
    """Sec. 3.4: tau counts consecutive correct predictions from the window start until the
    first mismatch; checked against a left-to-right scan over every 0/1 pattern, gamma <= 8."""
    for K in range(1, 9):
        pats = np.array(list(product((0, 1), repeat=K)), dtype=np.int64)
        tau = oracle.simulated_accept_length(pats)
        for pat, t in zip(pats, tau):
            scan = 0
            while scan < K and pat[scan] == 1:
                scan += 1
            assert t == scan


def test_greedy_reward_identical_draft_is_full_window():
    rng = np.random.default_rng(0)
    z = rng.normal(size=(6, 8, 50))
    out = oracle.accept_reward(z, z, mode=REWARD_GREEDY, windows_per_rollout=3, rollouts_per_group=2)
    assert np.all(out["tau"] == 8)
    np.testing.assert_array_equal(out["advantage"], 0.0)


def test_greedy_reward_leading_run():
    rng = np.random.default_rng(1)
    zp = rng.normal(size=(4, 5, 20))
    zq = rng.normal(size=(4, 5, 20))
    xs = np.argmax(zp, axis=-1)
    # plant matches: window n matches on its first n+1 depths then mismatches
    for n in range(4):
        for k in range(5):
            tok = xs[n, k] if k <= n else (xs[n, k] + 1) % 20
            zq[n, k, tok] = 50.0
    out = oracle.accept_reward(zp, zq, mode=REWARD_GREEDY)
    assert list(out["tau"]) == [1, 2, 3, 4]


def test_debiased_reward_cancels_shared_difficulty():
    """Eq. debiased_reward: a reference draft identical to the current one gives R = 0."""
    rng = np.random.default_rng(2)
    zp = rng.normal(size=(8, 4, 30))
    zq = zp + rng.normal(size=(8, 4, 30))
    out = oracle.accept_reward(zp, zq, ref_draft=zq.copy(), mode=REWARD_GREEDY)
    assert np.all(out["R"] == 0.0)
    out = oracle.accept_reward(zp, zq, ref_draft=zq.copy(), mode=REWARD_SAMPLING, T=1.0, seed=3)
    assert np.all(out["R"] == 0.0)


def test_sampling_reward_mean_matches_rejection_probabilities():
    """Averaged over many counter-based draws, tau under sampling verification has mean
    sum_k prod_{j<k} min(1, p~(S_j)/q~(S_j)) (Sec. 2.3 acceptance rule, Sec. 3.4 tau)."""
    rng = np.random.default_rng(4)
    K, V, T = 4, 25, 0.9
    zp = rng.normal(0, 1, size=(1, K, V))
    zq = zp + rng.normal(0, 0.7, size=(1, K, V))
    n_rep = 20000
    zp_rep = np.repeat(zp, n_rep, axis=0)
    zq_rep = np.repeat(zq, n_rep, axis=0)
    out = oracle.accept_reward(zp_rep, zq_rep, mode=REWARD_SAMPLING, T=T, seed=11,
                               row_offset=123456789)
    thr = out["thr"][0]
    expect = sum(np.prod(thr[:k]) for k in range(1, K + 1))
    tau = out["tau"].astype(np.float64)
    sigma = tau.std() / math.sqrt(n_rep)
    assert abs(tau.mean() - expect) < 5 * sigma + 1e-12


# ---------------------------------------------------------------- advantages

def test_advantages_are_standardised_within_groups():
    rng = np.random.default_rng(5)
    x = rng.normal(3.0, 2.0, size=64)
    A = oracle.group_advantages(x, 16, clip=1e9)
    for g in range(4):
        grp = x[16 * g:16 * (g + 1)]
        sd = grp.std()
        a = A[16 * g:16 * (g + 1)]
        assert abs(a.mean()) < 1e-14
        assert abs(a.std() - sd / (sd + 1e-6)) < 1e-12
    # invariant to a constant added to every reward of a group
    np.testing.assert_allclose(oracle.group_advantages(x + 7.5, 16, 1e9), A, atol=1e-12)
    # constant group: zero advantage (eps keeps the division finite)
    np.testing.assert_array_equal(oracle.group_advantages(np.full(16, 2.5), 16, 5.0), 0.0)


def test_advantages_are_clipped():
    x = np.array([0.0] * 15 + [100.0])
    A = oracle.group_advantages(x, 16, clip=2.0)
    assert A[-1] == 2.0 and np.all(A[:-1] < 0)
    assert abs(A[-1]) <= 2.0


def test_rollout_length_is_window_mean():
    R = np.arange(12, dtype=np.float64)
    np.testing.assert_array_equal(oracle.rollout_lengths(R, 4), [1.5, 5.5, 9.5])


# ---------------------------------------------------------------- Philox4x32-10

def _curand():
    cands = [os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "lib64", "libcurand.so")]
    cands += glob.glob("/usr/local/cuda*/lib64/libcurand.so*")
    found = ctypes.util.find_library("curand")
    if found:
        cands.append(found)
    for c in cands:
        try:
            return ctypes.CDLL(c)
        except OSError:
            continue
    pytest.skip("libcurand not found")


def _curand_philox_block(lib, seed, block):
    """4 raw words of cuRAND's host Philox4x32-10 generator at output block ``block``.

    The host generator emits block b from counter (b >> 16 as a 64-bit number in
    words 0-1, b & 0xffff in word 2, 0) under key (seed_lo, seed_hi); the offset
    argument counts 32-bit outputs.
    """
    g = ctypes.c_void_p()
    assert lib.curandCreateGeneratorHost(ctypes.byref(g), 161) == 0  # PHILOX4_32_10
    try:
        assert lib.curandSetPseudoRandomGeneratorSeed(g, ctypes.c_ulonglong(seed)) == 0
        assert lib.curandSetGeneratorOffset(g, ctypes.c_ulonglong(4 * block)) == 0
        out = np.zeros(4, dtype=np.uint32)
        assert lib.curandGenerate(g, out.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(4)) == 0
    finally:
        lib.curandDestroyGenerator(g)
    return out


def test_philox_matches_curand_host_generator():
    """The oracle's Philox against an independent implementation (cuRAND's host generator)."""
    lib = _curand()
    rng = np.random.default_rng(6)
    cases = [(0, 0, 0), (0, 1, 0), (0, 0, 1), (5, 77, 3), (2**63 + 12345, 2**33 + 9, 7)]
    cases += [(int(rng.integers(0, 2**63)), int(rng.integers(0, 2**40)), int(rng.integers(0, 8)))
              for _ in range(8)]
    for seed, n, k in cases:
        ref = _curand_philox_block(lib, seed, (n << 16) + k)
        got = oracle.philox4x32_10(n & 0xFFFFFFFF, n >> 32, k, 0, seed & 0xFFFFFFFF, seed >> 32)
        assert [int(x) for x in got] == [int(x) for x in ref], (seed, n, k)


def test_uniform_is_exact_odd_multiple_in_open_interval():
    u = oracle.uniform01(0, np.arange(100000), np.arange(100000) % 8)
    assert np.all(u > 0) and np.all(u < 1)
    m = u * 2**24
    assert np.all(m == np.round(m)) and np.all(m % 2 == 1)
    assert np.all(u.astype(np.float32).astype(np.float64) == u)


def test_uniform_chi_square_and_serial_correlation():
    n = 1 << 20
    u = oracle.uniform01(42, np.arange(n) // 8, np.arange(n) % 8)
    bins = 1 << 12
    counts = np.bincount((u * bins).astype(np.int64), minlength=bins)
    e = n / bins
    chi2 = np.sum((counts - e) ** 2 / e)
    # chi-square with 4095 dof: mean 4095, sd ~90.5; accept within 6 sd
    assert abs(chi2 - (bins - 1)) < 6 * math.sqrt(2 * (bins - 1))
    r = np.corrcoef(u[:-1], u[1:])[0, 1]
    assert abs(r) < 6 / math.sqrt(n)


# ------------------------------------------------------------------ sampled draft tokens

def test_gumbel_max_draws_follow_the_scaled_draft_distribution():
    """S ~ q~ (Sec. 2.3): over 40000 windows with the same logits, the frequencies of the
    Gumbel-max tokens match q~ within 5 binomial standard deviations per token."""
    import oracle
    V, T, n = 6, 0.8, 40000
    z = np.array([1.0, 0.2, -0.5, 2.0, 0.0, 1.5])
    draft = np.broadcast_to(z, (n, 1, V))
    S = oracle.sampled_trajectory(draft, T, seed=123)[:, 0]
    q = np.exp(oracle.log_softmax(z, T))
    freq = np.bincount(S, minlength=V) / n
    assert np.all(np.abs(freq - q) <= 5 * np.sqrt(q * (1 - q) / n)), (freq, q)


def test_sampled_draft_reward_has_the_wtv_expected_length():
    """Accepting a token drawn from q~ with probability min(1, p~/q~) accepts with probability
    sum_v min(p~, q~) = a^sample at every depth, independently, so the mean of tau over many
    windows is the WTV expected length sum_k prod_{j<=k} a^s_j."""
    import oracle
    rng = np.random.default_rng(5)
    K, V, T, n = 3, 5, 1.2, 20000
    zp = rng.normal(0, 1.5, size=(K, V))
    zq = zp + rng.normal(0, 1.0, size=(K, V))
    tgt = np.broadcast_to(zp, (n, K, V))
    dr = np.broadcast_to(zq, (n, K, V))
    out = oracle.accept_reward(tgt, dr, None, oracle.REWARD_SAMPLED_DRAFT, T=T, seed=9)
    a = oracle.acceptance_sampling(zp, zq, T)
    want = sum(np.prod(a[:k + 1]) for k in range(K))
    tau = out["tau"].astype(np.float64)
    assert abs(tau.mean() - want) <= 5 * tau.std() / np.sqrt(n), (tau.mean(), want)
    ref = oracle.accept_reward(tgt, dr, dr, oracle.REWARD_SAMPLED_DRAFT, T=T, seed=9)
    np.testing.assert_array_equal(ref["tau"], ref["tau_ref"])     # common random numbers
