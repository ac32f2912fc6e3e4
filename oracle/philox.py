"""Philox4x32-10 counter-based generator, numpy (test infrastructure only).

Written from the published definition: J. K. Salmon, M. A. Moraes, R. O. Dror and
D. E. Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3", SC'11, Sec. 4 (the
Philox S-box built from two 32x32->64 multiplies, a Weyl sequence for the round
keys, ten rounds).  The multipliers and Weyl increments are the constants given
there.

The GRPO reward under sampling verification draws one uniform per (window,
depth); it is keyed here as counter = (n_lo, n_hi, k, 0) with n the global
window index and k the depth, key = (seed_lo, seed_hi), and u is built from the
first output word as ((x0 >> 9) * 2 + 1) * 2^-24, an odd multiple of 2^-24 in
(0, 1) that fp32 represents exactly.
"""

from __future__ import annotations

import numpy as np

PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9   # golden ratio
PHILOX_W1 = 0xBB67AE85   # sqrt(3) - 1
_MASK32 = np.uint64(0xFFFFFFFF)
_SH32 = np.uint64(32)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Ten Philox rounds on 4 x 32-bit counter words with a 2 x 32-bit key.

    Each round multiplies words 0 and 2 by the two constants (full 64-bit
    products), and the new state is (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2),
    hi(M0*c0) ^ c3 ^ k1, lo(M0*c0)); the key advances by the Weyl increments
    between rounds.  Inputs are array-likes of uint32 values; returns four
    uint32 arrays.
    """
    x0, x1, x2, x3 = (np.asarray(v, dtype=np.uint64) & _MASK32 for v in (c0, c1, c2, c3))
    ka = np.uint64(k0) & _MASK32
    kb = np.uint64(k1) & _MASK32
    for rnd in range(10):
        if rnd > 0:
            ka = (ka + np.uint64(PHILOX_W0)) & _MASK32
            kb = (kb + np.uint64(PHILOX_W1)) & _MASK32
        prod0 = np.uint64(PHILOX_M0) * x0          # < 2^64, exact in uint64
        prod1 = np.uint64(PHILOX_M1) * x2
        hi0, lo0 = prod0 >> _SH32, prod0 & _MASK32
        hi1, lo1 = prod1 >> _SH32, prod1 & _MASK32
        x0, x1, x2, x3 = hi1 ^ x1 ^ ka, lo1, hi0 ^ x3 ^ kb, lo0
    return tuple(v.astype(np.uint32) for v in (x0, x1, x2, x3))


def uniform01(seed: int, window, depth) -> np.ndarray:
    """u(seed, n, k) in (0, 1): the uniform the sampling reward draws for window n, depth k."""
    n = np.asarray(window, dtype=np.uint64)
    k = np.asarray(depth, dtype=np.uint64)
    n, k = np.broadcast_arrays(n, k)
    x0, _, _, _ = philox4x32_10(n & _MASK32, n >> _SH32, k, np.zeros_like(n),
                                seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    m = (x0.astype(np.uint64) >> np.uint64(9)).astype(np.float64)
    return (2.0 * m + 1.0) * 2.0 ** -24


def gumbel_uniforms(seed: int, window: int, depth: int, V: int) -> np.ndarray:
    """The V uniforms of the sampled-draft reward's Gumbel-max draw for window n, depth k:
    element v takes output word v mod 4 of counter (n_lo, n_hi, k, 1 + v div 4) (word 3 = 0 is
    the acceptance draw's counter, so the two never share a counter), mapped to (0, 1) as
    uniform01 maps x0."""
    n = np.uint64(window)
    c3 = np.arange((V + 3) // 4, dtype=np.uint64) + np.uint64(1)
    words = philox4x32_10(np.full_like(c3, n & _MASK32), np.full_like(c3, n >> _SH32),
                          np.full_like(c3, np.uint64(depth)), c3, seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    x = np.stack(words, axis=1).reshape(-1)[:V]            # element v = 4 c + w
    m = (x.astype(np.uint64) >> np.uint64(9)).astype(np.float64)
    return (2.0 * m + 1.0) * 2.0 ** -24
