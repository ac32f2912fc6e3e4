"""Brute-force simulation of speculative verification, in exact rationals.

Used only to pin the oracle: it never looks at the oracle's formulas.  A window of
gamma positions is drafted token by token from fixed per-position distributions
(the teacher-forced setting of Sec. 3.1: every position sees the ground-truth
prefix), and verified left to right until the first rejection.  Every draft path
in V^gamma and every accept/reject outcome is enumerated with its probability,
and the accepted length L is averaged over all of them.
"""

from fractions import Fraction
from itertools import product


def expected_accepted_length_sampling(p, q):
    """E[L] under sampling verification (Sec. 2.3): draft y_j ~ q_j, accept w.p. min(1, p_j(y)/q_j(y)).

    ``p`` and ``q`` are lists (one per position) of lists of Fractions summing to 1.
    """
    gamma = len(p)
    V = len(p[0])
    total = Fraction(0)
    for path in product(range(V), repeat=gamma):
        p_path = Fraction(1)
        for j, y in enumerate(path):
            p_path *= q[j][y]
        if p_path == 0:
            continue
        alphas = [min(Fraction(1), p[j][y] / q[j][y]) for j, y in enumerate(path)]
        for outcome in product((0, 1), repeat=gamma):
            p_out = Fraction(1)
            for j, b in enumerate(outcome):
                p_out *= alphas[j] if b else (1 - alphas[j])
            L = 0
            while L < gamma and outcome[L]:
                L += 1
            total += p_path * p_out * L
    return total


def expected_accepted_length_greedy(p_star, q):
    """E[L] under greedy verification (Sec. 2.3): draft y_j ~ q_j, accepted iff y_j == x*_j.

    ``p_star`` lists the target's argmax token per position.
    """
    gamma = len(q)
    V = len(q[0])
    total = Fraction(0)
    for path in product(range(V), repeat=gamma):
        p_path = Fraction(1)
        for j, y in enumerate(path):
            p_path *= q[j][y]
        L = 0
        while L < gamma and path[L] == p_star[L]:
            L += 1
        total += p_path * L
    return total


def acceptance_by_rejection(p, q):
    """E_{y~q}[min(1, p(y)/q(y))]: the left-hand side of Eq. acc_sample, enumerated."""
    return sum((qy * min(Fraction(1), py / qy) for py, qy in zip(p, q) if qy > 0), Fraction(0))
