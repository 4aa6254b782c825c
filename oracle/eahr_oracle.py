"""The ordered certification rule of EAHR, applied to given ranked prefixes.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Paper: arXiv 2608.07152, Sec. 2.2.  At access depths d = (d_i):
  u_i = g_i(d_i + 1) if list i is Open, 0 if it is Exhausted;
  L(x) = sum of g_i(r_i(x)) over the lists in which x has been read;
  U(x) = L(x) + sum of u_i over the Open lists in which x has not been read;
  B    = sum_i u_i (the shared bound of every unseen item).
With A the ordered prefix already fixed and R = O \\ A, the item x+ of R
with the greatest L (ties: smaller id) is appended when
  (L(x+), x+) > (U(y), y) for every other y in R   and   L(x+) > B,
where (a, x) > (b, y) means a > b, or a == b and x has the smaller id.
The decision repeats until q_K positions are fixed.
"""
from __future__ import annotations

from fractions import Fraction

from .rrf_oracle import RANK_SCALED, contribution


def certify(prefixes, exhausted, weights, k: int, K: int, form: str = RANK_SCALED):
    """Return (A, done): the fixed ordered prefix A and whether the result is
    complete (|A| == K, or no unread or observed item can still have F > 0)."""
    ranks: dict[int, dict[int, int]] = {}
    for i, P in enumerate(prefixes):
        for r, x in enumerate(P):
            ranks.setdefault(int(x), {})[i] = r + 1
    u = [Fraction(0) if exhausted[i] else contribution(len(P) + 1, weights[i], k, form)
         for i, P in enumerate(prefixes)]
    B = sum(u, Fraction(0))
    L = {x: sum((contribution(r, weights[i], k, form) for i, r in rs.items()), Fraction(0))
         for x, rs in ranks.items()}
    U = {x: L[x] + sum((u[i] for i in range(len(prefixes))
                        if not exhausted[i] and i not in rs), Fraction(0))
         for x, rs in ranks.items()}
    A = []
    R = set(ranks)
    while len(A) < K and R:
        x = max(R, key=lambda y: (L[y], -y))
        beaten = all((L[x], -x) > (U[y], -y) for y in R if y != x)
        if not (beaten and L[x] > B):
            break
        A.append(x)
        R.remove(x)
    done = len(A) == K or (B == 0 and all(U[y] == 0 for y in R))
    return A, done


def equal_depth_run(lists, weights, k: int, K: int, step: int = 16,
                    form: str = RANK_SCALED):
    """Controlled-stream protocol of Sec. 3.4: every list advances to the same
    depth, and certification is checked every ``step`` ranks.  A list whose
    whole length has been read is Exhausted.  Returns (A, depths, exhausted)
    at the first checkpoint whose result is complete."""
    n = [len(x) for x in lists]
    d = 0
    while True:
        d += step
        depths = [min(d, ni) for ni in n]
        exhausted = [di >= ni for di, ni in zip(depths, n)]
        prefixes = [lst[:di] for lst, di in zip(lists, depths)]
        A, done = certify(prefixes, exhausted, weights, k, K, form)
        if done:
            return A, depths, exhausted
