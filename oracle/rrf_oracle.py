"""Complete-list weighted RRF and the EAHR target T*_K, in exact rationals.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Paper: arXiv 2608.07152, Sec. 2.1.
  F(x) = sum over retrievers i with x in U_i of g_i(r_i(x)).
  Rank-scaled weighted RRF (the paper's form):
      g_i(r) = 0 if w_i = 0, else 1 / (r / w_i + k - 1).
  Numerator-weighted form (the form w_i / (k + r) that the paper contrasts
  with its own; with w_i = 1 it equals the rank-scaled form at k + 1):
      g_i(r) = w_i / (k + r).
  U+ = {x : F(x) > 0}, q_K = min(K, |U+|); T*_K = the first q_K items of U+
  sorted by F descending, ties by ascending id.  Zero-score items are never
  appended.
"""
from __future__ import annotations

from fractions import Fraction

import numpy as np

RANK_SCALED = "rank_scaled"
NUMERATOR = "numerator"


def contribution(r: int, w, k: int, form: str = RANK_SCALED) -> Fraction:
    """g(r) for rank r >= 1 (Sec. 2.1)."""
    w = Fraction(w)
    if r < 1:
        raise ValueError("ranks start at 1")
    if w == 0:
        return Fraction(0)
    if form == RANK_SCALED:
        return 1 / (Fraction(r) / w + k - 1)
    if form == NUMERATOR:
        return w / (k + r)
    raise ValueError(form)


def fused_scores(rankings, weights, k: int, form: str = RANK_SCALED) -> dict:
    """F(x) for every item of any ranking, as exact Fractions."""
    F: dict[int, Fraction] = {}
    for lst, w in zip(rankings, weights):
        for pos, x in enumerate(lst):
            x = int(x)
            F[x] = F.get(x, Fraction(0)) + contribution(pos + 1, w, k, form)
    return F


def target_topk(rankings, weights, k: int, K: int, form: str = RANK_SCALED):
    """T*_K of Sec. 2.1: [(id, F)] for the first q_K items of U+."""
    F = fused_scores(rankings, weights, k, form)
    pos = [(f, x) for x, f in F.items() if f > 0]
    pos.sort(key=lambda t: (-t[0], t[1]))
    return [(x, f) for f, x in pos[:K]]


def target_topk_large(rankings, weights, k: int, K: int, form: str = RANK_SCALED):
    """T*_K for long rankings.  binary64 fused scores (relative error a few
    ulps) select every item whose value is within 1e-9 relative of the K-th
    largest; those candidates are then ranked with ``target_topk``'s exact
    rule.  Returns the same list as ``target_topk``."""
    rankings = [np.asarray(r, np.int64) for r in rankings]
    n_ids = int(max((r.max() + 1) if r.size else 0 for r in rankings))
    Fd = np.zeros(n_ids, np.float64)
    for lst, w in zip(rankings, weights):
        w = Fraction(w)
        if w == 0 or lst.size == 0:
            continue
        r = np.arange(1, lst.size + 1, dtype=np.float64)
        if form == RANK_SCALED:
            g = 1.0 / (r / float(w) + (k - 1))
        else:
            g = float(w) / (k + r)
        np.add.at(Fd, lst, g)
    positive = np.nonzero(Fd > 0)[0]
    if positive.size <= K:
        cand = set(positive.tolist())
    else:
        kth = np.partition(Fd[positive], positive.size - K)[positive.size - K]
        cand = set(positive[Fd[positive] >= kth * (1 - 1e-9)].tolist())
    F: dict[int, Fraction] = {}
    for lst, w in zip(rankings, weights):
        idx = np.nonzero(np.isin(lst, np.fromiter(cand, np.int64, len(cand))))[0]
        for p in idx.tolist():
            x = int(lst[p])
            F[x] = F.get(x, Fraction(0)) + contribution(p + 1, w, k, form)
    pos = [(f, x) for x, f in F.items() if f > 0]
    pos.sort(key=lambda t: (-t[0], t[1]))
    return [(x, f) for f, x in pos[:K]]


def as_float(f: Fraction) -> float:
    """Correctly rounded binary64 value of a Fraction (Python's int/int true
    division rounds correctly)."""
    return f.numerator / f.denominator
