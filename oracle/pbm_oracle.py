"""PBM oracle: exact sparse scores, range bounds and the complete sparse ranking.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Paper: arXiv 2608.07152.
  * Sec. 2.1   complete ranked list: items ordered by score, ties broken by
               the identifier order (here: ascending id).
  * Sec. 2.3.2 sparse score S(x) = sum_{t in Q} q_t p_t(x) over the nonzero
               query terms Q, with q_t >= 0 and impacts p_t(x) >= 0; a
               contiguous identifier range R has block maxima
               m_t(R) = max_{x in R} p_t(x) (0 without a posting of t) and
               the bound H(R) = sum_{t in Q} q_t m_t(R) >= S(x) for x in R.
  * App. A.2   both sums are evaluated in float32 in one fixed term order
               sigma; missing terms contribute p_t(x) = 0; with the same
               operations in the same order the machine values keep
               S_hat(x) <= H_hat(R).

Readings (the paper fixes neither):
  * sigma is the order in which the query lists its terms; every step is a
    float32 multiplication rounded to nearest-even followed by a float32
    addition rounded to nearest-even (no fused multiply-add):
        acc <- RN(acc + RN(q_t * p_t(x)))   for t in sigma, acc starting at +0;
  * the ranges are the fixed blocks [r B, (r + 1) B) of the identifier
    space for a block size B;
  * the sparse ranking's support is U_s = {x : S_hat(x) > 0} (Sec. 2.1: the
    sparse retriever ranks the items with positive query scores; items
    outside U_s have no rank and contribute nothing to fusion).  An item
    with no posting of a query term, with only zero impacts or zero-weight
    terms, or whose float32 products all round to zero, is outside U_s.

Postings are term-major (CSR): the postings of term t are entries
term_off[t] .. term_off[t+1]-1 of (docs, imps), docs strictly ascending.
"""
from __future__ import annotations

import numpy as np


def check_postings(term_off, docs, imps, n_items: int) -> None:
    """Raise ValueError unless the postings are well formed: offsets
    nondecreasing and covering docs, item ids in range and strictly
    ascending within a term, impacts finite and nonnegative (App. A.2)."""
    term_off = np.asarray(term_off, np.int64)
    docs = np.asarray(docs, np.int64)
    imps = np.asarray(imps, np.float32)
    if term_off.ndim != 1 or term_off.size < 1 or term_off[0] != 0:
        raise ValueError("term offsets must start at 0")
    if np.any(np.diff(term_off) < 0) or term_off[-1] != docs.size or docs.size != imps.size:
        raise ValueError("term offsets must be nondecreasing and cover the postings")
    if docs.size and (docs.min() < 0 or docs.max() >= n_items):
        raise ValueError("item id out of range")
    if not np.all(np.isfinite(imps)) or np.any(imps < 0):
        raise ValueError("impacts must be finite and nonnegative")
    for t in range(term_off.size - 1):
        d = docs[term_off[t]:term_off[t + 1]]
        if d.size > 1 and np.any(np.diff(d) <= 0):
            raise ValueError(f"postings of term {t} are not strictly ascending")


def check_query(q_terms, q_weights, n_terms: int) -> None:
    """Raise ValueError unless the query terms are distinct vocabulary terms
    and the weights finite and nonnegative (Sec. 2.3.2, App. A.2)."""
    q_terms = np.asarray(q_terms, np.int64)
    q_weights = np.asarray(q_weights, np.float32)
    if q_terms.shape != q_weights.shape or q_terms.ndim != 1:
        raise ValueError("one weight per query term")
    if q_terms.size and (q_terms.min() < 0 or q_terms.max() >= n_terms):
        raise ValueError("query term out of range")
    if np.unique(q_terms).size != q_terms.size:
        raise ValueError("query terms must be distinct")
    if not np.all(np.isfinite(q_weights)) or np.any(q_weights < 0):
        raise ValueError("query weights must be finite and nonnegative")


def sparse_scores(q_terms, q_weights, term_off, docs, imps, n_items: int) -> np.ndarray:
    """S_hat(x) for every item (Sec. 2.3.2 in the float32 order of App. A.2):
    term by term in query order, acc <- RN(acc + RN(q_t * p_t(x))); an item
    without a posting of t adds RN(q_t * 0) = +0, which leaves acc as it is."""
    term_off = np.asarray(term_off, np.int64)
    docs = np.asarray(docs, np.int64)
    imps = np.asarray(imps, np.float32)
    S = np.zeros(n_items, np.float32)
    for t, w in zip(np.asarray(q_terms, np.int64), np.asarray(q_weights, np.float32)):
        lo, hi = term_off[t], term_off[t + 1]
        d = docs[lo:hi]
        contrib = np.multiply(np.float32(w), imps[lo:hi], dtype=np.float32)   # RN product
        S[d] = np.add(S[d], contrib, dtype=np.float32)                        # RN sum
    return S


def sparse_ranking(q_terms, q_weights, term_off, docs, imps, n_items: int):
    """The complete sparse ranked list (Sec. 2.1): the support U_s = {x :
    S_hat(x) > 0} ordered by (S_hat desc, id asc); returns (ids int64,
    scores float32), both of length |U_s|."""
    S = sparse_scores(q_terms, q_weights, term_off, docs, imps, n_items)
    ids = np.nonzero(S > 0)[0].astype(np.int64)
    order = np.lexsort((ids, -S[ids].astype(np.float64)))
    return ids[order], S[ids[order]]


def block_maxima(term_off, docs, imps, n_items: int, block: int):
    """m_t(R) for every term t and block R = [r B, (r + 1) B) that holds a
    posting of t (Sec. 2.3.2): a dict {t: (ranges int64, maxima float32)}."""
    term_off = np.asarray(term_off, np.int64)
    docs = np.asarray(docs, np.int64)
    imps = np.asarray(imps, np.float32)
    out = {}
    for t in range(term_off.size - 1):
        d = docs[term_off[t]:term_off[t + 1]]
        p = imps[term_off[t]:term_off[t + 1]]
        r = d // block
        ranges = np.unique(r)
        maxima = np.array([p[r == x].max() for x in ranges], np.float32)
        out[t] = (ranges, maxima)
    return out


def range_bounds(q_terms, q_weights, term_off, docs, imps, n_items: int, block: int) -> np.ndarray:
    """H_hat(R) for every block R (Sec. 2.3.2, App. A.2): the same float32
    steps as sparse_scores, in the same term order, over m_t(R) instead of
    p_t(x); a block without a posting of t adds +0."""
    n_ranges = (n_items + block - 1) // block
    H = np.zeros(n_ranges, np.float32)
    maxima = block_maxima(term_off, docs, imps, n_items, block)
    for t, w in zip(np.asarray(q_terms, np.int64), np.asarray(q_weights, np.float32)):
        r, m = maxima[int(t)]
        contrib = np.multiply(np.float32(w), m, dtype=np.float32)
        H[r] = np.add(H[r], contrib, dtype=np.float32)
    return H
