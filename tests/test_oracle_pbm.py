"""Pins of the PBM oracle (arXiv 2608.07152, Sec. 2.1, Sec. 2.3.2, App. A.2).

Each test checks the oracle against something other than itself: a case
worked by hand, exact rational arithmetic where every float32 step is exact,
the rounding behaviour the fixed term order implies, the single-term closed
form, and the App. A.2 bound S_hat(x) <= H_hat(R).
"""
from fractions import Fraction

import numpy as np
import pytest

from oracle import pbm_oracle as po


def csr(n_terms, postings):
    """Term-major CSR from {term: [(doc, impact), ...]} (docs ascending)."""
    off, docs, imps = [0], [], []
    for t in range(n_terms):
        for d, p in postings.get(t, []):
            docs.append(d)
            imps.append(p)
        off.append(len(docs))
    return np.array(off, np.int64), np.array(docs, np.int64), np.array(imps, np.float32)


def test_hand_worked_case():
    # Sec. 2.3.2: S(x) = sum_t q_t p_t(x); query terms 0 (q = 2) and 2 (q = 0.5).
    # item 0: 2*1.5 + 0.5*4 = 5;  item 1: 0.5*2 = 1;  item 2: 2*0.5 = 1;
    # item 3: term 1 only (not in the query) -> 0;  item 4: 2*3 = 6;
    # item 5: no postings -> 0.  All values are exact in float32.
    off, docs, imps = csr(3, {0: [(0, 1.5), (2, 0.5), (4, 3.0)],
                              1: [(3, 7.0)],
                              2: [(0, 4.0), (1, 2.0)]})
    po.check_postings(off, docs, imps, 6)
    S = po.sparse_scores([0, 2], [2.0, 0.5], off, docs, imps, 6)
    assert S.tolist() == [5.0, 1.0, 1.0, 0.0, 6.0, 0.0]
    ids, sc = po.sparse_ranking([0, 2], [2.0, 0.5], off, docs, imps, 6)
    # Sec. 2.1: ties (items 1 and 2 at 1) by ascending id; items 3 and 5 score
    # 0, so they are outside the support U_s and have no rank
    assert ids.tolist() == [4, 0, 1, 2]
    assert sc.tolist() == [6.0, 5.0, 1.0, 1.0]
    # blocks of 2 ids: R0 = {0,1}, R1 = {2,3}, R2 = {4,5}
    # m_0 = (1.5, 0.5, 3), m_2 = (4, 0, 0) -> H = (2*1.5 + 0.5*4, 2*0.5, 2*3)
    H = po.range_bounds([0, 2], [2.0, 0.5], off, docs, imps, 6, 2)
    assert H.tolist() == [5.0, 1.0, 6.0]


def test_support_is_the_items_with_positive_score():
    # Sec. 2.1: the sparse retriever ranks U_s, the items with positive query
    # scores; items outside it have no rank (and contribute 0 to fusion).
    # Query: term 0 (q = 1), term 1 (q = 0), term 2 (q = 2^-100).
    #   item 0: p_0 = 3                      -> S = 3           in U_s
    #   item 1: only term 1 (zero weight)    -> S = RN(0 * 5) = 0
    #   item 2: p_0 = 0 (a zero impact)      -> S = 0
    #   item 3: p_2 = 2^-60: 2^-160 is below half the smallest subnormal
    #           (2^-150), so RN(q_2 p_2) = 0 -> S = 0
    #   item 4: no posting at all            -> S = 0
    #   item 5: p_2 = 2^-40: q_2 p_2 = 2^-140, a float32 subnormal > 0
    #   item 6: p_0 = 3, tie with item 0     -> after it by id
    tiny = 2.0 ** -100
    off, docs, imps = csr(4, {0: [(0, 3.0), (2, 0.0), (6, 3.0)],
                              1: [(1, 5.0)],
                              2: [(3, 2.0 ** -60), (5, 2.0 ** -40)],
                              3: [(4, 9.0)]})
    S = po.sparse_scores([0, 1, 2], [1.0, 0.0, tiny], off, docs, imps, 7)
    assert S[3] == 0 and S[5] == np.float32(2.0 ** -140) and S[5] > 0
    ids, sc = po.sparse_ranking([0, 1, 2], [1.0, 0.0, tiny], off, docs, imps, 7)
    assert ids.tolist() == [0, 6, 5]
    assert sc.tolist() == [3.0, 3.0, float(np.float32(2.0 ** -140))]
    # a query that matches nothing has an empty ranked list
    ids, sc = po.sparse_ranking([1], [0.0], off, docs, imps, 7)
    assert ids.size == 0 and sc.size == 0


def _dyadic_instance(rng, n_items, n_terms, nnz):
    postings = {}
    for t in range(n_terms):
        d = np.sort(rng.choice(n_items, size=min(nnz, n_items), replace=False))
        # small integers times 1/8: every product and partial sum below is
        # exact in float32 (at most 2^12 * 2^3 * few terms << 2^24 units)
        p = rng.integers(0, 64, size=d.size) / 8.0
        postings[t] = list(zip(d.tolist(), p.tolist()))
    return postings


def test_exact_rational_sums_on_dyadic_inputs():
    rng = np.random.default_rng(11)
    for trial in range(20):
        n_items, n_terms = 37 + trial, 9
        postings = _dyadic_instance(rng, n_items, n_terms, nnz=12)
        off, docs, imps = csr(n_terms, postings)
        q_terms = rng.choice(n_terms, size=5, replace=False)
        q_w = rng.integers(0, 16, size=5) / 4.0
        S = po.sparse_scores(q_terms, q_w, off, docs, imps, n_items)
        exact = [Fraction(0)] * n_items
        for t, w in zip(q_terms.tolist(), q_w.tolist()):
            for d, p in postings[t]:
                exact[d] += Fraction(w) * Fraction(p)
        assert [Fraction(float(s)) for s in S] == exact
        # complete ranking by (score desc, id asc) against a sort of the
        # exact rationals
        ids, _ = po.sparse_ranking(q_terms, q_w, off, docs, imps, n_items)
        want = sorted((x for x in range(n_items) if exact[x] > 0), key=lambda x: (-exact[x], x))
        assert ids.tolist() == want


def test_sum_follows_the_query_term_order():
    # App. A.2: one fixed order sigma.  Contributions 1, 2^-24, 2^-24 on one
    # item: in the order (1, 2^-24, 2^-24) each addition is a tie that rounds
    # to even and leaves 1; in the order (2^-24, 2^-24, 1) the two small
    # terms first make 2^-23, and 1 + 2^-23 is exact.
    tiny = 2.0 ** -24
    off, docs, imps = csr(3, {0: [(0, 1.0)], 1: [(0, tiny)], 2: [(0, tiny)]})
    S1 = po.sparse_scores([0, 1, 2], [1.0, 1.0, 1.0], off, docs, imps, 1)
    S2 = po.sparse_scores([1, 2, 0], [1.0, 1.0, 1.0], off, docs, imps, 1)
    assert S1[0] == np.float32(1.0)
    assert S2[0] == np.float32(1.0 + 2.0 ** -23)
    # and the product is rounded before the sum (no fused multiply-add):
    # acc = 2^-24 from term 0; term 1 has q = p = 1 + 2^-23, exact product
    # 1 + 2^-22 + 2^-46, rounded to 1 + 2^-22.  acc + (1 + 2^-22) lies
    # exactly halfway between 1 + 2 * 2^-23 and 1 + 3 * 2^-23 and rounds to
    # the even one, 1 + 2^-22; a fused multiply-add would see the extra
    # 2^-46 and round up to 1 + 3 * 2^-23.
    a = 1.0 + 2.0 ** -23
    off, docs, imps = csr(2, {0: [(0, tiny)], 1: [(0, a)]})
    S = po.sparse_scores([0, 1], [1.0, a], off, docs, imps, 1)
    assert S[0] == np.float32(1.0 + 2.0 ** -22)


def test_single_term_closed_form():
    # one query term: the ranking is that term's postings with a positive
    # impact, by (impact desc, id asc); nothing else has a rank
    rng = np.random.default_rng(3)
    n_items = 200
    d = np.sort(rng.choice(n_items, size=60, replace=False))
    p = rng.integers(0, 20, size=60).astype(np.float32) * np.float32(0.37)
    off, docs, imps = csr(1, {0: list(zip(d.tolist(), p.tolist()))})
    ids, sc = po.sparse_ranking([0], [1.0], off, docs, imps, n_items)
    pos = [(float(np.float32(x)), int(y)) for x, y in zip(p, d) if x > 0]
    want = [y for _, y in sorted(pos, key=lambda z: (-z[0], z[1]))]
    assert ids.tolist() == want
    assert np.all(sc > 0)


def test_range_bound_covers_every_item():
    # App. A.2: S_hat(x) <= H_hat(R) for every x in R, whatever the order
    rng = np.random.default_rng(5)
    for trial in range(10):
        n_items, n_terms, block = 300 + trial * 7, 20, 16
        postings = {}
        for t in range(n_terms):
            k = int(rng.integers(1, 80))
            d = np.sort(rng.choice(n_items, size=k, replace=False))
            p = rng.gamma(2.0, 1.3, size=k).astype(np.float32)
            postings[t] = list(zip(d.tolist(), p.tolist()))
        off, docs, imps = csr(n_terms, postings)
        q_terms = rng.choice(n_terms, size=8, replace=False)
        q_w = rng.gamma(1.5, 0.7, size=8).astype(np.float32)
        S = po.sparse_scores(q_terms, q_w, off, docs, imps, n_items)
        H = po.range_bounds(q_terms, q_w, off, docs, imps, n_items, block)
        assert np.all(S <= H[np.arange(n_items) // block])
        # the complete ranking is U_s without repeats, scores nonincreasing
        ids, sc = po.sparse_ranking(q_terms, q_w, off, docs, imps, n_items)
        assert sorted(ids.tolist()) == np.nonzero(S > 0)[0].tolist()
        assert np.all(np.diff(sc.astype(np.float64)) <= 0)


def test_block_maxima_by_brute_force():
    rng = np.random.default_rng(9)
    n_items, block = 50, 8
    d = np.sort(rng.choice(n_items, size=30, replace=False))
    p = rng.random(30).astype(np.float32)
    off, docs, imps = csr(1, {0: list(zip(d.tolist(), p.tolist()))})
    ranges, maxima = po.block_maxima(off, docs, imps, n_items, block)[0]
    for r in range(-(-n_items // block)):
        inside = [pp for dd, pp in zip(d, p) if dd // block == r]
        if inside:
            k = ranges.tolist().index(r)
            assert maxima[k] == max(inside)
        else:
            assert r not in ranges.tolist()


def test_invalid_inputs_are_rejected():
    off, docs, imps = csr(2, {0: [(1, 1.0), (3, 2.0)], 1: [(0, 0.5)]})
    po.check_postings(off, docs, imps, 4)
    with pytest.raises(ValueError):
        po.check_postings(off, docs, np.array([1.0, -1.0, 0.5], np.float32), 4)
    with pytest.raises(ValueError):
        po.check_postings(off, np.array([3, 1, 0]), imps, 4)
    with pytest.raises(ValueError):
        po.check_postings(off, docs, imps, 3)
    with pytest.raises(ValueError):
        po.check_query([0, 0], [1.0, 1.0], 2)
    with pytest.raises(ValueError):
        po.check_query([0], [float("nan")], 2)
