"""Pins of the RRF / EAHR oracle (arXiv 2608.07152, Sec. 2.1, 2.2, 3.4, 4.2)."""
import itertools
import json
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import eahr_oracle as eo
from oracle import rrf_oracle as ro
import synth

F = Fraction


def test_rank_scaled_reduces_to_plain_rrf_at_unit_weight():
    # Sec. 2.1: with w_i = 1 the contribution is 1 / (r + k - 1)
    for r in (1, 2, 59, 1000):
        assert ro.contribution(r, 1, 60) == F(1, r + 59)
    assert ro.contribution(5, 0, 60) == 0
    # rank-scaled weight divides the rank: w = 2 halves the effective rank
    assert ro.contribution(10, 2, 60) == F(1, 5 + 59)
    # numerator form, as in "w / (60 + rank)"
    assert ro.contribution(7, 1, 60, ro.NUMERATOR) == F(1, 67)
    assert ro.contribution(7, 3, 60, ro.NUMERATOR) == F(3, 67)
    # equal at w = 1 once the constants are aligned
    assert ro.contribution(9, 1, 61) == ro.contribution(9, 1, 60, ro.NUMERATOR)


def test_contributions_are_nonnegative_and_nonincreasing():
    for form in (ro.RANK_SCALED, ro.NUMERATOR):
        for w in (F(1, 3), 1, 2, 7):
            g = [ro.contribution(r, w, 60, form) for r in range(1, 200)]
            assert all(x > 0 for x in g)
            assert all(a > b for a, b in zip(g, g[1:]))


def test_target_topk_worked_example():
    # dense  = [3, 1, 2, 0], sparse = [1, 3, 0, 2], k = 60, w = 1:
    # F(1) = F(3) = 1/60 + 1/61 (tie -> id 1 first), F(2) = F(0) = 1/62 + 1/63
    T = ro.target_topk([[3, 1, 2, 0], [1, 3, 0, 2]], [1, 1], 60, 3)
    assert [x for x, _ in T] == [1, 3, 0]
    assert T[0][1] == F(1, 60) + F(1, 61)
    assert T[2][1] == F(1, 62) + F(1, 63)


def test_zero_score_items_are_never_appended():
    # sparse support {5}; dense weight 0 -> only item 5 has F > 0
    T = ro.target_topk([[1, 2, 5, 3], [5]], [0, 1], 60, 3)
    assert T == [(5, F(1, 60))]


def test_certification_rule_reproduces_complete_list_target_exhaustively():
    # Sec. 2.2 proves that the certified prefix equals T*_K.  Check it for
    # every pair of rankings of 5 items at every pair of depths.
    items = list(range(5))
    perms = list(itertools.permutations(items))
    rng = np.random.default_rng(0)
    for a, b in [(perms[i], perms[j]) for i, j in rng.integers(0, len(perms), (150, 2))]:
        for K in (1, 2, 5):
            T = [x for x, _ in ro.target_topk([a, b], [1, 1], 60, K)]
            for da in range(6):
                for db in range(6):
                    A, done = eo.certify([a[:da], b[:db]], [da == 5, db == 5], [1, 1], 60, K)
                    assert A == T[:len(A)]                 # never a wrong prefix
                    if da == 5 and db == 5:
                        assert done and A == T             # complete lists decide


def test_certification_with_weights_and_partial_sparse_support():
    rng = np.random.default_rng(1)
    for trial in range(100):
        n = 7
        dense = rng.permutation(n).tolist()
        sparse = rng.permutation(n)[: rng.integers(0, n + 1)].tolist()
        w = [F(int(rng.integers(1, 4)), int(rng.integers(1, 3))), F(int(rng.integers(0, 3)))]
        form = ro.RANK_SCALED if trial % 2 else ro.NUMERATOR
        T = [x for x, _ in ro.target_topk([dense, sparse], w, 60, 4, form)]
        A, done = eo.certify([dense, sparse], [True, True], w, 60, 4, form)
        assert done and A == T


def test_large_target_matches_exact_target():
    rng = np.random.default_rng(2)
    n = 3000
    d = rng.permutation(n)
    s = rng.permutation(n)[:2000]
    for K in (1, 20, 50):
        for form, k in ((ro.RANK_SCALED, 60), (ro.NUMERATOR, 60)):
            assert ro.target_topk_large([d, s], [1, 1], k, K, form) == \
                ro.target_topk([d, s], [1, 1], k, K, form)


# --------------------------------------------------------------------------
# controlled rank streams (Sec. 3.4 protocol, Sec. 4.2 outcomes)
# --------------------------------------------------------------------------

def _block_shuffle(first, rng, block=32):
    out = np.array(first)
    for b in range(0, len(out), block):
        out[b:b + block] = rng.permutation(out[b:b + block])
    return out


@pytest.mark.parametrize("seed", [1729, 2027, 65537])
@pytest.mark.parametrize("n", [640, 2000])
def test_correlated_block32_streams_fix_top20_at_depth_32(seed, n):
    rng = np.random.default_rng(seed)
    first = rng.permutation(n)
    second = _block_shuffle(first, rng)
    A, depths, exhausted = eo.equal_depth_run([first.tolist(), second.tolist()],
                                              [1, 1], 60, 20, step=16)
    assert depths == [32, 32] and not any(exhausted)
    assert A == [x for x, _ in ro.target_topk([first, second], [1, 1], 60, 20)]


GOLDEN = json.load(open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                                   "controlled_streams.json")))


@pytest.mark.parametrize("n", GOLDEN["protocol"]["collection_sizes"])
def test_oracle_correlated_streams_at_the_printed_sizes(n):
    """The paper's printed outcome (tests/golden/controlled_streams.json):
    at every collection size and seed, correlated rankings fix the ordered
    Top-20 at depth 32."""
    K = GOLDEN["protocol"]["K"]
    for seed in GOLDEN["protocol"]["seeds"]:
        a, b = synth.controlled_streams(n, "correlated", seed)
        A, depths, exhausted = eo.equal_depth_run([a.tolist(), b.tolist()], [1, 1], 60, K,
                                                  step=16)
        assert depths == [GOLDEN["outcomes"]["correlated_depth"]] * 2 and not any(exhausted)
        assert A == [x for x, _ in ro.target_topk_large([a, b], [1, 1], 60, K)]


def test_oracle_partial_overlap_depth_near_the_printed_median():
    """The paper prints a median depth of 1264 for partial overlap (500 of
    the first list's Top-1000 plus 500 outside items in the second list's
    Top-1000); the random streams differ, so the check is loose."""
    n = GOLDEN["protocol"]["collection_sizes"][0]
    depths = []
    for seed in GOLDEN["protocol"]["seeds"]:
        a, b = synth.controlled_streams(n, "partial", seed)
        _, d, exhausted = eo.equal_depth_run([a.tolist(), b.tolist()], [1, 1], 60, 20, step=16)
        assert not any(exhausted)
        depths.append(d[0])
    med = GOLDEN["outcomes"]["partial_overlap_median_depth"]
    assert 0.8 * med <= float(np.median(depths)) <= 1.6 * med, depths


@pytest.mark.parametrize("seed", [1729, 2027, 65537])
def test_reversed_streams_exhaust_both_lists(seed):
    n = 400
    rng = np.random.default_rng(seed)
    first = rng.permutation(n)
    second = first[::-1]
    A, depths, exhausted = eo.equal_depth_run([first.tolist(), second.tolist()],
                                              [1, 1], 60, 20, step=16)
    assert exhausted == [True, True] and depths == [n, n]
    assert A == [x for x, _ in ro.target_topk([first, second], [1, 1], 60, 20)]


def test_all_tied_streams_are_identical_id_ordered_lists():
    n = 500
    ids = list(range(n))                 # equal scores -> id order in both lists
    A, depths, _ = eo.equal_depth_run([ids, ids], [1, 1], 60, 20, step=16)
    assert depths == [32, 32] and A == list(range(20))
