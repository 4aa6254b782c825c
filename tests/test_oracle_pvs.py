"""Pins of the PVS oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: exact
rational arithmetic, closed forms, worked cases, invariances, or brute force
(arXiv 2608.07152, Sec. 2.3.1 and Appendix A.1).
"""
import math
from fractions import Fraction

import numpy as np
import pytest

from oracle import pvs_oracle as po

F = Fraction


def exact_dot(q, v):
    return sum((F(float(a)) * F(float(b)) for a, b in zip(q, v)), F(0))


def f32_round_exact(x: Fraction) -> np.float32:
    """Nearest float32 to the rational x, ties to even, by exact comparison
    with the neighbouring float32 values (independent of the oracle's route
    through binary64)."""
    f = np.float32(float(x))
    cands = {f, np.nextafter(f, np.float32(np.inf)), np.nextafter(f, np.float32(-np.inf))}
    best = None
    for c in cands:
        if not np.isfinite(c):
            continue
        d = abs(F(float(c)) - x)
        key = (d, int(np.frombuffer(np.float32(c).tobytes(), np.uint32)[0]) & 1)
        if best is None or key < best[0]:
            best = (key, c)
    return np.float32(best[1])


# --------------------------------------------------------------------------
# quantization (Sec. 2.3.1)
# --------------------------------------------------------------------------

def test_zero_vector_uses_unit_scale_and_zero_codes():
    Q = po.quantize(np.zeros((1, 16), np.float32))
    assert Q.s[0] == 1.0 and not Q.z.any()
    assert Q.vnorm[0] == 0.0 and Q.enorm[0] == 0.0


def test_scale_is_f32_of_maxabs_over_127_and_extreme_code_is_127():
    rng = np.random.default_rng(1)
    V = rng.standard_normal((200, 33)).astype(np.float32)
    Q = po.quantize(V)
    for i in range(V.shape[0]):
        maxabs = np.abs(V[i]).max()
        # s_v is the float32 nearest to ||v||_inf / 127 (exact rational check)
        assert Q.s[i] == f32_round_exact(F(float(maxabs)) / 127)
        j = int(np.abs(V[i]).argmax())
        assert abs(int(Q.z[i, j])) == 127
        assert np.all(np.abs(Q.z[i].astype(int)) <= 127)
        # codes carry the sign of the coordinate (or are zero)
        assert np.all(Q.z[i].astype(int) * np.sign(V[i]) >= 0)


def test_codes_are_nearest_integers_of_the_f32_quotient():
    rng = np.random.default_rng(2)
    V = (rng.standard_normal((100, 40)) * rng.uniform(1e-3, 1e3, (100, 1))).astype(np.float32)
    Q = po.quantize(V)
    for i in range(V.shape[0]):
        s = F(float(Q.s[i]))
        for j in range(V.shape[1]):
            t = F(float(np.float32(V[i, j]) / np.float32(Q.s[i])))  # IEEE f32 quotient
            assert abs(t - int(Q.z[i, j])) <= F(1, 2)
        # the residual really is v - s z
        e = [F(float(V[i, j])) - s * int(Q.z[i, j]) for j in range(V.shape[1])]
        assert F(float(Q.enorm[i])) ** 2 >= sum(x * x for x in e)


def test_half_way_quotients_round_away_from_zero():
    # s = (127/128)/127 = 1/128 exactly; 2.5/128 / (1/128) = 2.5 exactly.
    V = np.array([[127 / 128, 2.5 / 128, -2.5 / 128, 0.5 / 128, -1.5 / 128]], np.float32)
    Q = po.quantize(V)
    assert Q.s[0] == np.float32(1 / 128)
    assert Q.z[0].tolist() == [127, 3, -3, 1, -2]


def test_power_of_two_scaling_is_exact():
    rng = np.random.default_rng(3)
    V = rng.standard_normal((50, 64)).astype(np.float32)
    A = po.quantize(V)
    for k in (-40, -3, 5, 30):
        B = po.quantize((V * np.float32(2.0 ** k)).astype(np.float32))
        assert np.array_equal(A.z, B.z)
        assert np.array_equal(A.s * np.float32(2.0 ** k), B.s)
        assert np.array_equal(A.vnorm * np.float32(2.0 ** k), B.vnorm)
        assert np.array_equal(A.enorm * np.float32(2.0 ** k), B.enorm)


def test_subnormal_scale_underflow_and_clipping():
    tiny = 2.0 ** -149
    # maxabs/127 underflows to 0: the smallest subnormal scale is used
    Q = po.quantize(np.array([[3 * tiny, -tiny, 0.0]], np.float32))
    assert Q.s[0] == np.float32(tiny)
    assert Q.z[0].tolist() == [3, -1, 0]
    # maxabs/127 rounds down to one subnormal step: the code clips at 127
    Q = po.quantize(np.array([[190 * tiny]], np.float32))
    assert Q.s[0] == np.float32(tiny) and Q.z[0, 0] == 127
    assert F(float(Q.enorm[0])) >= 63 * F(tiny)


def test_non_finite_input_is_reported():
    for bad in (np.nan, np.inf, -np.inf):
        V = np.ones((3, 8), np.float32)
        V[1, 4] = bad
        assert po.quantize(V).status == 1


# --------------------------------------------------------------------------
# norm bounds and gamma (App. A.1)
# --------------------------------------------------------------------------

def test_norm_bound_exact_cases():
    assert po.norm_bound([3.0, 4.0]) == 5.0
    assert po.norm_bound([0.0, 0.0]) == 0.0
    assert po.norm_bound([1.0]) == 1.0
    assert po.norm_bound([-3 * 2.0 ** -130, 4 * 2.0 ** -130]) == np.float32(5 * 2.0 ** -130)
    assert po.norm_bound([0.5] * 4) == 1.0


@pytest.mark.parametrize("seed", range(5))
def test_norm_bound_is_a_tight_upper_bound(seed):
    rng = np.random.default_rng(seed)
    for m in (1, 7, 128, 768):
        x = rng.standard_normal(m) * 10.0 ** rng.uniform(-30, 30)
        x = x.astype(np.float32).astype(np.float64)
        nb = po.norm_bound(x)
        ss = sum((F(float(v)) ** 2 for v in x), F(0))
        assert F(float(nb)) ** 2 >= ss                       # upper bound
        assert float(nb) <= math.sqrt(float(ss)) * (1 + 2.0 ** -20)  # tight


def test_gamma_is_smallest_f32_above_a_over_one_minus_a():
    for m in (1, 128, 384, 768, 1024, 4096):
        a = F(8 * m + 64, 2 ** 23)
        target = a / (1 - a)
        g = po.gamma(m)
        assert F(float(g)) >= target
        assert F(float(np.nextafter(g, np.float32(0)))) < target


def _qhat_queries():
    rng = np.random.default_rng(31)
    out = [rng.standard_normal(m).astype(np.float32) for m in (1, 7, 128, 768)]
    out.append((rng.standard_normal(96) * 1e30).astype(np.float32))
    # subnormal scale: max |q_j| / 127 lies below the smallest normal float32
    out.append((rng.standard_normal(64) * 1e-40).astype(np.float32))
    # one dominant entry and one that quantizes far from its value:
    # ||q_hat|| exceeds ||q|| by ~2e-5 relative (below)
    out.append(np.array([1.0, 0.004], np.float32))
    return out


@pytest.mark.parametrize("k", range(len(_qhat_queries())))
def test_query_encoding_bounds_the_norm_of_the_dequantized_query(k):
    """Sec. 2.3.1: q_hat = s_q z_q, and E needs ||q_hat||_2; App. A.1 wants it
    rounded up.  The stored bound must satisfy, in exact rationals,
    ||s_q z_q|| <= qhat <= (1 + 2^-20) ||s_q z_q|| (+ one subnormal step where
    the bound itself is subnormal).  Neither ||z_q|| (s_q dropped) nor ||q||
    (the query before quantization) passes this on the cases below."""
    q = _qhat_queries()[k]
    qe = po.encode_query(q)
    Q = po.quantize(q.reshape(1, -1))
    assert qe.status == 0
    assert np.array_equal(qe.z, Q.z[0]) and qe.s == Q.s[0]
    n2 = sum(((F(float(qe.s)) * int(z)) ** 2 for z in qe.z.tolist()), F(0))
    qh = F(float(qe.qhat))
    assert qh * qh >= n2                                     # an upper bound
    slack = qh - F(2.0 ** -149) if qh < F(2.0 ** -126) else qh
    assert slack * slack <= (1 + F(1, 2 ** 20)) ** 2 * n2   # and a tight one
    if k == len(_qhat_queries()) - 1:
        # this case separates ||q_hat|| from ||q|| by more than the tolerance
        qn2 = sum((F(float(x)) ** 2 for x in q.tolist()), F(0))
        assert qn2 * (1 + F(1, 2 ** 19)) < n2


# --------------------------------------------------------------------------
# intervals (Sec. 2.3.1 + App. A.1)
# --------------------------------------------------------------------------

def _exact_interval_terms(qe, q, Q, i, m):
    """c, E and G from the paper's formulas, evaluated exactly over the
    stored (already upward-rounded) norms."""
    dot = int(np.dot(qe.z[:m].astype(np.int64), Q.z[i, :m].astype(np.int64)))
    c_exact = F(float(qe.s)) * F(float(Q.s[i])) * dot
    E = F(float(qe.enorm)) * F(float(Q.vnorm[i])) + F(float(qe.qhat)) * F(float(Q.enorm[i]))
    return dot, c_exact, E


def _corpora():
    rng = np.random.default_rng(11)
    out = {}
    V = rng.standard_normal((300, 96)).astype(np.float32)
    out["normal"] = V / np.linalg.norm(V, axis=1, keepdims=True)
    base = rng.standard_normal((10, 96))
    D = base[rng.integers(0, 10, 300)] + 1e-4 * rng.standard_normal((300, 96))
    out["near_duplicates"] = (D / np.linalg.norm(D, axis=1, keepdims=True)).astype(np.float32)
    out["integers"] = rng.integers(-3, 4, (300, 96)).astype(np.float32)
    out["heavy_tail"] = (rng.standard_cauchy((300, 96))).astype(np.float32)
    out["tiny"] = (rng.standard_normal((300, 96)) * 1e-35).astype(np.float32)
    out["huge"] = (rng.standard_normal((300, 96)) * 1e15).astype(np.float32)
    S = rng.standard_normal((300, 96)).astype(np.float32)
    S[rng.random((300, 96)) < 0.9] = 0
    out["sparse"] = S
    return out


@pytest.mark.parametrize("name", list(_corpora().keys()))
def test_interval_contains_authoritative_score(name):
    V = _corpora()[name]
    rng = np.random.default_rng(5)
    m = V.shape[1]
    Q = po.quantize(V)
    assert Q.status == 0
    for t in range(4):
        q = V[rng.integers(0, V.shape[0])] + 0.3 * rng.standard_normal(m).astype(np.float32) * np.abs(V).max()
        q = q.astype(np.float32)
        qe = po.encode_query(q)
        lo, hi = po.intervals(qe, Q, m)
        s = po.exact_scores(q, V)
        assert np.all(lo <= s) and np.all(s <= hi), name


def test_interval_endpoints_round_the_paper_formula_outward():
    rng = np.random.default_rng(7)
    V = rng.standard_normal((60, 48)).astype(np.float32)
    q = rng.standard_normal(48).astype(np.float32)
    Q = po.quantize(V)
    qe = po.encode_query(q)
    lo, hi = po.intervals(qe, Q, 48)
    gam = F(float(qe.gamma))
    for i in range(V.shape[0]):
        dot, c_exact, E = _exact_interval_terms(qe, q, Q, i, 48)
        # the float centre: two IEEE float32 products (round to nearest)
        c = F(float(np.float32(np.float32(qe.s) * np.float32(Q.s[i])) * np.float32(dot)))
        assert abs(c - c_exact) <= 3 * F(2.0 ** -24) * abs(c_exact)
        G = (abs(c) + E + F(float(qe.qnorm)) * F(float(Q.vnorm[i]))) * gam
        half = E + G
        # outward rounding: the interval covers c +/- (E + G) exactly
        assert F(float(lo[i])) <= c - half
        assert F(float(hi[i])) >= c + half
        # and is at most a few float32 roundings wider
        width = F(float(hi[i])) - F(float(lo[i]))
        assert width <= 2 * half * (1 + F(1, 2 ** 19)) + 2 * F(2.0 ** -23) * abs(c)


def test_interval_one_matches_vector_form_and_dot_is_exact():
    rng = np.random.default_rng(8)
    V = rng.standard_normal((20, 1024)).astype(np.float32)
    q = rng.standard_normal(1024).astype(np.float32)
    Q = po.quantize(V)
    qe = po.encode_query(q)
    lo, hi = po.intervals(qe, Q, 1024)
    for i in range(20):
        dot = sum(int(a) * int(b) for a, b in zip(qe.z.tolist(), Q.z[i].tolist()))
        l1, h1 = po.interval_one(dot, qe, Q.s[i], Q.vnorm[i], Q.enorm[i])
        assert l1 == lo[i] and h1 == hi[i]


def test_padded_code_stride_gives_same_intervals():
    rng = np.random.default_rng(9)
    V = rng.standard_normal((30, 100)).astype(np.float32)
    q = rng.standard_normal(100).astype(np.float32)
    A = po.quantize(V)
    B = po.quantize(V, ldz=128)
    assert np.array_equal(A.z, B.z[:, :100]) and not B.z[:, 100:].any()
    qe = po.encode_query(q)
    la, ha = po.intervals(qe, A, 100)
    lb, hb = po.intervals(qe, B, 100)
    assert np.array_equal(la, lb) and np.array_equal(ha, hb)


# --------------------------------------------------------------------------
# authoritative score and dense ranking (Sec. 2.1)
# --------------------------------------------------------------------------

def test_exact_score_rounds_halfway_cases_correctly():
    # 1 + 2^-24 is halfway between 1 and 1 + 2^-23: ties to even -> 1
    assert po.exact_score_one(np.array([1.0, 2.0 ** -24], np.float32),
                              np.array([1.0, 1.0], np.float32)) == np.float32(1.0)
    # a tiny positive extra term breaks the tie upward, although the binary64
    # sum alone is exactly the halfway point
    s = po.exact_score_one(np.array([1.0, 2.0 ** -24, 2.0 ** -60], np.float32),
                           np.array([1.0, 1.0, 1.0], np.float32))
    assert s == np.float32(1.0 + 2.0 ** -23)
    s = po.exact_score_one(np.array([1.0, 2.0 ** -24, -(2.0 ** -60)], np.float32),
                           np.array([1.0, 1.0, 1.0], np.float32))
    assert s == np.float32(1.0)
    # (1 + 2^-23) + 2^-24 is halfway with an odd lower neighbour: ties to even -> up
    s = po.exact_score_one(np.array([1.0 + 2.0 ** -23, 2.0 ** -24], np.float32),
                           np.array([1.0, 1.0], np.float32))
    assert s == np.float32(1.0 + 2.0 ** -22)


@pytest.mark.parametrize("seed", range(3))
def test_exact_scores_equal_rational_rounding(seed):
    rng = np.random.default_rng(seed)
    m = 64
    V = rng.standard_normal((120, m)).astype(np.float32)
    V[::7] *= np.float32(1e-20)
    V[3] = -V[2]                                    # exact cancellation pair
    q = rng.standard_normal(m).astype(np.float32)
    s = po.exact_scores(q, V)
    for i in range(V.shape[0]):
        assert s[i] == f32_round_exact(exact_dot(q, V[i])), i
        assert po.exact_score_one(q, V[i]) == s[i]


def test_exact_scores_cancellation_is_exactly_zero():
    q = np.array([1e20, 1.0, -1e20], np.float32)
    v = np.array([1.0, 1.0, 1.0], np.float32)
    assert po.exact_scores(q, v[None])[0] == np.float32(1.0)


def test_exact_scores_in_the_subnormal_range_and_canonical_zero():
    """Products below the float32 range: scores are the rational rounding
    (including subnormal results), and any score that rounds to zero is +0."""
    rng = np.random.default_rng(11)
    m = 64
    V = (rng.standard_normal((80, m)) * 2.0 ** -75).astype(np.float32)
    q = (rng.standard_normal(m) * 2.0 ** -75).astype(np.float32)
    s = po.exact_scores(q, V)
    zeros = 0
    for i in range(V.shape[0]):
        want = f32_round_exact(exact_dot(q, V[i]))
        assert s[i] == want, i
        assert po.exact_score_one(q, V[i]).view(np.uint32) == s[i].view(np.uint32)
        if want == 0:
            zeros += 1
            assert s[i].view(np.uint32) == 0, i          # +0, never -0
    assert zeros > 0
    # exact value -2^-151: rounds to zero from below
    tiny = np.float32(2.0 ** -75)
    z = po.exact_scores(np.array([tiny], np.float32), np.array([[-tiny / 2]], np.float32))
    assert z.view(np.uint32)[0] == 0
    # 3 * 2^-150 lies between 2^-149 and 2^-148, nearer the latter
    three = po.exact_score_one(np.full(3, tiny, np.float32), np.full(3, tiny, np.float32))
    assert three == np.float32(2.0 ** -148)


def test_dense_ranking_brute_force_with_ties():
    rng = np.random.default_rng(4)
    base = rng.integers(-2, 3, (6, 5)).astype(np.float32)
    V = base[rng.integers(0, 6, 40)]                # many exact duplicates
    q = rng.integers(-2, 3, 5).astype(np.float32)
    ids, sc = po.dense_ranking(q, V)
    exact = [exact_dot(q, V[i]) for i in range(40)]
    expected = sorted(range(40), key=lambda i: (-exact[i], i))
    assert ids.tolist() == expected
    assert all(sc[k] == f32_round_exact(exact[ids[k]]) for k in range(40))
    vis = np.ones(40, bool)
    vis[::3] = False
    ids2, _ = po.dense_ranking(q, V, vis)
    assert ids2.tolist() == [i for i in expected if vis[i]]


# ---------------------------------------------------------------------------
# scalar-quantization intervals (one scale for the corpus; ablation of
# Sec. 3.5 / 4.4, reading of this library)
# ---------------------------------------------------------------------------

def test_global_scale_is_f32_of_corpus_maxabs_over_127():
    rng = np.random.default_rng(61)
    V = (rng.standard_normal((40, 24)) * rng.gamma(1.0, 2.0, size=(40, 1))).astype(np.float32)
    s = po.global_scale(V)
    mx = Fraction(float(np.abs(V).max()))
    # s = RN_f32(mx / 127): the float32 nearest to the exact quotient
    cands = sorted({np.float32(float(mx / 127)), np.nextafter(np.float32(float(mx / 127)), 0),
                    np.nextafter(np.float32(float(mx / 127)), np.inf)},
                   key=lambda c: (abs(Fraction(float(c)) - mx / 127), int(np.float32(c).view(np.uint32)) & 1))
    assert s == cands[0]
    assert po.global_scale(np.zeros((3, 5), np.float32)) == np.float32(1.0)
    bad = V.copy()
    bad[3, 4] = np.inf
    assert np.isnan(po.global_scale(bad))


def test_global_quantization_reduces_to_per_vector_when_every_row_has_the_corpus_max():
    # rows with one common infinity norm: the global scale is every row's own
    # scale, so codes, residual bounds and intervals coincide with Sec. 2.3.1
    rng = np.random.default_rng(62)
    V = rng.standard_normal((64, 32)).astype(np.float32)
    V /= np.abs(V).max(axis=1, keepdims=True)
    V[np.arange(64), rng.integers(0, 32, 64)] = np.where(rng.random(64) < 0.5, 1.0, -1.0)
    Qp = po.quantize(V)
    Qg = po.quantize_global(V)
    assert Qg.status == 0
    assert np.array_equal(Qp.s, Qg.s)
    assert np.array_equal(Qp.z, Qg.z)
    assert np.array_equal(Qp.vnorm.view(np.uint32), Qg.vnorm.view(np.uint32))
    assert np.array_equal(Qp.enorm.view(np.uint32), Qg.enorm.view(np.uint32))


@pytest.mark.parametrize("seed", [63, 64])
def test_global_quantization_intervals_contain_the_exact_scores(seed):
    rng = np.random.default_rng(seed)
    m = 48
    # rows of very different norms: the global scale is coarse for the small ones
    V = (rng.standard_normal((300, m)) * rng.gamma(0.7, 1.0, size=(300, 1))).astype(np.float32)
    q = rng.standard_normal(m).astype(np.float32)
    Qg = po.quantize_global(V)
    assert Qg.status == 0
    qe = po.encode_query(q)
    lo, hi = po.intervals(qe, Qg, m)
    s = po.exact_scores(q, V)
    assert np.all(lo <= s) and np.all(s <= hi)
    # coarser codes, wider intervals than per-vector quantization on average
    lo_p, hi_p = po.intervals(qe, po.quantize(V), m)
    assert np.mean(hi - lo) > np.mean(hi_p - lo_p)
    # a row of all-small entries has all-zero codes and its residual is itself
    tiny = np.full((1, m), 1e-3 * float(po.global_scale(V)), np.float32)
    Qt = po.quantize_global(tiny, s=po.global_scale(V))
    assert Qt.status == 0 and not Qt.z.any()
    assert Qt.enorm[0] == Qt.vnorm[0]


def test_global_quantization_rejects_rows_outside_the_range():
    V = np.array([[1.0, -0.5, 0.25]], np.float32)
    s = po.global_scale(V)
    ok = po.quantize_global(np.array([[1.0, 0.0, 0.0]], np.float32), s=s)
    assert ok.status == 0 and ok.z[0, 0] == 127
    out = po.quantize_global(np.array([[1.5, 0.0, 0.0]], np.float32), s=s)
    assert out.status == 3
