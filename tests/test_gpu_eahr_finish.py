"""EAHR_POLICY_ADAPTIVE's exact finishes against the oracle's complete-list
fusion (arXiv 2608.07152 Sec. 2.1 T*_K, Sec. 2.2 bounds and its last
paragraph).

After some geometric reading the driver takes LB, the K-th largest lower
bound L(x) over the items read; only the items with U(x) >= LB can still be
in T*_K.  Their missing ranks come from the device: a dense rank by counting
the rows above the item's authoritative score (each row's interval decides
unless the score lies inside it, then the row is scored exactly), a sparse
rank from the host list; the rank intervals the bounds alone give often
order the candidates already (an F known only as an interval is reported as
NaN, its position certified), else the rows in question are scored.  Every
case compares the ordered Top-K ids and every reported F (correctly
rounded) with the oracle, and checks which finish ran
(stats["complete"]: 0 certified by reading; 2 rank intervals from the
bounds, 3 exact ranks; 1 complete-list fusion, the finish of a cursor
without bounds of every row).
"""
from fractions import Fraction

import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po
from oracle import rrf_oracle as ro

pytestmark = pytest.mark.gpu

M, N = 192, 120_011


@pytest.fixture(scope="module")
def corpus():
    centres = synth.mixture_centres(256, M, seed=301, device="cpu")
    V = synth.mixture_rows(N, centres, 0.35, seed=302).numpy()
    Q = synth.mixture_queries(6, centres, 0.5, seed=303).numpy()
    index = pvs.pvs_build(V)
    yield V, Q, index
    pvs.pvs_index_free(index)


def _sparse(dense_ids, dense_sc, tau, seed, keep=None):
    proxy = torch.from_numpy(dense_sc[np.argsort(dense_ids)].astype(np.float64))
    order = synth.copula_ranking(proxy, tau, seed=seed).numpy()
    if keep is not None:
        order = order[np.isin(order, keep)]
    return order.astype(np.int64)


def _check(got, F, T):
    assert got.tolist() == [x for x, _ in T]
    for (x, f), v in zip(T, F):
        if not np.isnan(v):
            assert v == ro.as_float(f)


def _run(index, q, sparse, snap=None, step=16, **kw):
    """Adaptive EAHR; step = 16 keeps geometric pulls small, so that the
    lists are read to the finish threshold before certification could end the
    request (step = 0, the default, reads 2^11 ranks per list at once)."""
    cur = pvs.pvs_cursor_open(index, q, snap)
    try:
        return pvs.eahr_topk(cur, sparse, policy=pvs.EAHR_POLICY_ADAPTIVE, step=step, **kw)
    finally:
        pvs.pvs_cursor_close(cur)


@pytest.mark.parametrize("tau", [0.5, 0.0, -0.5, -1.0])
def test_rank_query_finish_matches_complete_list_fusion(corpus, tau):
    V, Q, index = corpus
    q = Q[0]
    dense_ids, dense_sc = po.dense_ranking(q, V)
    sparse = _sparse(dense_ids, dense_sc, tau, 310)
    T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
    ids, F, st = _run(index, q, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR)
    _check(ids, F, T)
    assert st["complete"] in (0, 2, 3)
    if tau <= 0:
        assert st["complete"] in (2, 3)
        assert st["depth"][0] + st["depth"][1] < N   # finished well before the end
    # the default first pull (2^11 ranks per list): the same result
    ids, F, st = _run(index, q, sparse, step=0, K=20, k=60, form=pvs.EAHR_NUMERATOR)
    _check(ids, F, T)
    assert st["complete"] in (0, 2, 3)


@pytest.mark.parametrize("K,weights,form", [
    (1, (1, 1), pvs.EAHR_NUMERATOR),
    (100, (1, 1), pvs.EAHR_NUMERATOR),
    (20, ((3, 2), (1, 3)), pvs.EAHR_RANK_SCALED),
    (20, ((1, 7), 1), pvs.EAHR_NUMERATOR),
    (20, (5, (1, 2)), pvs.EAHR_RANK_SCALED),
])
def test_rank_query_finish_sizes_weights_and_forms(corpus, K, weights, form):
    V, Q, index = corpus
    q = Q[1]
    dense_ids, dense_sc = po.dense_ranking(q, V)
    sparse = _sparse(dense_ids, dense_sc, 0.0, 311)
    oform = ro.NUMERATOR if form == pvs.EAHR_NUMERATOR else ro.RANK_SCALED
    ow = [w if np.isscalar(w) else Fraction(*w) for w in weights]
    T = ro.target_topk_large([dense_ids, sparse], ow, 60, K, oform)
    ids, F, st = _run(index, q, sparse, K=K, k=60, form=form, weights=weights)
    _check(ids, F, T)
    assert st["complete"] in (2, 3)


def test_rank_query_finish_with_a_partial_sparse_support(corpus):
    """U_s a third of the items (Sec. 2.1: the others contribute nothing)."""
    V, Q, index = corpus
    q = Q[2]
    dense_ids, dense_sc = po.dense_ranking(q, V)
    keep = np.random.default_rng(312).choice(N, N // 3, replace=False)
    sparse = _sparse(dense_ids, dense_sc, -0.5, 313, keep=keep)
    T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
    ids, F, st = _run(index, q, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR)
    _check(ids, F, T)
    assert st["complete"] in (2, 3)


def test_rank_query_finish_on_a_snapshot_with_deletions_and_appends():
    m, n0 = 128, 60_000
    centres = synth.mixture_centres(128, m, seed=320, device="cpu")
    V = synth.mixture_rows(n0 + 20_000, centres, 0.35, seed=321).numpy()
    q = synth.mixture_queries(1, centres, 0.5, seed=322).numpy()[0]
    index = pvs.pvs_build(V[:n0])
    try:
        pvs.pvs_append(index, V[n0:])
        dead = np.random.default_rng(323).choice(n0 + 20_000, 7_000, replace=False)
        pvs.pvs_tombstone(index, dead)
        snap = pvs.pvs_snapshot_create(index)
        try:
            visible = np.ones(n0 + 20_000, bool)
            visible[dead] = False
            dense_ids, dense_sc = po.dense_ranking(q, V, visible=visible)
            for tau, seed in ((0.0, 324), (-0.5, 325)):
                order = synth.copula_ranking(torch.from_numpy(dense_sc.astype(np.float64)),
                                             tau, seed=seed).numpy()
                sparse = dense_ids[order]
                T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
                ids, F, st = _run(index, q, sparse, snap=snap, K=20, k=60,
                                  form=pvs.EAHR_NUMERATOR)
                _check(ids, F, T)
                assert st["complete"] in (2, 3)
        finally:
            pvs.pvs_snapshot_free(snap)
    finally:
        pvs.pvs_index_free(index)


def test_exact_ranks_decide_fused_ties(corpus):
    """The sparse list is the dense ranking reversed: x at dense rank i has
    sparse rank N + 1 - i, so every fused value is shared by two items and
    ties go to the smaller id (Sec. 2.1).  Rank intervals cannot settle such
    a tie; the rows around each score are scored and every F is exact."""
    V, Q, index = corpus
    q = Q[4]
    dense_ids, _ = po.dense_ranking(q, V)
    sparse = dense_ids[::-1].copy()
    for K in (20, 7):
        T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, K, ro.NUMERATOR)
        assert T[0][1] == T[1][1]                      # tied pairs
        ids, F, st = _run(index, q, sparse, K=K, k=60, form=pvs.EAHR_NUMERATOR)
        _check(ids, F, T)
        assert st["complete"] == 3
        assert not np.isnan(F).any()


def test_complete_list_fusion_finish_and_many_candidates(corpus):
    """A full-scan cursor keeps no bounds of every row, so the finish is
    complete-list fusion; K = 3,000 (candidates beyond one rank query at
    first) ends either way with the oracle's T*_K."""
    V, Q, index = corpus
    q = Q[3]
    dense_ids, dense_sc = po.dense_ranking(q, V)
    sparse = _sparse(dense_ids, dense_sc, -0.5, 314)
    T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
    cur = pvs.pvs_cursor_open(index, q)
    try:
        pvs.pvs_cursor_set_generator(cur, pvs.PVS_GEN_FULL_SCAN)
        ids, F, st = pvs.eahr_topk(cur, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR,
                                   policy=pvs.EAHR_POLICY_ADAPTIVE, step=16)
    finally:
        pvs.pvs_cursor_close(cur)
    _check(ids, F, T)
    assert st["complete"] == 1
    T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 3000, ro.NUMERATOR)
    ids, F, st = _run(index, q, sparse, K=3000, k=60, form=pvs.EAHR_NUMERATOR)
    _check(ids, F, T)
    assert st["complete"] in (1, 2, 3)


def test_rank_query_finish_on_grouped_cursors_and_a_bad_sparse_list(corpus):
    """Cursors from one grouped interval pass; then a repeated id far down
    the sparse list, which the finish reads when it needs a sparse rank."""
    V, Q, index = corpus
    Qg = Q[2:6]
    refs = []
    for i in range(4):
        dense_ids, dense_sc = po.dense_ranking(Qg[i], V)
        sparse = _sparse(dense_ids, dense_sc, -0.5, 330 + i)
        refs.append((sparse, ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20,
                                                  ro.NUMERATOR)))
    curs = pvs.pvs_cursor_open_group(index, Qg)
    try:
        for c, (sparse, T) in zip(curs, refs):
            ids, F, st = pvs.eahr_topk(c, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR,
                                       policy=pvs.EAHR_POLICY_ADAPTIVE, step=16)
            _check(ids, F, T)
            assert st["complete"] in (2, 3)
    finally:
        for c in curs:
            pvs.pvs_cursor_close(c)
    bad = refs[0][0].copy()
    bad[-1] = bad[0]
    with pytest.raises(pvs.PvsError) as e:
        _run(index, Qg[0], bad, K=20, k=60, form=pvs.EAHR_NUMERATOR)
    assert e.value.status == pvs.PVS_ERR_INVALID


def test_exact_count_near_equal_scores():
    """Rows whose scores sit within a few ulps of a candidate's: exact copies
    of the top rows (equal scores, ids decide) and copies perturbed by 1e-7.
    The bounded fp32 dot cannot place them, so the error-free dot must; the
    reversed sparse list makes every finish take exact ranks."""
    rng = np.random.default_rng(340)
    m, base_n = 64, 30_000
    V = synth.unit_normal(base_n, m, seed=341).numpy()
    q = synth.unit_normal(1, m, seed=342).numpy()[0]
    ids0, _ = po.dense_ranking(q, V)
    bottom = ids0[-40:]                      # the sparse list's top items
    copies = np.repeat(V[bottom], 3, axis=0)
    near = copies + (1e-7 * rng.standard_normal(copies.shape)).astype(np.float32)
    W = np.concatenate([V, copies, near]).astype(np.float32)
    W = W[rng.permutation(W.shape[0])]
    dense_ids, _ = po.dense_ranking(q, W)
    sparse = dense_ids[::-1].copy()
    T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
    index = pvs.pvs_build(W)
    try:
        ids, F, st = _run(index, q, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR)
    finally:
        pvs.pvs_index_free(index)
    _check(ids, F, T)
    assert st["complete"] == 3
    assert not np.isnan(F).any()


def _tied_mid_sparse(dense_ids, pairs, rng):
    """A sparse list whose first `pairs` items lie in the middle of the dense
    ranking (B_k), with the dense top item A_k placed at B_k's dense rank:
    F(A_k) = F(B_k) exactly, so only exact dense ranks of mid-distribution
    scores order each pair (ties: smaller id first)."""
    n = len(dense_ids)
    mid = n // 2
    B = dense_ids[mid - 5 * pairs:mid + 5 * pairs:10][:pairs]
    A = dense_ids[:pairs]
    rank = np.empty(int(dense_ids.max()) + 1, np.int64)
    rank[dense_ids] = np.arange(1, n + 1)
    S = np.full(n, -1, np.int64)
    S[:pairs] = B
    S[rank[B] - 1] = A
    used = np.zeros(rank.shape[0], bool)
    used[A] = used[B] = True
    rest = dense_ids[~used[dense_ids]].copy()
    rng.shuffle(rest)
    S[S < 0] = rest
    return S


def test_exact_ranks_of_mid_scores_through_the_residual_codes():
    """Exact dense ranks of items in the middle of the score distribution,
    where a third of the rows' intervals straddle each score: the residual
    codes place all but a few of those rows without their fp32 rows (the
    refined count stays far below the straddlers), and the codes are
    extended over rows appended after they were first built."""
    rng = np.random.default_rng(350)
    m, n0, n1 = 128, 50_000, 12_000
    centres = synth.mixture_centres(64, m, seed=351, device="cpu")
    V = synth.mixture_rows(n0, centres, 0.35, seed=352).numpy()
    q = synth.mixture_queries(1, centres, 0.5, seed=353).numpy()[0]
    pairs = 10
    index = pvs.pvs_build(V)
    try:
        dense_ids, _ = po.dense_ranking(q, V)
        S = _tied_mid_sparse(dense_ids, pairs, rng)
        T = ro.target_topk_large([dense_ids, S], [1, 1], 60, 2 * pairs, ro.NUMERATOR)
        assert T[0][1] == T[1][1]
        cur = pvs.pvs_cursor_open(index, q)
        try:
            ids, F, st = pvs.eahr_topk(cur, S, K=2 * pairs, k=60, form=pvs.EAHR_NUMERATOR,
                                       policy=pvs.EAHR_POLICY_ADAPTIVE)
            refined = pvs.pvs_cursor_stats(cur)["refined"]
        finally:
            pvs.pvs_cursor_close(cur)
        _check(ids, F, T)
        assert st["complete"] == 3
        assert not np.isnan(F).any()
        assert refined < n0 // 8, refined
        # rows near the middle scores appended after the codes were built,
        # some rows deleted; a snapshot sees both
        W = V[dense_ids[n0 // 2 - n1 // 2:n0 // 2 + n1 // 2]]
        W = (W + 1e-3 * rng.standard_normal(W.shape)).astype(np.float32)
        pvs.pvs_append(index, W)
        U = np.concatenate([V, W])
        dead = rng.choice(n0 + n1, 2_000, replace=False)
        pvs.pvs_tombstone(index, dead)
        visible = np.ones(n0 + n1, bool)
        visible[dead] = False
        snap = pvs.pvs_snapshot_create(index)
        try:
            dense_ids, _ = po.dense_ranking(q, U, visible=visible)
            S = _tied_mid_sparse(dense_ids, pairs, rng)
            T = ro.target_topk_large([dense_ids, S], [1, 1], 60, 2 * pairs, ro.NUMERATOR)
            ids, F, st = _run(index, q, S, snap=snap, step=0, K=2 * pairs, k=60,
                              form=pvs.EAHR_NUMERATOR)
            _check(ids, F, T)
            assert st["complete"] == 3
            assert not np.isnan(F).any()
        finally:
            pvs.pvs_snapshot_free(snap)
    finally:
        pvs.pvs_index_free(index)


@pytest.mark.parametrize("m", [4096, 4200])
def test_exact_ranks_at_the_widest_residual_rows_and_beyond(m):
    """m_pad = 4096, the widest rows given residual codes (16 KB of query
    codes in shared memory), and m_pad = 4224, whose exact counts read the
    fp32 rows of every straddling row: the same exact ranks either way."""
    rng = np.random.default_rng(360 + m)
    n, pairs = 6_000, 6
    V = synth.unit_normal(n, m, seed=361 + m).numpy()
    q = synth.unit_normal(1, m, seed=362 + m).numpy()[0]
    dense_ids, _ = po.dense_ranking(q, V)
    S = _tied_mid_sparse(dense_ids, pairs, rng)
    T = ro.target_topk_large([dense_ids, S], [1, 1], 60, 2 * pairs, ro.NUMERATOR)
    index = pvs.pvs_build(V)
    try:
        ids, F, st = _run(index, q, S, step=0, K=2 * pairs, k=60, form=pvs.EAHR_NUMERATOR)
    finally:
        pvs.pvs_index_free(index)
    _check(ids, F, T)
    assert st["complete"] == 3
    assert not np.isnan(F).any()
