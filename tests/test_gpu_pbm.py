"""PBM sparse rank generator through the C ABI against the oracle
(arXiv 2608.07152 Sec. 2.1, Sec. 2.3.2, Sec. 2.4, App. A.2).

Every emitted rank and score is compared bit for bit with the oracle's
complete sparse ranked list, whose support U_s is the items with a positive
score (Sec. 2.1); the range bounds with the oracle's H_hat(R).
"""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pbm_oracle as po
from oracle import pvs_oracle as pvo
from oracle import rrf_oracle as ro

pytestmark = pytest.mark.gpu


def csr(n_terms, postings):
    off, docs, imps = [0], [], []
    for t in range(n_terms):
        for d, p in postings.get(t, []):
            docs.append(d)
            imps.append(p)
        off.append(len(docs))
    return np.array(off, np.int64), np.array(docs, np.int32), np.array(imps, np.float32)


def random_postings(rng, n_items, n_terms, max_df, integer=False):
    postings = {}
    for t in range(n_terms):
        k = int(rng.integers(0, max_df + 1))
        if k == 0:
            continue
        d = np.sort(rng.choice(n_items, size=min(k, n_items), replace=False))
        p = (rng.integers(1, 4, size=d.size).astype(np.float32) if integer
             else rng.gamma(2.0, 1.1, size=d.size).astype(np.float32))
        postings[t] = list(zip(d.tolist(), p.tolist()))
    return csr(n_terms, postings)


def pull_all(cur, chunks, n_support):
    ids, sc = [], []
    k = 0
    while True:
        n = chunks[k % len(chunks)]
        k += 1
        i, s, st = pvs.pbm_next(cur, n)
        ids.append(i)
        sc.append(s)
        if st == pvs.PVS_EXHAUSTED:
            assert sum(len(x) for x in ids) == n_support
            break
        assert len(i) == n
    # an exhausted list stays exhausted and delivers nothing
    i, s, st = pvs.pbm_next(cur, 5)
    assert st == pvs.PVS_EXHAUSTED and len(i) == 0
    return np.concatenate(ids), np.concatenate(sc)


def check_against_oracle(off, docs, imps, n_items, terms, weights, block, chunks):
    ref_ids, ref_sc = po.sparse_ranking(terms, weights, off, docs, imps, n_items)
    index = pvs.pbm_build(off, docs, imps, n_items, block=block)
    try:
        cur = pvs.pbm_cursor_open(index, terms, weights)
        try:
            nr = pvs.pbm_index_ranges(index)
            H = pvs.pbm_cursor_range_bounds(cur, 0, nr)
            ref_H = po.range_bounds(terms, weights, off, docs, imps, n_items, block)
            assert np.array_equal(H.view(np.uint32), ref_H.view(np.uint32))
            ids, sc = pull_all(cur, chunks, len(ref_ids))
            stats = pvs.pbm_cursor_stats(cur)
        finally:
            pvs.pbm_cursor_close(cur)
    finally:
        pvs.pbm_index_free(index)
    assert np.array_equal(ids, ref_ids)
    assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
    assert stats["emitted"] == len(ref_ids) and stats["state"] == pvs.PVS_EXHAUSTED
    # only ranges with a positive bound are expanded (S <= H: the others hold
    # no item of U_s)
    assert stats["ranges_expanded"] == int(np.count_nonzero(ref_H > 0))
    return stats


def test_hand_worked_case():
    off, docs, imps = csr(3, {0: [(0, 1.5), (2, 0.5), (4, 3.0)], 1: [(3, 7.0)],
                              2: [(0, 4.0), (1, 2.0)]})
    check_against_oracle(off, docs, imps, 6, [0, 2], [2.0, 0.5], 2, [1])
    check_against_oracle(off, docs, imps, 6, [2, 0], [0.5, 2.0], 4, [4])


@pytest.mark.parametrize("block", [1, 2, 7, 16, 128, 4096])
def test_random_instances_every_block_size(block):
    rng = np.random.default_rng(100 + block)
    for trial in range(3):
        n_items = int(rng.integers(50, 3000))
        n_terms = 40
        off, docs, imps = random_postings(rng, n_items, n_terms, max_df=n_items // 3)
        nq = int(rng.integers(1, 9))
        terms = rng.choice(n_terms, size=nq, replace=False).astype(np.int32)
        weights = rng.gamma(1.5, 0.8, size=nq).astype(np.float32)
        chunks = [int(x) for x in rng.integers(1, 300, size=5)]
        check_against_oracle(off, docs, imps, n_items, terms, weights, block, chunks)


def test_ties_zero_weights_and_empty_terms():
    rng = np.random.default_rng(7)
    n_items, n_terms = 1500, 30
    off, docs, imps = random_postings(rng, n_items, n_terms, max_df=400, integer=True)
    # integer impacts and weights: many exactly tied scores, ordered by id
    terms = np.array([3, 11, 0, 25], np.int32)
    check_against_oracle(off, docs, imps, n_items, terms, np.ones(4, np.float32), 16, [37, 5])
    # a zero weight contributes nothing; a term without postings neither
    empty = [t for t in range(n_terms) if off[t] == off[t + 1]]
    terms2 = np.array([3, 11] + empty[:1], np.int32)
    w2 = np.array([0.0, 2.0] + [1.0] * len(empty[:1]), np.float32)
    check_against_oracle(off, docs, imps, n_items, terms2, w2, 64, [100])
    # no query terms, or only zero weights: every score is 0, U_s is empty
    check_against_oracle(off, docs, imps, n_items, np.zeros(0, np.int32),
                         np.zeros(0, np.float32), 16, [999])
    check_against_oracle(off, docs, imps, n_items, np.array([3, 11], np.int32),
                         np.zeros(2, np.float32), 16, [1])
    # every item in U_s: one term posted on every item
    full = csr(2, {0: [(x, 1.0 + (x % 5)) for x in range(700)], 1: [(3, 2.0)]})
    check_against_oracle(*full, 700, np.array([0], np.int32), np.ones(1, np.float32), 32,
                         [700])
    check_against_oracle(*full, 700, np.array([0], np.int32), np.ones(1, np.float32), 32,
                         [699, 1, 5])


def test_bm25_corpus_deep_pulls_and_large_windows():
    n_items, n_terms = 150_000, 20_000
    off, docs, imps = synth.bm25_postings(n_items, n_terms, 30.0, seed=21)
    off, docs, imps = off.numpy(), docs.numpy(), imps.numpy()
    queries = synth.sparse_queries(3, torch.from_numpy(off), seed=22, mean_terms=5.0)
    for qi, (terms, weights) in enumerate(queries):
        # chunks of 20, then large pulls (windows above the sort-everything
        # size go through the 64-bit selection)
        stats = check_against_oracle(off, docs, imps, n_items, terms, weights, 128,
                                     [20] * 50 + [70_000, 100_000])
        q_postings = sum(int(off[t + 1] - off[t]) for t in terms)
        assert stats["postings_visited"] == q_postings      # every posting once, at the end
        H = po.range_bounds(terms, weights, off, docs, imps, n_items, 128)
        sizes = np.minimum(128, n_items - 128 * np.arange(H.size))
        assert stats["items_scored"] == int(sizes[H > 0].sum())
        # pulls of 20 inside an earlier pull's certified window need no device work
        assert stats["pulls_from_window"] > 0


def test_first_ranks_touch_few_ranges():
    n_items, n_terms = 400_000, 30_000
    off, docs, imps = synth.bm25_postings(n_items, n_terms, 30.0, seed=31)
    off, docs, imps = off.numpy(), docs.numpy(), imps.numpy()
    terms, weights = synth.sparse_queries(1, torch.from_numpy(off), seed=32, mean_terms=4.0)[0]
    ref_ids, ref_sc = po.sparse_ranking(terms, weights, off, docs, imps, n_items)
    index = pvs.pbm_build(torch.from_numpy(off).cuda(), torch.from_numpy(docs).cuda(),
                          torch.from_numpy(imps).cuda(), n_items)
    try:
        cur = pvs.pbm_cursor_open(index, terms, weights)
        try:
            got_i, got_s = [], []
            for _ in range(10):
                i, s, st = pvs.pbm_next(cur, 20)
                assert st == pvs.PVS_OK and len(i) == 20
                got_i.append(i)
                got_s.append(s)
            stats = pvs.pbm_cursor_stats(cur)
        finally:
            pvs.pbm_cursor_close(cur)
    finally:
        pvs.pbm_index_free(index)
    assert np.array_equal(np.concatenate(got_i), ref_ids[:200])
    assert np.array_equal(np.concatenate(got_s).view(np.uint32), ref_sc[:200].view(np.uint32))
    # the bounds let PBM leave most ranges unexpanded for a short prefix
    assert stats["ranges_expanded"] < stats["ranges"]


def test_invalid_inputs_fail_loudly():
    off, docs, imps = csr(2, {0: [(1, 1.0), (3, 2.0)], 1: [(0, 0.5)]})
    def build_err(o, d, p, n=4, block=0):
        with pytest.raises(pvs.PvsError) as e:
            pvs.pbm_build(o, d, p, n, block=block)
        return e.value.status
    assert build_err(off, docs, np.array([1.0, -1.0, 0.5], np.float32)) == pvs.PVS_ERR_INVALID
    assert build_err(off, docs, np.array([1.0, np.nan, 0.5], np.float32)) == pvs.PVS_ERR_NONFINITE
    assert build_err(off, np.array([3, 1, 0], np.int32), imps) == pvs.PVS_ERR_INVALID
    assert build_err(off, docs, imps, n=3) == pvs.PVS_ERR_INVALID           # id 3 out of range
    assert build_err(np.array([0, 3, 2], np.int64), docs, imps) == pvs.PVS_ERR_INVALID
    assert build_err(off, docs, imps, block=5000) == pvs.PVS_ERR_INVALID
    index = pvs.pbm_build(off, docs, imps, 4)
    try:
        for terms, w, code in (([0, 0], [1.0, 1.0], pvs.PVS_ERR_INVALID),
                               ([0, 2], [1.0, 1.0], pvs.PVS_ERR_INVALID),
                               ([0], [-1.0], pvs.PVS_ERR_INVALID),
                               ([1], [float("inf")], pvs.PVS_ERR_NONFINITE)):
            with pytest.raises(pvs.PvsError) as e:
                pvs.pbm_cursor_open(index, terms, w)
            assert e.value.status == code
        cur = pvs.pbm_cursor_open(index, [0, 1], [1.0, 1.0])
        try:
            with pytest.raises(pvs.PvsError):
                pvs.pbm_next(cur, 0)
            i, s, st = pvs.pbm_next(cur, 10)
            # item 2 has no posting: score 0, outside U_s
            assert st == pvs.PVS_EXHAUSTED and i.tolist() == [3, 1, 0]
            i, s, st = pvs.pbm_next(cur, 10)
            assert st == pvs.PVS_EXHAUSTED and len(i) == 0
        finally:
            pvs.pbm_cursor_close(cur)
    finally:
        pvs.pbm_index_free(index)


@pytest.mark.parametrize("tau_terms", [3, 6])
def test_eahr_with_pbm_matches_complete_list_fusion(tau_terms):
    n, m = 30_000, 64
    V = synth.unit_normal(n, m, seed=41).numpy()
    q = synth.unit_normal(1, m, seed=42).numpy()[0]
    off, docs, imps = synth.bm25_postings(n, 5_000, 25.0, seed=43)
    off, docs, imps = off.numpy(), docs.numpy(), imps.numpy()
    terms, weights = synth.sparse_queries(1, torch.from_numpy(off), seed=44,
                                          mean_terms=float(tau_terms))[0]
    dense_ids, _ = pvo.dense_ranking(q, V)
    sparse_ids, _ = po.sparse_ranking(terms, weights, off, docs, imps, n)
    T = ro.target_topk_large([dense_ids, sparse_ids], [1, 1], 60, 20, ro.NUMERATOR)
    dindex = pvs.pvs_build(V)
    sindex = pvs.pbm_build(off, docs, imps, n)
    try:
        dcur = pvs.pvs_cursor_open(dindex, q)
        scur = pvs.pbm_cursor_open(sindex, terms, weights)
        try:
            ids, F, st = pvs.eahr_topk_pbm(dcur, scur, K=20, k=60, form=pvs.EAHR_NUMERATOR)
        finally:
            pvs.pbm_cursor_close(scur)
            pvs.pvs_cursor_close(dcur)
    finally:
        pvs.pbm_index_free(sindex)
        pvs.pvs_index_free(dindex)
    assert ids.tolist() == [x for x, _ in T]
    for (x, f), got in zip(T, F):
        if not np.isnan(got):
            assert got == ro.as_float(f)


def _eahr_pbm(V, q, off, docs, imps, n, terms, weights, snap_ids=None,
              policy=pvs.EAHR_POLICY_GEOMETRIC, step=0):
    """eahr_topk_pbm over a fresh PVS index of V and PBM index of the postings;
    snap_ids: ids to delete in a snapshot that both cursors see."""
    dindex = pvs.pvs_build(V)
    sindex = pvs.pbm_build(off, docs, imps, n)
    snap = None
    try:
        if snap_ids is not None:
            pvs.pvs_tombstone(dindex, snap_ids)
            snap = pvs.pvs_snapshot_create(dindex)
        dcur = pvs.pvs_cursor_open(dindex, q, snap=snap)
        scur = pvs.pbm_cursor_open(sindex, terms, weights, snap=snap)
        try:
            return pvs.eahr_topk_pbm(dcur, scur, K=20, k=60, form=pvs.EAHR_NUMERATOR,
                                     policy=policy, step=step)
        finally:
            pvs.pbm_cursor_close(scur)
            pvs.pvs_cursor_close(dcur)
    finally:
        if snap is not None:
            pvs.pvs_snapshot_free(snap)
        pvs.pbm_index_free(sindex)
        pvs.pvs_index_free(dindex)


def test_eahr_over_the_positive_score_support_differs_from_ranking_every_item():
    """Sec. 2.1: the sparse channel ranks only U_s = {S > 0}; an item outside
    it contributes nothing.  With BM25 queries of 1-3 terms U_s is a small
    part of the corpus, and ranking every item (zero scores last, by id)
    would hand each zero-score item a spurious 1 / (60 + r): the two targets
    differ, and EAHR must return the one over U_s."""
    n, m = 40_000, 64
    V = synth.unit_normal(n, m, seed=51).numpy()
    Q = synth.unit_normal(6, m, seed=52).numpy()
    off, docs, imps = synth.bm25_postings(n, 8_000, 25.0, seed=53)
    off, docs, imps = off.numpy(), docs.numpy(), imps.numpy()
    queries = synth.sparse_queries(6, torch.from_numpy(off), seed=54, mean_terms=1.0)
    differ = 0
    for qi, (terms, weights) in enumerate(queries):
        terms, weights = terms[:3], weights[:3]
        dense_ids, _ = pvo.dense_ranking(Q[qi], V)
        sparse_ids, _ = po.sparse_ranking(terms, weights, off, docs, imps, n)
        assert 0 < sparse_ids.size < n // 4
        T = ro.target_topk_large([dense_ids, sparse_ids], [1, 1], 60, 20, ro.NUMERATOR)
        S = po.sparse_scores(terms, weights, off, docs, imps, n)
        every = np.concatenate([sparse_ids, np.nonzero(S == 0)[0]])   # zero scores last, by id
        T_every = ro.target_topk_large([dense_ids, every], [1, 1], 60, 20, ro.NUMERATOR)
        differ += [x for x, _ in T] != [x for x, _ in T_every]
        ids, F, st = _eahr_pbm(V, Q[qi], off, docs, imps, n, terms, weights)
        assert ids.tolist() == [x for x, _ in T]
        for (x, f), got in zip(T, F):
            if not np.isnan(got):
                assert got == ro.as_float(f)
        assert st["length"][1] == sparse_ids.size or not st["exhausted"][1]
    assert differ > 0


def test_pbm_on_a_snapshot_with_deletions():
    """Sec. 2.4: both channels of a request rank one fixed snapshot.  A PBM
    cursor opened on a PVS snapshot leaves deleted items out of its list,
    and EAHR over the two matches complete-list fusion of the visible items."""
    n, m = 30_000, 64
    rng = np.random.default_rng(61)
    V = synth.unit_normal(n, m, seed=62).numpy()
    q = synth.unit_normal(1, m, seed=63).numpy()[0]
    off, docs, imps = synth.bm25_postings(n, 5_000, 25.0, seed=64)
    off, docs, imps = off.numpy(), docs.numpy(), imps.numpy()
    terms, weights = synth.sparse_queries(1, torch.from_numpy(off), seed=65, mean_terms=4.0)[0]
    S = po.sparse_scores(terms, weights, off, docs, imps, n)
    # delete 5 % of the items, among them the ten best sparse ones
    dead = np.unique(np.concatenate([rng.choice(n, n // 20, replace=False),
                                     po.sparse_ranking(terms, weights, off, docs, imps, n)[0][:10]]))
    visible = np.ones(n, bool)
    visible[dead] = False
    ref_ids, ref_sc = po.sparse_ranking(terms, weights, off, docs, imps, n)
    keep = visible[ref_ids]
    ref_ids, ref_sc = ref_ids[keep], ref_sc[keep]
    dindex = pvs.pvs_build(V)
    sindex = pvs.pbm_build(off, docs, imps, n, block=64)
    try:
        pvs.pvs_tombstone(dindex, dead)
        snap = pvs.pvs_snapshot_create(dindex)
        try:
            cur = pvs.pbm_cursor_open(sindex, terms, weights, snap=snap)
            try:
                ids, sc = pull_all(cur, [20, 333], len(ref_ids))
            finally:
                pvs.pbm_cursor_close(cur)
            # a cursor without the snapshot does not see the same items
            dcur = pvs.pvs_cursor_open(dindex, q, snap=snap)
            scur = pvs.pbm_cursor_open(sindex, terms, weights)
            try:
                with pytest.raises(pvs.PvsError) as e:
                    pvs.eahr_topk_pbm(dcur, scur, K=20, k=60, form=pvs.EAHR_NUMERATOR)
                assert e.value.status == pvs.PVS_ERR_INVALID
            finally:
                pvs.pbm_cursor_close(scur)
                pvs.pvs_cursor_close(dcur)
        finally:
            pvs.pvs_snapshot_free(snap)
    finally:
        pvs.pbm_index_free(sindex)
        pvs.pvs_index_free(dindex)
    assert np.array_equal(ids, ref_ids)
    assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
    dense_ids, _ = pvo.dense_ranking(q, V, visible=visible)
    T = ro.target_topk_large([dense_ids, ref_ids], [1, 1], 60, 20, ro.NUMERATOR)
    got, F, _ = _eahr_pbm(V, q, off, docs, imps, n, terms, weights, snap_ids=dead)
    assert got.tolist() == [x for x, _ in T]
    assert not visible[got].size or visible[got].all()
    assert S[dead].max() > 0      # deleted items that PBM would otherwise rank


@pytest.mark.parametrize("deleted", [False, True])
def test_eahr_pbm_adaptive_finish_matches_complete_list_fusion(deleted):
    """EAHR_POLICY_ADAPTIVE over PVS + PBM (Sec. 2.2, last paragraph): after
    2^12 ranks the candidates' missing sparse ranks come from the query's
    complete PBM ranking computed on the device (S in the query's term order,
    as the expand kernel evaluates it), the dense ones from the rows' bounds.
    Independent channels make both lists deep; with deletions both cursors
    rank one snapshot."""
    n, m = 60_000, 64
    rng = np.random.default_rng(71)
    V = synth.unit_normal(n, m, seed=72).numpy()
    Q = synth.unit_normal(3, m, seed=73).numpy()
    off, docs, imps = synth.bm25_postings(n, 6_000, 25.0, seed=74)
    off, docs, imps = off.numpy(), docs.numpy(), imps.numpy()
    queries = synth.sparse_queries(3, torch.from_numpy(off), seed=75, mean_terms=8.0)
    dead = rng.choice(n, n // 25, replace=False) if deleted else None
    visible = np.ones(n, bool)
    if deleted:
        visible[dead] = False
    finishes = []
    for qi, (terms, weights) in enumerate(queries):
        dense_ids, _ = pvo.dense_ranking(Q[qi], V, visible=visible)
        sparse_ids, _ = po.sparse_ranking(terms, weights, off, docs, imps, n)
        sparse_ids = sparse_ids[visible[sparse_ids]]
        T = ro.target_topk_large([dense_ids, sparse_ids], [1, 1], 60, 20, ro.NUMERATOR)
        for step in (16, 0):
            ids, F, st = _eahr_pbm(V, Q[qi], off, docs, imps, n, terms, weights, snap_ids=dead,
                                   policy=pvs.EAHR_POLICY_ADAPTIVE, step=step)
            assert ids.tolist() == [x for x, _ in T]
            for (x, f), got in zip(T, F):
                if not np.isnan(got):
                    assert got == ro.as_float(f)
            finishes.append(st["complete"])
    assert any(c in (2, 3) for c in finishes)


def test_pooled_cursors_on_streams_from_several_threads():
    """Closed cursors are reused by later opens (term counts that grow and
    shrink, with and without a snapshot), and cursors on their own streams
    serve queries from four host threads at once: every ranking equals the
    oracle's."""
    import threading
    n = 20_000
    off, docs, imps = synth.bm25_postings(n, 4_000, 20.0, seed=81)
    off, docs, imps = off.numpy(), docs.numpy(), imps.numpy()
    rng = np.random.default_rng(82)
    queries = []
    for k in (1, 7, 20, 3, 12, 2, 9, 5):
        terms = rng.choice(4_000, k, replace=False).astype(np.int32)
        queries.append((terms, rng.uniform(0.5, 2.0, k).astype(np.float32)))
    refs = [po.sparse_ranking(t, w, off, docs, imps, n) for t, w in queries]
    index = pvs.pbm_build(off, docs, imps, n)
    errors, results = [], {}
    try:
        def serve(k):
            try:
                torch.cuda.set_device(0)
                stream = torch.cuda.Stream()
                for j in range(k, len(queries), 4):
                    for _ in range(2):   # the second open reuses a pooled cursor
                        cur = pvs.pbm_cursor_open(index, *queries[j], stream=stream)
                        try:
                            results[(j, _)] = pull_all(cur, [20, 77], len(refs[j][0]))
                        finally:
                            pvs.pbm_cursor_close(cur)
            except Exception as e:   # reported on the main thread
                errors.append(e)
        threads = [threading.Thread(target=serve, args=(k,)) for k in range(4)]
        for t in threads:
            t.start()
        for t in threads:
            t.join()
    finally:
        pvs.pbm_index_free(index)
    assert not errors, errors
    assert len(results) == 2 * len(queries)
    for (j, _), (ids, sc) in results.items():
        ref_ids, ref_sc = refs[j]
        assert np.array_equal(ids, ref_ids)
        assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
