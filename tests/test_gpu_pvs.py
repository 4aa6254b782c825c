"""GPU parity of the PVS path against the oracle, through the C ABI.

Bars (arXiv 2608.07152 Sec. 2.1, 2.3.1, App. A.1):
  * codes, scales and norm bounds: bit-exact with the oracle quantizer;
  * intervals: bit-exact with the oracle's interval arithmetic, and sound
    (lo <= authoritative score <= hi) for every vector;
  * authoritative scores: bit-exact (both sides compute the correctly rounded
    exact inner product, so the 1e-5 relative allowance is not needed);
  * emitted ranks: identical ids in identical order (the 2^-20 near-tie swap
    allowance is not needed either: swaps are counted and must be zero).
"""
import math

import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po
from oracle import rrf_oracle as ro

pytestmark = pytest.mark.gpu


def _edge_rows(m, rng):
    rows = [np.zeros(m), np.eye(1, m, 0)[0], -np.eye(1, m, m - 1)[0]]
    r = np.zeros(m)
    r[0], r[1], r[2] = 127 / 128, 2.5 / 128, -2.5 / 128          # halfway quotients
    rows.append(r)
    r = np.zeros(m)
    r[0], r[1] = 3 * 2.0 ** -149, -(2.0 ** -149)                   # subnormal scale
    rows.append(r)
    r = np.zeros(m)
    r[0] = 190 * 2.0 ** -149                                        # clipped code
    rows.append(r)
    rows.append(rng.standard_normal(m) * 1e30)
    rows.append(rng.standard_normal(m) * 1e-30)
    rows.append(rng.integers(-3, 4, m).astype(float))
    return np.array(rows, dtype=np.float32)


def _count_swaps(got_ids, ref_ids, ref_scores_by_id):
    """Adjacent near-tie swaps against the oracle order; raises if any other
    difference exists."""
    got = list(got_ids)
    ref = list(ref_ids)
    swaps = 0
    i = 0
    while i < len(ref):
        if got[i] == ref[i]:
            i += 1
            continue
        a, b = ref[i], ref[i + 1]
        sa, sb = ref_scores_by_id[a], ref_scores_by_id[b]
        assert got[i] == b and got[i + 1] == a, f"rank {i}: {got[i]} != {ref[i]}"
        assert abs(float(sa) - float(sb)) < 2.0 ** -20 * max(abs(float(sa)), abs(float(sb)))
        swaps += 1
        i += 2
    return swaps


@pytest.mark.parametrize("m", [100, 128, 768])
def test_build_matches_oracle_quantizer(m):
    rng = np.random.default_rng(m)
    V = np.concatenate([_edge_rows(m, rng), rng.standard_normal((500, m)).astype(np.float32)])
    V = np.ascontiguousarray(V, dtype=np.float32)
    Q = po.quantize(V)
    for src in (V, torch.from_numpy(V).cuda()):
        index = pvs.pvs_build(src)
        try:
            codes, scale, vnorm, enorm = pvs.pvs_index_export(index, 0, V.shape[0])
        finally:
            pvs.pvs_index_free(index)
        assert np.array_equal(codes, Q.z)
        assert np.array_equal(scale.view(np.uint32), Q.s.view(np.uint32))
        assert np.array_equal(vnorm.view(np.uint32), Q.vnorm.view(np.uint32))
        assert np.array_equal(enorm.view(np.uint32), Q.enorm.view(np.uint32))


def test_non_finite_inputs_fail():
    V = np.ones((100, 64), np.float32)
    V[57, 3] = np.nan
    with pytest.raises(pvs.PvsError) as e:
        pvs.pvs_build(V)
    assert e.value.status == pvs.PVS_ERR_NONFINITE
    index = pvs.pvs_build(np.ones((10, 64), np.float32))
    try:
        q = np.ones(64, np.float32)
        q[0] = np.inf
        with pytest.raises(pvs.PvsError) as e:
            pvs.pvs_cursor_open(index, q)
        assert e.value.status == pvs.PVS_ERR_NONFINITE
        with pytest.raises(pvs.PvsError) as e:
            pvs.pvs_append(index, np.full((3, 64), np.nan, np.float32))
        assert e.value.status == pvs.PVS_ERR_NONFINITE
        assert pvs.pvs_index_size(index) == 10
    finally:
        pvs.pvs_index_free(index)


@pytest.mark.parametrize("n,m", [(10_037, 128), (3_005, 768), (2_111, 1024), (777, 100)])
def test_intervals_bit_exact_and_sound(n, m):
    centres = synth.mixture_centres(64, m, seed=3, device="cpu")
    V = synth.mixture_rows(n, centres, 0.35, seed=4).numpy()
    qs = synth.mixture_queries(3, centres, 0.5, seed=5).numpy()
    Q = po.quantize(V)
    index = pvs.pvs_build(V)
    try:
        for q in qs:
            qe = po.encode_query(q)
            ref_lo, ref_hi = po.intervals(qe, Q, m)
            cur = pvs.pvs_cursor_open(index, q)
            try:
                lo, hi = pvs.pvs_cursor_bounds(cur, 0, n)
            finally:
                pvs.pvs_cursor_close(cur)
            assert np.array_equal(lo.view(np.uint32), ref_lo.view(np.uint32))
            assert np.array_equal(hi.view(np.uint32), ref_hi.view(np.uint32))
            s = po.exact_scores(q, V)
            assert np.all(lo <= s) and np.all(s <= hi)
    finally:
        pvs.pvs_index_free(index)


def test_exact_scores_match_oracle_including_halfway_cases():
    m = 64
    rng = np.random.default_rng(9)
    V = rng.standard_normal((400, m)).astype(np.float32)
    V[::9] *= np.float32(1e-20)
    V[10] = -V[11]
    # rows whose exact score sits on or next to a float32 halfway point
    q = np.zeros(m, np.float32)
    q[0], q[1], q[2], q[3] = 1.0, 2.0 ** -24, 2.0 ** -60, 0.5
    specials = []
    for a, b, c in [(1, 1, 0), (1, 1, 1), (1, 1, -1), (1, 0, 0), (1, 1, 2)]:
        v = np.zeros(m, np.float32)
        v[0], v[1], v[2] = a, b, c
        specials.append(v)
    V = np.concatenate([V, np.array(specials)]).astype(np.float32)
    index = pvs.pvs_build(V)
    try:
        for query in (q, rng.standard_normal(m).astype(np.float32)):
            cur = pvs.pvs_cursor_open(index, query)
            try:
                got = pvs.pvs_cursor_score_ids(cur, np.arange(V.shape[0]))
                st = pvs.pvs_cursor_stats(cur)
            finally:
                pvs.pvs_cursor_close(cur)
            ref = po.exact_scores(query, V)
            assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))
        assert st["exact_fallbacks"] >= 0
    finally:
        pvs.pvs_index_free(index)


def test_exact_scores_at_extreme_magnitudes():
    """Rows whose float32 products overflow (but cancel) or underflow: the
    float32 error-free path must hand these to the binary64 / exact paths."""
    m = 64
    rng = np.random.default_rng(17)
    big = (rng.standard_normal((60, m)) * 1e10).astype(np.float32)
    big[:, 0], big[:, 1] = 3e19, -3e19          # products beyond float32 range cancel
    big[1, 1] = 3e19                            # exact score beyond float32 range: inf
    big[2, 0] = np.nextafter(np.float32(3e19), np.float32(np.inf))
    tiny = (rng.standard_normal((60, m)) * 2.0 ** -75).astype(np.float32)
    tiny[0] = 0.0
    tiny[0, :3] = 2.0 ** -75
    V = np.concatenate([big, tiny])
    qb = (rng.standard_normal(m) * 1e10).astype(np.float32)
    qb[0] = qb[1] = 3e19
    qb_c = (rng.standard_normal(m) * 1e19).astype(np.float32)
    qt = np.zeros(m, np.float32)
    qt[:3] = 2.0 ** -75
    qt[3:] = (rng.standard_normal(m - 3) * 2.0 ** -75).astype(np.float32)
    index = pvs.pvs_build(V)
    try:
        for query in (qb, qb_c, qt):
            cur = pvs.pvs_cursor_open(index, query)
            try:
                got = pvs.pvs_cursor_score_ids(cur, np.arange(V.shape[0]))
            finally:
                pvs.pvs_cursor_close(cur)
            ref = po.exact_scores(query, V)
            assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))
    finally:
        pvs.pvs_index_free(index)


def test_exact_fallback_path_is_taken_and_exact():
    m = 64
    q = np.zeros(m, np.float32)
    q[0], q[1], q[2] = 1.0, 2.0 ** -24, 2.0 ** -60
    V = np.zeros((3, m), np.float32)
    V[:, 0] = 1.0
    V[:, 1] = 1.0
    V[1, 2] = 1.0
    V[2, 2] = -1.0
    index = pvs.pvs_build(V)
    try:
        cur = pvs.pvs_cursor_open(index, q)
        got = pvs.pvs_cursor_score_ids(cur, np.arange(3))
        st = pvs.pvs_cursor_stats(cur)
        pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)
    assert got.tolist() == [1.0, np.float32(1 + 2.0 ** -23), 1.0]
    assert st["exact_fallbacks"] == 3


def _rank_all(index, q, chunk, total):
    cur = pvs.pvs_cursor_open(index, q)
    ids, scores, statuses = [], [], []
    try:
        while True:
            a, b, st = pvs.pvs_next(cur, chunk)
            ids.append(a)
            scores.append(b)
            statuses.append(st)
            if st == pvs.PVS_EXHAUSTED or sum(len(x) for x in ids) >= total:
                break
        stats = pvs.pvs_cursor_stats(cur)
        tail = pvs.pvs_next(cur, chunk) if statuses[-1] == pvs.PVS_EXHAUSTED else None
    finally:
        pvs.pvs_cursor_close(cur)
    return np.concatenate(ids), np.concatenate(scores), statuses, stats, tail


def test_config1_full_ranking_in_chunks_of_100():
    """N = 10,000, d = 128, i.i.d. normal rows normalised (seed 0), 16 queries:
    the complete ranking, pulled 100 ranks at a time, equals the oracle."""
    V = synth.unit_normal(10_000, 128, seed=0)
    Qs = synth.unit_normal(16, 128, seed=1000).numpy()
    Vh = V.numpy()
    index = pvs.pvs_build(V.cuda())
    try:
        for q in Qs:
            ids, sc, statuses, stats, tail = _rank_all(index, q, 100, 10_000)
            ref_ids, ref_sc = po.dense_ranking(q, Vh)
            by_id = dict(zip(ref_ids.tolist(), ref_sc.tolist()))
            assert _count_swaps(ids, ref_ids, by_id) == 0
            assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
            assert statuses[:-1] == [pvs.PVS_OK] * 99 and statuses[-1] == pvs.PVS_EXHAUSTED
            assert tail[0].size == 0 and tail[2] == pvs.PVS_EXHAUSTED
            assert stats["emitted"] == 10_000 and stats["interval_passes"] == 1
            assert stats["refined"] <= 10_000
    finally:
        pvs.pvs_index_free(index)


@pytest.mark.parametrize("n", [1, 2, 63, 64, 65, 129])
def test_small_and_ragged_corpora(n):
    rng = np.random.default_rng(n)
    V = rng.standard_normal((n, 96)).astype(np.float32)
    q = rng.standard_normal(96).astype(np.float32)
    index = pvs.pvs_build(V)
    try:
        ids, sc, statuses, _, _ = _rank_all(index, q, 7, n)
        ref_ids, ref_sc = po.dense_ranking(q, V)
        assert np.array_equal(ids, ref_ids) and np.array_equal(sc, ref_sc)
        assert statuses[-1] == pvs.PVS_EXHAUSTED
    finally:
        pvs.pvs_index_free(index)


def test_ties_and_degenerate_queries():
    V = np.tile(np.linspace(-1, 1, 32, dtype=np.float32), (300, 1))   # identical rows
    index = pvs.pvs_build(V)
    try:
        for q in (np.ones(32, np.float32), np.zeros(32, np.float32), -np.ones(32, np.float32)):
            ids, sc, _, _, _ = _rank_all(index, q, 64, 300)
            assert ids.tolist() == list(range(300))
            assert len(set(sc.tolist())) == 1
    finally:
        pvs.pvs_index_free(index)
    V = np.random.default_rng(1).standard_normal((500, 32)).astype(np.float32)
    index = pvs.pvs_build(V)
    try:
        ids, sc, _, _, _ = _rank_all(index, np.zeros(32, np.float32), 100, 500)
        assert ids.tolist() == list(range(500)) and not sc.any()
    finally:
        pvs.pvs_index_free(index)


def test_many_tied_rows_take_the_radix_selection_paths():
    """6,000 identical rows above 1,500 others: after the first pull more than
    2,048 working-set rows reach the selection's lower bound, so the one-launch
    pull falls back to the radix selection, and the emission orders more than
    2,048 candidates."""
    rng = np.random.default_rng(23)
    m = 64
    q = rng.standard_normal(m).astype(np.float32)
    top = (q / np.linalg.norm(q)).astype(np.float32)
    V = np.concatenate([np.tile(top, (6_000, 1)),
                        (rng.standard_normal((1_500, m)) * 0.05).astype(np.float32)])
    V = V[rng.permutation(len(V))]
    index = pvs.pvs_build(V)
    try:
        ref_ids, ref_sc = po.dense_ranking(q, V, np.ones(len(V), bool))
        cur = pvs.pvs_cursor_open(index, q)
        try:
            got_i, got_s = [], []
            for _ in range(8):
                i, sc, _ = pvs.pvs_next(cur, 100)
                got_i.append(i)
                got_s.append(sc)
            st = pvs.pvs_cursor_stats(cur)
        finally:
            pvs.pvs_cursor_close(cur)
        assert np.array_equal(np.concatenate(got_i), ref_ids[:800])
        assert np.array_equal(np.concatenate(got_s), ref_sc[:800])
        assert st["state"] >= 0
    finally:
        pvs.pvs_index_free(index)


def test_empty_index_and_zero_pulls():
    index = pvs.pvs_build(np.zeros((0, 64), np.float32))
    try:
        cur = pvs.pvs_cursor_open(index, np.ones(64, np.float32))
        ids, sc, st = pvs.pvs_next(cur, 10)
        assert ids.size == 0 and st == pvs.PVS_EXHAUSTED
        pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)
    index = pvs.pvs_build(np.ones((5, 64), np.float32))
    try:
        cur = pvs.pvs_cursor_open(index, np.ones(64, np.float32))
        ids, sc, st = pvs.pvs_next(cur, 0)
        assert ids.size == 0 and st == pvs.PVS_OK
        with pytest.raises(pvs.PvsError):
            pvs.pvs_next(cur, -1)
        pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)


def test_large_pull_uses_radix_sort_and_matches():
    centres = synth.mixture_centres(16, 64, seed=7, device="cpu")
    V = synth.mixture_rows(40_000, centres, 0.35, seed=8).numpy()
    q = synth.mixture_queries(1, centres, 0.5, seed=9).numpy()[0]
    index = pvs.pvs_build(V)
    try:
        cur = pvs.pvs_cursor_open(index, q)
        a, sa, _ = pvs.pvs_next(cur, 25_000)
        b, sb, st = pvs.pvs_next(cur, 25_000)
        pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)
    ref_ids, ref_sc = po.dense_ranking(q, V)
    assert np.array_equal(np.concatenate([a, b]), ref_ids)
    assert np.array_equal(np.concatenate([sa, sb]), ref_sc)
    assert st == pvs.PVS_EXHAUSTED


def test_snapshots_appends_and_tombstones():
    """Config-5 mechanics at small scale: near-duplicates, appends, deletions;
    each snapshot ranks exactly its visible set."""
    m = 256
    centres = synth.mixture_centres(32, m, seed=11, device="cpu")
    base = synth.mixture_rows(8_000, centres, 0.35, seed=12)
    rng = np.random.default_rng(13)
    dup_src = base[torch.from_numpy(rng.integers(0, 6_400, 1_600))]
    base[6_400:] = synth.near_duplicate_rows(dup_src, 1e-4, seed=14)
    all_rows = [base.numpy()]
    index = pvs.pvs_build(base.cuda())
    visible = np.ones(8_000, bool)
    snaps = [(pvs.pvs_snapshot_create(index), visible.copy(), 8_000)]
    try:
        for step in range(3):
            new = synth.mixture_rows(800, centres, 0.35, seed=20 + step).numpy()
            pvs.pvs_append(index, new)
            all_rows.append(new)
            visible = np.concatenate([visible, np.ones(800, bool)])
            live = np.nonzero(visible)[0]
            dead = rng.choice(live, int(0.02 * live.size), replace=False)
            pvs.pvs_tombstone(index, dead)
            visible[dead] = False
            snaps.append((pvs.pvs_snapshot_create(index), visible.copy(), visible.size))
        V = np.concatenate(all_rows)
        qs = synth.mixture_queries(3, centres, 0.5, seed=30).numpy()
        for snap, vis, rows in snaps:
            assert pvs.pvs_snapshot_visible(snap) == int(vis.sum())
            for q in qs:
                cur = pvs.pvs_cursor_open(index, q, snap)
                ids, sc, st = pvs.pvs_next(cur, 300)
                pvs.pvs_cursor_close(cur)
                ref_ids, ref_sc = po.dense_ranking(q, V[:rows], vis)
                assert np.array_equal(ids, ref_ids[:300])
                assert np.array_equal(sc, ref_sc[:300])
    finally:
        for snap, _, _ in snaps:
            pvs.pvs_snapshot_free(snap)
        pvs.pvs_index_free(index)


@pytest.mark.parametrize("tau", [0.5, 0.0, -0.5])
def test_eahr_topk_matches_complete_list_fusion(tau):
    m = 128
    centres = synth.mixture_centres(64, m, seed=40, device="cpu")
    V = synth.mixture_rows(30_000, centres, 0.35, seed=41).numpy()
    qs = synth.mixture_queries(4, centres, 0.5, seed=42).numpy()
    index = pvs.pvs_build(V)
    try:
        for qi, q in enumerate(qs):
            dense_ids, dense_sc = po.dense_ranking(q, V)
            proxy = torch.from_numpy(po.exact_scores(q, V).astype(np.float64))
            sparse = synth.copula_ranking(proxy, tau, seed=100 + qi).numpy()
            cur = pvs.pvs_cursor_open(index, q)
            try:
                ids, F, st = pvs.eahr_topk(cur, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR)
            finally:
                pvs.pvs_cursor_close(cur)
            T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
            assert ids.tolist() == [x for x, _ in T]
            for (x, f), got in zip(T, F):
                if not math.isnan(got):
                    assert got == ro.as_float(f)
    finally:
        pvs.pvs_index_free(index)


def test_cursors_on_separate_streams_and_threads_match_oracle():
    """Interleaved pulls of cursors on their own streams (their interval
    passes serialised per index, pulls overlapping) and cursors driven from
    two host threads both give the oracle's rankings."""
    import threading
    centres = synth.mixture_centres(32, 128, seed=50, device="cpu")
    V = synth.mixture_rows(20_000, centres, 0.35, seed=51).numpy()
    qs = synth.mixture_queries(6, centres, 0.5, seed=52).numpy()
    refs = [po.dense_ranking(q, V) for q in qs]
    index = pvs.pvs_build(V)
    try:
        streams = [torch.cuda.Stream() for _ in range(4)]
        ids_t = torch.zeros((4, 250), dtype=torch.int64, device="cuda")
        sc_t = torch.zeros((4, 250), dtype=torch.float32, device="cuda")
        curs = []
        for k in range(4):
            c = pvs.pvs_cursor_open(index, qs[k])
            pvs.pvs_cursor_set_stream(c, streams[k])
            curs.append(c)
        for p in range(10):
            for k, c in enumerate(curs):
                pvs.pvs_next_device(c, 25, ids_t[k, 25 * p:], sc_t[k, 25 * p:])
        for c in curs:
            assert pvs.pvs_cursor_sync(c) == pvs.PVS_OK
            pvs.pvs_cursor_close(c)
        torch.cuda.synchronize()
        for k in range(4):
            assert np.array_equal(ids_t[k].cpu().numpy(), refs[k][0][:250])
            assert np.array_equal(sc_t[k].cpu().numpy(), refs[k][1][:250])

        results, errors = {}, []

        def worker(k):
            try:
                c = pvs.pvs_cursor_open(index, qs[k])
                pvs.pvs_cursor_set_stream(c, streams[k % 2])
                got = [pvs.pvs_next(c, 40)[0] for _ in range(5)]
                pvs.pvs_cursor_close(c)
                results[k] = np.concatenate(got)
            except Exception as e:
                errors.append(e)

        threads = [threading.Thread(target=worker, args=(k,)) for k in (4, 5)]
        for t in threads:
            t.start()
        for t in threads:
            t.join()
        assert not errors
        for k in (4, 5):
            assert np.array_equal(results[k], refs[k][0][:200])
    finally:
        pvs.pvs_index_free(index)


def test_eahr_rejects_bad_sparse_lists_and_used_cursors():
    V = np.random.default_rng(0).standard_normal((200, 32)).astype(np.float32)
    index = pvs.pvs_build(V)
    try:
        q = V[0]
        cur = pvs.pvs_cursor_open(index, q)
        with pytest.raises(pvs.PvsError):
            pvs.eahr_topk(cur, np.array([5, 5, 6]), K=3, step=1)
        pvs.pvs_cursor_close(cur)
        cur = pvs.pvs_cursor_open(index, q)
        with pytest.raises(pvs.PvsError):
            pvs.eahr_topk(cur, np.array([1000]), K=3, step=1)
        pvs.pvs_cursor_close(cur)
        cur = pvs.pvs_cursor_open(index, q)
        pvs.pvs_next(cur, 1)
        with pytest.raises(pvs.PvsError):
            pvs.eahr_topk(cur, np.arange(200), K=3)
        pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)


@pytest.mark.parametrize("crowded", [False, True])
def test_first_working_set_from_per_slot_bounds(crowded):
    """The first working set after an interval pass is selected from each row
    slot's four largest lower bounds (a slot = a CTA's row position in a
    64-row tile).  That threshold is never above the exact one, so the ranks
    stay exact; with the best rows crowded into one slot it is much lower and
    the working set larger, and the ranks must still be exact (Sec. 2.1,
    2.3.1)."""
    n, m = 2_000_003, 32
    rng = np.random.default_rng(211)
    V = rng.standard_normal((n, m)).astype(np.float32)
    V /= np.linalg.norm(V, axis=1, keepdims=True)
    q = rng.standard_normal(m).astype(np.float32)
    q /= np.linalg.norm(q)
    if crowded:
        # rows of slot 5 of the first CTA (tiles 0, 152, 304, ... of 64 rows)
        # are near-copies of the query: every one of them beats every other row
        rows = np.arange(5, n, 64 * 152)
        V[rows] = q + 0.01 * rng.standard_normal((rows.size, m)).astype(np.float32)
        V[rows] /= np.linalg.norm(V[rows], axis=1, keepdims=True)
    index = pvs.pvs_build(V)
    try:
        cur = pvs.pvs_cursor_open(index, q)
        try:
            got = [pvs.pvs_next(cur, 20) for _ in range(50)]
            st = pvs.pvs_cursor_stats(cur)
        finally:
            pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)
    ids = np.concatenate([g[0] for g in got])
    sc = np.concatenate([g[1] for g in got])
    ref_ids, ref_sc = po.dense_ranking(q, V)
    assert np.array_equal(ids, ref_ids[:1000])
    assert np.array_equal(sc.view(np.uint32), ref_sc[:1000].view(np.uint32))
    assert st["interval_passes"] == 1


@pytest.mark.parametrize("tau", [0.5, 0.0])
def test_frozen_scheduler_over_a_pvs_cursor(tau):
    """Sec. 3.5's frozen scheduler (EAHR_POLICY_FROZEN) driving a real dense
    cursor: the ordered Top-20 equals complete-list fusion, and every pull of
    either list reads one 16-rank step (the last pull of a list that runs out
    may read fewer)."""
    n, m = 30_000, 64
    centres = synth.mixture_centres(64, m, seed=80, device="cpu")
    V = synth.mixture_rows(n, centres, 0.35, seed=81).numpy()
    q = synth.mixture_queries(1, centres, 0.5, seed=82).numpy()[0]
    dense_ids, dense_sc = po.dense_ranking(q, V)
    proxy = torch.from_numpy(dense_sc[np.argsort(dense_ids)].astype(np.float64))
    sparse = synth.copula_ranking(proxy, tau, seed=83).numpy()
    T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
    index = pvs.pvs_build(V)
    try:
        cur = pvs.pvs_cursor_open(index, q)
        try:
            ids, F, st = pvs.eahr_topk(cur, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR,
                                       policy=pvs.EAHR_POLICY_FROZEN, step=16)
        finally:
            pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)
    assert ids.tolist() == [x for x, _ in T]
    for (x, f), got in zip(T, F):
        if not np.isnan(got):
            assert got == ro.as_float(f)
    for i in range(2):
        d, p = st["depth"][i], st["pulls"][i]
        assert p >= 1 and 16 * (p - 1) < d <= 16 * p
        if not st["exhausted"][i]:
            assert d == 16 * p


@pytest.mark.parametrize("pages", [1, 4, 13])
def test_readahead_with_mixed_calls_matches_the_oracle(pages):
    """A pull may compute ranks ahead of the caller (pvs_cursor_set_readahead);
    Sec. 2.1's stable prefix makes any mix of host, device and batched calls
    of any sizes deliver the complete ranking in order."""
    n, m = 20_011, 128
    V = synth.unit_normal(n, m, seed=90).numpy()
    q = synth.unit_normal(1, m, seed=91).numpy()[0]
    ref_ids, ref_sc = po.dense_ranking(q, V)
    index = pvs.pvs_build(V)
    got_i, got_s = [], []
    try:
        cur = pvs.pvs_cursor_open(index, q)
        try:
            pvs.pvs_cursor_set_readahead(cur, pages)
            for k, kind in ((7, "host"), (20, "dev"), (3, "host"), (20, "batch_host"),
                            (11, "batch_dev"), (300, "host"), (257, "dev"), (64, "batch_dev"),
                            (1, "dev"), (999, "batch_host"), (5, "host")):
                if kind == "host":
                    i, s, _ = pvs.pvs_next(cur, k)
                elif kind == "dev":
                    ti = torch.empty(k, dtype=torch.int64, device="cuda")
                    ts = torch.empty(k, dtype=torch.float32, device="cuda")
                    got, _ = pvs.pvs_next_device(cur, k, ti, ts)
                    assert pvs.pvs_cursor_sync(cur) >= 0
                    i, s = ti[:got].cpu().numpy(), ts[:got].cpu().numpy()
                elif kind == "batch_host":
                    ib, sb, nb = pvs.pvs_next_batch([cur], k)
                    i, s = ib[0, :nb[0]], sb[0, :nb[0]]
                else:
                    ti = torch.empty((1, k), dtype=torch.int64, device="cuda")
                    ts = torch.empty((1, k), dtype=torch.float32, device="cuda")
                    nb = pvs.pvs_next_batch([cur], k, ti, ts)
                    assert pvs.pvs_cursor_sync(cur) >= 0
                    i, s = ti[0, :nb[0]].cpu().numpy(), ts[0, :nb[0]].cpu().numpy()
                assert len(i) == k
                got_i.append(np.asarray(i))
                got_s.append(np.asarray(s))
            st = pvs.pvs_cursor_stats(cur)
        finally:
            pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)
    ids = np.concatenate(got_i)
    sc = np.concatenate(got_s).astype(np.float32)
    assert st["emitted"] == ids.size
    assert np.array_equal(ids, ref_ids[:ids.size])
    assert np.array_equal(sc.view(np.uint32), ref_sc[:ids.size].view(np.uint32))
