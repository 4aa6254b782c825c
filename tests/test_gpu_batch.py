"""Batched (tensor-core) PVS path against the oracle, through the C ABI.

* pvs_batch_bounds: the exact Int8 dot products of up to 256 queries come
  from one bf16 tcgen05 GEMM (codes |z| <= 127, sums < 2^24: exact in fp32);
  its epilogue must reproduce the oracle's intervals bit for bit
  (Sec. 2.3.1, App. A.1).
* pvs_cursor_open_batch + pvs_next_batch / pvs_next: every cursor's ranks
  equal the oracle's complete ranking, including past the batch horizon
  (where a cursor falls back to its own interval pass).
"""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po

pytestmark = pytest.mark.gpu


def _mixture(n, m, nq, seed, comps=64):
    centres = synth.mixture_centres(comps, m, seed=seed, device="cpu")
    V = synth.mixture_rows(n, centres, 0.35, seed=seed + 1).numpy()
    Q = synth.mixture_queries(nq, centres, 0.5, seed=seed + 2).numpy()
    return V, Q


@pytest.mark.parametrize("n,m,nq", [(300, 128, 32), (3_005, 768, 37), (10_037, 128, 5),
                                    (2_111, 1024, 64), (777, 100, 256)])
def test_batch_bounds_bit_exact(n, m, nq):
    V, Q = _mixture(n, m, nq, seed=n + m)
    Qz = po.quantize(V)
    index = pvs.pvs_build(V)
    try:
        lo, hi = pvs.pvs_batch_bounds(index, Q)
    finally:
        pvs.pvs_index_free(index)
    for qi in range(nq):
        qe = po.encode_query(Q[qi])
        ref_lo, ref_hi = po.intervals(qe, Qz, m)
        assert np.array_equal(lo[qi].view(np.uint32), ref_lo.view(np.uint32)), qi
        assert np.array_equal(hi[qi].view(np.uint32), ref_hi.view(np.uint32)), qi


def test_open_batch_ranks_match_oracle_past_the_horizon():
    V, Q = _mixture(20_000, 128, 40, seed=7)
    refs = [po.dense_ranking(q, V) for q in Q]
    index = pvs.pvs_build(V)
    try:
        curs = pvs.pvs_cursor_open_batch(index, Q, horizon=100)
        got = [[] for _ in curs]
        for step in range(12):                      # 600 ranks: past ~3x the horizon
            ids, sc, n_out = pvs.pvs_next_batch(curs, 50)
            for i in range(len(curs)):
                got[i].append((ids[i, :n_out[i]], sc[i, :n_out[i]]))
        for i, c in enumerate(curs):
            st = pvs.pvs_cursor_stats(c)
            assert st["batch_passes"] == 1
            pvs.pvs_cursor_close(c)
            gi = np.concatenate([g[0] for g in got[i]])
            gs = np.concatenate([g[1] for g in got[i]])
            assert np.array_equal(gi, refs[i][0][:600])
            assert np.array_equal(gs, refs[i][1][:600])
    finally:
        pvs.pvs_index_free(index)


def test_open_batch_groups_snapshots_and_device_outputs():
    V, Q = _mixture(5_000, 64, 300, seed=11, comps=16)
    index = pvs.pvs_build(V)
    rng = np.random.default_rng(3)
    dead = rng.choice(5_000, 250, replace=False)
    pvs.pvs_tombstone(index, dead)
    snap = pvs.pvs_snapshot_create(index)
    vis = np.ones(5_000, bool)
    vis[dead] = False
    try:
        curs = pvs.pvs_cursor_open_batch(index, Q, horizon=40, snap=snap)  # two groups
        assert len(curs) == 300
        ids_t = torch.zeros((300, 30), dtype=torch.int64, device="cuda")
        sc_t = torch.zeros((300, 30), dtype=torch.float32, device="cuda")
        got_ids, got_sc = [], []
        for step in range(3):
            # one group per call: cursors of one batch share the index stream
            n_out = pvs.pvs_next_batch(curs, 30, ids_t, sc_t)
            assert all(n_out == 30)
            for c in curs[:1]:
                assert pvs.pvs_cursor_sync(c) == pvs.PVS_OK
            torch.cuda.synchronize()
            got_ids.append(ids_t.cpu().numpy().copy())
            got_sc.append(sc_t.cpu().numpy().copy())
        for i in (0, 1, 137, 255, 256, 299):
            ref_ids, ref_sc = po.dense_ranking(Q[i], V, vis)
            gi = np.concatenate([g[i] for g in got_ids])
            gs = np.concatenate([g[i] for g in got_sc])
            assert np.array_equal(gi, ref_ids[:90])
            assert np.array_equal(gs, ref_sc[:90])
        for c in curs:
            pvs.pvs_cursor_close(c)
    finally:
        pvs.pvs_snapshot_free(snap)
        pvs.pvs_index_free(index)


def test_batch_sync_stats_and_close_agree_with_per_cursor_calls():
    V, Q = _mixture(4_000, 96, 40, seed=21, comps=16)
    index = pvs.pvs_build(V)
    side = torch.cuda.Stream()
    try:
        curs = pvs.pvs_cursor_open_batch(index, Q, horizon=30)
        ids, sc, n_out = pvs.pvs_next_batch(curs, 25)
        assert all(n_out == 25)
        # two cursors move to another stream: the batch helpers group by stream
        for c in curs[:2]:
            pvs.pvs_cursor_set_stream(c, side)
        for c in curs[:2]:
            i2, s2, n2 = pvs.pvs_next(c, 10)
        states = pvs.pvs_cursor_sync_batch(curs)
        assert list(states) == [pvs.pvs_cursor_sync(c) for c in curs]
        assert all(s == pvs.PVS_OK for s in states)
        many = pvs.pvs_cursor_stats_batch(curs)
        one = [pvs.pvs_cursor_stats(c) for c in curs]
        for a, b in zip(many, one):
            for key in ("visible", "emitted", "refined", "exact_fallbacks", "pulls",
                        "candidates", "state", "batch_passes"):
                assert a[key] == b[key], key
        assert [s["emitted"] for s in many[:3]] == [35, 35, 25]
        for i in (0, 5, 39):
            ref_ids, ref_sc = po.dense_ranking(Q[i], V, np.ones(len(V), bool))
            assert np.array_equal(ids[i], ref_ids[:25])
            assert np.array_equal(sc[i], ref_sc[:25])
        pvs.pvs_cursor_close_batch(curs)
        assert len(pvs.pvs_cursor_sync_batch([])) == 0
        pvs.pvs_cursor_close_batch([])
    finally:
        pvs.pvs_index_free(index)


def test_open_batch_rejects_a_non_finite_query_and_stays_usable():
    V, Q = _mixture(2_000, 64, 8, seed=31, comps=8)
    index = pvs.pvs_build(V)
    try:
        bad = Q.copy()
        bad[5, 3] = np.nan
        with pytest.raises(pvs.PvsError) as err:
            pvs.pvs_cursor_open_batch(index, bad, horizon=20)
        assert err.value.status == pvs.PVS_ERR_NONFINITE
        curs = pvs.pvs_cursor_open_batch(index, Q, horizon=20)
        ids, sc, n_out = pvs.pvs_next_batch(curs, 20)
        for i in range(len(Q)):
            ref_ids, ref_sc = po.dense_ranking(Q[i], V, np.ones(len(V), bool))
            assert np.array_equal(ids[i], ref_ids[:20])
            assert np.array_equal(sc[i], ref_sc[:20])
        pvs.pvs_cursor_close_batch(curs)
    finally:
        pvs.pvs_index_free(index)


def test_batched_opens_on_two_threads_and_streams():
    import threading
    V, Q = _mixture(6_000, 128, 64, seed=41, comps=16)
    index = pvs.pvs_build(V)
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    results, errors = {}, []

    def worker(k):
        try:
            for rep in range(3):
                part = Q[k * 32:(k + 1) * 32]
                curs = pvs.pvs_cursor_open_batch(index, part, horizon=40, stream=streams[k])
                ids, sc, n_out = pvs.pvs_next_batch(curs, 40)
                assert all(pvs.pvs_cursor_sync_batch(curs) >= 0)
                pvs.pvs_cursor_close_batch(curs)
                results[(k, rep)] = (ids.copy(), sc.copy())
        except Exception as e:
            errors.append(e)

    try:
        threads = [threading.Thread(target=worker, args=(k,)) for k in range(2)]
        for t in threads:
            t.start()
        for t in threads:
            t.join()
        assert not errors, errors
        vis = np.ones(len(V), bool)
        for k in range(2):
            for i in (0, 13, 31):
                ref_ids, ref_sc = po.dense_ranking(Q[k * 32 + i], V, vis)
                for rep in range(3):
                    ids, sc = results[(k, rep)]
                    assert np.array_equal(ids[i], ref_ids[:40])
                    assert np.array_equal(sc[i], ref_sc[:40])
    finally:
        pvs.pvs_index_free(index)
