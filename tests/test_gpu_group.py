"""Grouped interval pass (pvs_cursor_open_group) against the single-query
pass and the oracle (arXiv 2608.07152 Sec. 2.1, 2.3.1, App. A.1).

One streaming read of the codes scores every tile against up to eight
queries.  Each query's intervals must be bit-identical to the single-query
pass's and to the oracle's App. A.1 arithmetic, sound for every row, and the
ranks that follow identical to the oracle's complete dense ranking (ids in
order, score bits).
"""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po

pytestmark = pytest.mark.gpu


def _bounds(cur, n):
    return pvs.pvs_cursor_bounds(cur, 0, n)


def _oracle_bounds(V, q, m):
    Q = po.quantize(V, ldz=m)
    qe = po.encode_query(q)
    return po.intervals(qe, Q, m)


@pytest.mark.parametrize("m,n,nq", [(128, 9_731, 8), (100, 20_123, 3), (768, 30_011, 8),
                                    (768, 12_345, 2), (1024, 17_777, 5), (384, 40_961, 8),
                                    (256, 8_193, 4), (512, 25_000, 7),
                                    # 9 .. 16 queries: both warp groups on every tile
                                    (768, 30_011, 16), (128, 9_731, 12), (384, 40_961, 9),
                                    (512, 25_000, 16)])
def test_group_bounds_equal_single_pass_and_oracle(m, n, nq):
    V = synth.unit_normal(n, m, seed=81 + m, device="cuda")
    Q = synth.unit_normal(nq, m, seed=82 + m, device="cuda")
    Vh, Qh = V.cpu().numpy(), Q.cpu().numpy()
    index = pvs.pvs_build(V)
    try:
        curs = pvs.pvs_cursor_open_group(index, Q)
        try:
            got = [_bounds(c, n) for c in curs]
            stats = [pvs.pvs_cursor_stats(c) for c in curs]
            ranks = [pvs.pvs_next(c, 300) for c in curs]
        finally:
            for c in curs:
                pvs.pvs_cursor_close(c)
        single = []
        for i in range(nq):
            c = pvs.pvs_cursor_open(index, Q[i])
            try:
                single.append(_bounds(c, n))
            finally:
                pvs.pvs_cursor_close(c)
    finally:
        pvs.pvs_index_free(index)
    for i in range(nq):
        lo, hi = got[i]
        assert np.array_equal(lo.view(np.uint32), single[i][0].view(np.uint32))
        assert np.array_equal(hi.view(np.uint32), single[i][1].view(np.uint32))
        assert stats[i]["interval_passes"] == 1
        assert stats[i]["code_bytes"] == n * (((m + 63) // 64) * 64 + 12) // nq
    # oracle intervals and exact ranks for a few of the queries
    for i in sorted({0, nq - 1}):
        olo, ohi = _oracle_bounds(Vh, Qh[i], m)
        assert np.array_equal(got[i][0].view(np.uint32), olo.view(np.uint32))
        assert np.array_equal(got[i][1].view(np.uint32), ohi.view(np.uint32))
        ref_ids, ref_sc = po.dense_ranking(Qh[i], Vh)
        assert np.all(olo <= po.exact_scores(Qh[i], Vh))
        ids, sc, _ = ranks[i]
        assert np.array_equal(ids, ref_ids[:300])
        assert np.array_equal(sc.view(np.uint32), ref_sc[:300].view(np.uint32))


@pytest.mark.parametrize("nq", [8, 16])
def test_group_on_own_streams_with_deletions_and_deep_pulls(nq):
    n, m = 60_000, 768
    V = synth.unit_normal(n, m, seed=91, device="cuda")
    Q = synth.unit_normal(nq, m, seed=92)
    rng = np.random.default_rng(93)
    dead = rng.choice(n, 3_000, replace=False)
    visible = np.ones(n, bool)
    visible[dead] = False
    streams = [torch.cuda.Stream() for _ in range(nq)]
    pass_stream = torch.cuda.Stream()
    index = pvs.pvs_build(V)
    try:
        pvs.pvs_tombstone(index, dead)
        snap = pvs.pvs_snapshot_create(index)
        try:
            curs = pvs.pvs_cursor_open_group(index, Q, snap=snap, pass_stream=pass_stream,
                                             cursor_streams=streams)
            try:
                out = []
                for c in curs:
                    parts = [pvs.pvs_next(c, k) for k in (20, 20, 500, 3000)]
                    out.append((np.concatenate([p[0] for p in parts]),
                                np.concatenate([p[1] for p in parts])))
            finally:
                for c in curs:
                    pvs.pvs_cursor_close(c)
        finally:
            pvs.pvs_snapshot_free(snap)
    finally:
        pvs.pvs_index_free(index)
    Vh = V.cpu().numpy()
    for i in range(nq):
        ref_ids, ref_sc = po.dense_ranking(Q[i].numpy(), Vh, visible=visible)
        ids, sc = out[i]
        assert np.array_equal(ids, ref_ids[:3540])
        assert np.array_equal(sc.view(np.uint32), ref_sc[:3540].view(np.uint32))


def test_group_with_a_width_the_grouped_pass_does_not_serve_and_one_query():
    # 1100: no grouped kernel; 1024 with 16 queries: no split kernel (the
    # query fragments would not fit in registers); one query: a plain cursor
    for m, nq in ((1100, 3), (768, 1), (1024, 16)):
        n = 5_000
        V = synth.unit_normal(n, m, seed=95, device="cuda")
        Q = synth.unit_normal(nq, m, seed=96)
        index = pvs.pvs_build(V)
        try:
            curs = pvs.pvs_cursor_open_group(index, Q)
            try:
                got = [pvs.pvs_next(c, 100) for c in curs]
            finally:
                for c in curs:
                    pvs.pvs_cursor_close(c)
        finally:
            pvs.pvs_index_free(index)
        for i in range(nq):
            ref_ids, ref_sc = po.dense_ranking(Q[i].numpy(), V.cpu().numpy())
            assert np.array_equal(got[i][0], ref_ids[:100])
            assert np.array_equal(got[i][1].view(np.uint32), ref_sc[:100].view(np.uint32))


def test_group_errors_and_timeout():
    n, m = 300_000, 768
    V = synth.unit_normal(n, m, seed=97, device="cuda")
    Q = synth.unit_normal(4, m, seed=98)
    index = pvs.pvs_build(V)
    try:
        bad = Q.clone()
        bad[2, 7] = float("nan")
        with pytest.raises(pvs.PvsError) as e:
            pvs.pvs_cursor_open_group(index, bad)
        assert e.value.status == pvs.PVS_ERR_NONFINITE
        with pytest.raises(pvs.PvsError) as e:
            pvs.pvs_cursor_open_group(index, synth.unit_normal(pvs.PVS_GROUP_MAX + 1, m, seed=99))
        assert e.value.status == pvs.PVS_ERR_INVALID
        # the grouped pass's waits give up at once: the open fails, no cursor
        pvs.pvs_index_set_wait_limit(index, 0)
        with pytest.raises(pvs.PvsError) as e:
            pvs.pvs_cursor_open_group(index, Q)
        assert e.value.status == pvs.PVS_ERR_TIMEOUT
        pvs.pvs_index_set_wait_limit(index, 2_000_000_000)
        curs = pvs.pvs_cursor_open_group(index, Q)
        try:
            got = [pvs.pvs_next(c, 50) for c in curs]
        finally:
            for c in curs:
                pvs.pvs_cursor_close(c)
    finally:
        pvs.pvs_index_free(index)
    Vh = V.cpu().numpy()
    for i in (0, 3):
        ref_ids, ref_sc = po.dense_ranking(Q[i].numpy(), Vh)
        assert np.array_equal(got[i][0], ref_ids[:50])
        assert np.array_equal(got[i][1].view(np.uint32), ref_sc[:50].view(np.uint32))
