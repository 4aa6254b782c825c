"""Hierarchical Segment / Shard merging through the C ABI (arXiv 2608.07152
Sec. 2.4): the merged ranking of per-Segment exact rankings equals the
oracle's complete ranking of the union; copies with equal scores merge,
conflicting copies fail; EAHR over merged channels equals complete-list
fusion (Sec. 2.2)."""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pbm_oracle as pbo
from oracle import pvs_oracle as po
from oracle import rrf_oracle as ro

pytestmark = pytest.mark.gpu


def pull_all(merge, chunk):
    ids, sc = [], []
    while True:
        i, s, st = pvs.pvs_merge_next(merge, chunk)
        ids.append(i)
        sc.append(s)
        if st == pvs.PVS_EXHAUSTED:
            return np.concatenate(ids), np.concatenate(sc)


class Segments:
    """Dense segment indexes over row ranges of V (global id = row)."""

    def __init__(self, V, bounds):
        self.bounds = bounds
        self.index = [pvs.pvs_build(V[a:b]) for a, b in bounds]

    def cursors(self, q):
        return [pvs.pvs_cursor_open(x, q) for x in self.index]

    def free(self):
        for x in self.index:
            pvs.pvs_index_free(x)


def test_disjoint_segments_merge_to_the_union_ranking():
    V = synth.unit_normal(7001, 64, seed=90).numpy()
    q = synth.unit_normal(1, 64, seed=91).numpy()[0]
    bounds = [(0, 1500), (1500, 1501), (1501, 4000), (4000, 6999), (6999, 7001)]
    segs = Segments(V, bounds)
    try:
        curs = segs.cursors(q)
        merge = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, a) for c, (a, _) in zip(curs, bounds)])
        try:
            ids, sc = pull_all(merge, 113)
            st = pvs.pvs_merge_stats(merge)
        finally:
            pvs.pvs_merge_close(merge)
            for c in curs:
                pvs.pvs_cursor_close(c)
    finally:
        segs.free()
    ref_ids, ref_sc = po.dense_ranking(q, V)
    assert np.array_equal(ids, ref_ids)
    assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
    assert st["duplicates"] == 0 and st["emitted"] == 7001 and st["id_space"] == 7001


def test_shards_of_segments_equal_the_flat_merge():
    V = synth.unit_normal(6000, 48, seed=92).numpy()
    q = synth.unit_normal(1, 48, seed=93).numpy()[0]
    bounds = [(0, 1000), (1000, 2600), (2600, 3000), (3000, 4500), (4500, 6000)]
    segs = Segments(V, bounds)
    try:
        curs = segs.cursors(q)
        shard0 = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, a)
                                     for c, (a, _) in zip(curs[:3], bounds[:3])])
        # shard 1 numbers its segments from 0 and sits at offset 3000 in the request
        shard1 = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, a - 3000)
                                     for c, (a, _) in zip(curs[3:], bounds[3:])])
        top = pvs.pvs_merge_open([(pvs.PVS_CHILD_MERGE, shard0, 0),
                                  (pvs.PVS_CHILD_MERGE, shard1, 3000)])
        try:
            got = [pvs.pvs_merge_next(top, 20)[0] for _ in range(25)]
            ids = np.concatenate(got)
        finally:
            pvs.pvs_merge_close(top)
            pvs.pvs_merge_close(shard0)
            pvs.pvs_merge_close(shard1)
            for c in curs:
                pvs.pvs_cursor_close(c)
    finally:
        segs.free()
    ref_ids, _ = po.dense_ranking(q, V)
    assert np.array_equal(ids, ref_ids[:500])


def test_copies_with_equal_scores_merge_and_conflicts_fail():
    V = synth.unit_normal(5000, 32, seed=94).numpy()
    q = synth.unit_normal(1, 32, seed=95).numpy()[0]
    # rows 2000 .. 2999 live in both segments (same vectors, same ids)
    segs = Segments(V, [(0, 3000), (2000, 5000)])
    try:
        curs = segs.cursors(q)
        merge = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, curs[0], 0),
                                    (pvs.PVS_CHILD_DENSE, curs[1], 2000)])
        try:
            ids, sc = pull_all(merge, 256)
            st = pvs.pvs_merge_stats(merge)
        finally:
            pvs.pvs_merge_close(merge)
            for c in curs:
                pvs.pvs_cursor_close(c)
    finally:
        segs.free()
    ref_ids, ref_sc = po.dense_ranking(q, V)
    assert np.array_equal(ids, ref_ids)
    assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
    assert st["duplicates"] == 1000
    # the same ids with other vectors: conflicting copies invalidate the request
    W = V.copy()
    W[2000:3000] = synth.unit_normal(1000, 32, seed=96).numpy()
    a = pvs.pvs_build(V[0:3000])
    b = pvs.pvs_build(W[2000:5000])
    try:
        ca, cb = pvs.pvs_cursor_open(a, q), pvs.pvs_cursor_open(b, q)
        merge = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, ca, 0), (pvs.PVS_CHILD_DENSE, cb, 2000)])
        try:
            with pytest.raises(pvs.PvsError) as e:
                pull_all(merge, 256)
            assert e.value.status == pvs.PVS_ERR_INVALID
            with pytest.raises(pvs.PvsError):
                pvs.pvs_merge_next(merge, 10)            # failed for good
        finally:
            pvs.pvs_merge_close(merge)
            pvs.pvs_cursor_close(ca)
            pvs.pvs_cursor_close(cb)
    finally:
        pvs.pvs_index_free(a)
        pvs.pvs_index_free(b)


def sparse_segment(off, docs, imps, a, b):
    """Postings of the items a .. b-1, renumbered from 0 (one PBM segment)."""
    o, d, p = [0], [], []
    for t in range(len(off) - 1):
        dd = docs[off[t]:off[t + 1]]
        pp = imps[off[t]:off[t + 1]]
        k = (dd >= a) & (dd < b)
        d.append(dd[k] - a)
        p.append(pp[k])
        o.append(o[-1] + int(k.sum()))
    return (np.array(o, np.int64), np.concatenate(d).astype(np.int32),
            np.concatenate(p).astype(np.float32))


def test_sparse_segments_and_eahr_over_merged_channels():
    n, m = 12_000, 48
    bounds = [(0, 2500), (2500, 7000), (7000, 12_000)]
    V = synth.unit_normal(n, m, seed=97).numpy()
    q = synth.unit_normal(1, m, seed=98).numpy()[0]
    off, docs, imps = synth.bm25_postings(n, 3000, 20.0, seed=99)
    off, docs, imps = off.numpy(), docs.numpy(), imps.numpy()
    terms, weights = synth.sparse_queries(1, torch.from_numpy(off), seed=100, mean_terms=4.0)[0]
    sp_idx = [pvs.pbm_build(*sparse_segment(off, docs, imps, a, b), b - a) for a, b in bounds]
    segs = Segments(V, bounds)
    try:
        # the merged sparse ranking
        scur = [pvs.pbm_cursor_open(x, terms, weights) for x in sp_idx]
        smerge = pvs.pvs_merge_open([(pvs.PVS_CHILD_SPARSE, c, a) for c, (a, _) in zip(scur, bounds)])
        try:
            ids, sc = pull_all(smerge, 333)
        finally:
            pvs.pvs_merge_close(smerge)
            for c in scur:
                pvs.pbm_cursor_close(c)
        ref_ids, ref_sc = pbo.sparse_ranking(terms, weights, off, docs, imps, n)
        assert np.array_equal(ids, ref_ids)
        assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
        # EAHR over both merged channels
        dcur = segs.cursors(q)
        scur = [pvs.pbm_cursor_open(x, terms, weights) for x in sp_idx]
        dm = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, a) for c, (a, _) in zip(dcur, bounds)])
        sm = pvs.pvs_merge_open([(pvs.PVS_CHILD_SPARSE, c, a) for c, (a, _) in zip(scur, bounds)])
        try:
            got, F, st = pvs.eahr_topk_merge(dm, sm, K=20, k=60, form=pvs.EAHR_NUMERATOR)
        finally:
            pvs.pvs_merge_close(dm)
            pvs.pvs_merge_close(sm)
            for c in dcur:
                pvs.pvs_cursor_close(c)
            for c in scur:
                pvs.pbm_cursor_close(c)
    finally:
        segs.free()
        for x in sp_idx:
            pvs.pbm_index_free(x)
    dense_ids, _ = po.dense_ranking(q, V)
    T = ro.target_topk_large([dense_ids, ref_ids], [1, 1], 60, 20, ro.NUMERATOR)
    assert got.tolist() == [x for x, _ in T]
    for (x, f), g in zip(T, F):
        if not np.isnan(g):
            assert g == ro.as_float(f)


def test_merge_argument_errors():
    V = synth.unit_normal(200, 16, seed=101).numpy()
    index = pvs.pvs_build(V)
    try:
        c = pvs.pvs_cursor_open(index, V[0])
        try:
            with pytest.raises(pvs.PvsError):
                pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, 0), (pvs.PVS_CHILD_DENSE, c, 0)])
            with pytest.raises(pvs.PvsError):
                pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, -5)])
            with pytest.raises(pvs.PvsError):
                pvs.pvs_merge_open([(7, c, 0)])
            pvs.pvs_next(c, 3)
            with pytest.raises(pvs.PvsError):          # not fresh
                pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, 0)])
        finally:
            pvs.pvs_cursor_close(c)
    finally:
        pvs.pvs_index_free(index)
