"""Cursors pulled from several host threads at once through the C ABI
(arXiv 2608.07152 Sec. 2.1: each cursor's ranks are its query's exact
ranking whatever else runs).  Pulls of different sizes take launch paths
whose kernels need different amounts of shared memory; threads launching the
same kernel with different sizes must not disturb each other."""
import threading

import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po

pytestmark = pytest.mark.gpu

# page sizes: one-launch pulls (<= 256) and multi-launch pulls whose
# candidate sorts take 1 KB .. 64 KB of shared memory
SIZES = [20, 300, 700, 1500, 3000, 250, 5000, 64, 2222]


def test_concurrent_pulls_of_different_sizes():
    V = synth.unit_normal(40_000, 64, seed=201).numpy()
    Q = synth.unit_normal(8, 64, seed=202).numpy()
    index = pvs.pvs_build(V)
    streams = [torch.cuda.Stream() for _ in range(8)]
    got = [None] * 8
    errors = []

    def worker(k):
        try:
            order = SIZES[k % len(SIZES):] + SIZES[:k % len(SIZES)]
            for rep in range(3):
                cur = pvs.pvs_cursor_open(index, Q[k])
                pvs.pvs_cursor_set_stream(cur, streams[k].cuda_stream)
                ids = []
                for n in order:
                    i, _, _ = pvs.pvs_next(cur, n)
                    ids.append(i)
                pvs.pvs_cursor_close(cur)
                got[k] = np.concatenate(ids)
        except Exception as e:   # surfaced below
            errors.append(e)

    try:
        threads = [threading.Thread(target=worker, args=(k,)) for k in range(8)]
        for t in threads:
            t.start()
        for t in threads:
            t.join()
    finally:
        pvs.pvs_index_free(index)
    assert not errors, errors[0]
    total = sum(SIZES)
    for k in range(8):
        ref, _ = po.dense_ranking(Q[k], V)
        assert np.array_equal(got[k], ref[:total]), k


def test_concurrent_merges_over_segments_on_their_own_streams():
    """Two merge cursors over Segments with streams of their own, refilled
    concurrently inside each merge, from two host threads."""
    V = synth.unit_normal(24_000, 48, seed=203).numpy()
    Q = synth.unit_normal(2, 48, seed=204).numpy()
    bounds = [(0, 3000), (3000, 9000), (9000, 9001), (9001, 17000), (17000, 24000)]
    segs = [pvs.pvs_build(V[a:b]) for a, b in bounds]
    got = [None, None]
    errors = []

    def worker(k):
        try:
            curs = [pvs.pvs_cursor_open(x, Q[k]) for x in segs]
            m = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, a) for c, (a, _) in zip(curs, bounds)])
            parts = [pvs.pvs_merge_next(m, n)[0] for n in (16, 700, 3000, 9000, 40)]
            pvs.pvs_merge_close(m)
            for c in curs:
                pvs.pvs_cursor_close(c)
            got[k] = np.concatenate(parts)
        except Exception as e:   # surfaced below
            errors.append(e)

    try:
        threads = [threading.Thread(target=worker, args=(k,)) for k in range(2)]
        for t in threads:
            t.start()
        for t in threads:
            t.join()
    finally:
        for x in segs:
            pvs.pvs_index_free(x)
    assert not errors, errors[0]
    for k in range(2):
        ref, _ = po.dense_ranking(Q[k], V)
        assert np.array_equal(got[k], ref[:got[k].size]) and got[k].size == 12_756, k
