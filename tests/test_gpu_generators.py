"""The rank generators PVS is compared with in the ablation (arXiv
2608.07152 Sec. 3.5, 4.4), through the C ABI against the oracle:

* scalar-quantization intervals: an index with one scale for the corpus
  (pvs_build_ex, PVS_QUANT_GLOBAL); codes, norm bounds and intervals bit for
  bit against the oracle's one-scale quantization, ranks against the oracle;
* exhaustive float32 scanning (pvs_cursor_set_generator, PVS_GEN_FULL_SCAN);
* both inside EAHR give the same Top-K as PVS (Sec. 2.2: the result does
  not depend on the generator).
"""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po
from oracle import rrf_oracle as ro

pytestmark = pytest.mark.gpu


def corpus(n, m, seed):
    rng = np.random.default_rng(seed)
    # rows of very different norms: the one-scale index is coarse for most
    return (rng.standard_normal((n, m)) * rng.gamma(0.8, 1.0, size=(n, 1))).astype(np.float32)


def pull_all(cur, chunk):
    ids, sc = [], []
    while True:
        i, s, st = pvs.pvs_next(cur, chunk)
        ids.append(i)
        sc.append(s)
        if st == pvs.PVS_EXHAUSTED:
            return np.concatenate(ids), np.concatenate(sc)


@pytest.mark.parametrize("on_device", [False, True])
def test_global_scale_index_matches_the_oracle(on_device):
    n, m = 3001, 96
    V = corpus(n, m, 71)
    Q = po.quantize_global(V)
    src = torch.from_numpy(V).cuda() if on_device else V
    index = pvs.pvs_build(src, quantization=pvs.PVS_QUANT_GLOBAL)
    try:
        codes, scale, vnorm, enorm = pvs.pvs_index_export(index, 0, n)
        assert np.array_equal(codes, Q.z)
        assert np.array_equal(scale.view(np.uint32), Q.s.view(np.uint32))
        assert np.all(scale == po.global_scale(V))
        assert np.array_equal(vnorm.view(np.uint32), Q.vnorm.view(np.uint32))
        assert np.array_equal(enorm.view(np.uint32), Q.enorm.view(np.uint32))
        q = synth.unit_normal(1, m, seed=72).numpy()[0]
        qe = po.encode_query(q)
        ref_lo, ref_hi = po.intervals(qe, Q, m)
        cur = pvs.pvs_cursor_open(index, q)
        try:
            lo, hi = pvs.pvs_cursor_bounds(cur, 0, n)
        finally:
            pvs.pvs_cursor_close(cur)
        assert np.array_equal(lo.view(np.uint32), ref_lo.view(np.uint32))
        assert np.array_equal(hi.view(np.uint32), ref_hi.view(np.uint32))
        # the complete ranking, pulled in ragged chunks
        cur = pvs.pvs_cursor_open(index, q)
        try:
            ids, sc = pull_all(cur, 97)
            refined_sq = pvs.pvs_cursor_stats(cur)["refined"]
        finally:
            pvs.pvs_cursor_close(cur)
        ref_ids, ref_sc = po.dense_ranking(q, V)
        assert np.array_equal(ids, ref_ids)
        assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
    finally:
        pvs.pvs_index_free(index)


def test_global_scale_intervals_are_wider_so_more_rows_are_refined():
    n, m = 20_000, 128
    V = corpus(n, m, 73)
    q = synth.unit_normal(1, m, seed=74).numpy()[0]
    refined = {}
    for quant in (pvs.PVS_QUANT_PER_VECTOR, pvs.PVS_QUANT_GLOBAL):
        index = pvs.pvs_build(V, quantization=quant)
        try:
            cur = pvs.pvs_cursor_open(index, q)
            try:
                for _ in range(10):
                    pvs.pvs_next(cur, 20)
                refined[quant] = pvs.pvs_cursor_stats(cur)["refined"]
            finally:
                pvs.pvs_cursor_close(cur)
        finally:
            pvs.pvs_index_free(index)
    assert refined[pvs.PVS_QUANT_GLOBAL] > refined[pvs.PVS_QUANT_PER_VECTOR]


def test_global_scale_append_in_and_out_of_range():
    m = 32
    V = corpus(500, m, 75)
    s = po.global_scale(V)
    index = pvs.pvs_build(V, quantization=pvs.PVS_QUANT_GLOBAL)
    try:
        W = (V[:50] * 0.5).astype(np.float32)          # inside the scale's range
        pvs.pvs_append(index, W)
        codes, scale, _, enorm = pvs.pvs_index_export(index, 500, 50)
        Qw = po.quantize_global(W, s=s)
        assert np.array_equal(codes, Qw.z) and np.all(scale == s)
        assert np.array_equal(enorm.view(np.uint32), Qw.enorm.view(np.uint32))
        big = np.zeros((1, m), np.float32)
        big[0, 0] = 2.0 * float(np.abs(V).max())        # codes would leave [-127, 127]
        with pytest.raises(pvs.PvsError) as e:
            pvs.pvs_append(index, big)
        assert e.value.status == pvs.PVS_ERR_INVALID
        assert pvs.pvs_index_size(index) == 550
    finally:
        pvs.pvs_index_free(index)


def test_full_scan_generator_matches_the_oracle_with_deletions():
    n, m = 5003, 64
    V = synth.unit_normal(n, m, seed=76).numpy()
    q = synth.unit_normal(1, m, seed=77).numpy()[0]
    index = pvs.pvs_build(V)
    try:
        dead = np.arange(0, n, 7, dtype=np.int64)
        pvs.pvs_tombstone(index, dead)
        snap = pvs.pvs_snapshot_create(index)
        try:
            cur = pvs.pvs_cursor_open(index, q, snap=snap)
            try:
                pvs.pvs_cursor_set_generator(cur, pvs.PVS_GEN_FULL_SCAN)
                ids, sc = pull_all(cur, 301)
                st = pvs.pvs_cursor_stats(cur)
                with pytest.raises(pvs.PvsError):
                    pvs.pvs_cursor_set_generator(cur, pvs.PVS_GEN_INTERVALS)
            finally:
                pvs.pvs_cursor_close(cur)
        finally:
            pvs.pvs_snapshot_free(snap)
    finally:
        pvs.pvs_index_free(index)
    live = np.ones(n, bool)
    live[dead] = False
    ref_ids, ref_sc = po.dense_ranking(q, V, live)
    assert np.array_equal(ids, ref_ids)
    assert np.array_equal(sc.view(np.uint32), ref_sc.view(np.uint32))
    assert st["refined"] == live.sum()          # every visible row scored exactly once


def test_generator_argument_errors():
    V = synth.unit_normal(100, 16, seed=78).numpy()
    index = pvs.pvs_build(V)
    try:
        cur = pvs.pvs_cursor_open(index, V[0])
        try:
            with pytest.raises(pvs.PvsError):
                pvs.pvs_cursor_set_generator(cur, 7)
            pvs.pvs_next(cur, 5)
            with pytest.raises(pvs.PvsError):
                pvs.pvs_cursor_set_generator(cur, pvs.PVS_GEN_FULL_SCAN)
        finally:
            pvs.pvs_cursor_close(cur)
        with pytest.raises(pvs.PvsError):
            pvs.pvs_build(V, quantization=5)
    finally:
        pvs.pvs_index_free(index)


def test_eahr_result_does_not_depend_on_the_generator():
    n, m = 40_000, 64
    centres = synth.mixture_centres(64, m, seed=79, device="cpu")
    V = synth.mixture_rows(n, centres, 0.35, seed=79).numpy()
    q = synth.mixture_queries(1, centres, 0.5, seed=80).numpy()[0]
    dense_ids, dense_sc = po.dense_ranking(q, V)
    proxy = torch.from_numpy(dense_sc[np.argsort(dense_ids)].astype(np.float64))
    sparse = synth.copula_ranking(proxy, 0.5, seed=81).numpy()
    T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
    want = [x for x, _ in T]
    for quant, gen in ((pvs.PVS_QUANT_PER_VECTOR, pvs.PVS_GEN_INTERVALS),
                       (pvs.PVS_QUANT_GLOBAL, pvs.PVS_GEN_INTERVALS),
                       (pvs.PVS_QUANT_PER_VECTOR, pvs.PVS_GEN_FULL_SCAN)):
        index = pvs.pvs_build(V, quantization=quant)
        try:
            cur = pvs.pvs_cursor_open(index, q)
            try:
                pvs.pvs_cursor_set_generator(cur, gen)
                ids, F, st = pvs.eahr_topk(cur, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR)
            finally:
                pvs.pvs_cursor_close(cur)
        finally:
            pvs.pvs_index_free(index)
        assert ids.tolist() == want, (quant, gen)
