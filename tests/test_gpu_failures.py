"""The failure rules of the ranked-list contract, reached without a GPU fault
(arXiv 2608.07152 Sec. 2.1: a Failed list invalidates the request;
App. A.1: an authoritative score outside its interval fails the request).

  * interval violation: an index imported with one row's scale made wrong
    on the host (pvs_index_import) gives that row an interval that misses
    its exact score; the pull that scores it fails with PVS_ERR_INTERVAL,
    the cursor stays Failed, and EAHR returns the error with no result;
  * device wait timeout: with the index's wait limit at 0 the interval
    pass's waits give up instead of waiting for their tiles (the pass still
    waits for its own copies in flight before it exits); the pull fails with
    PVS_ERR_TIMEOUT, and with the limit restored a fresh cursor on the same
    index returns exact ranks.
"""
import ctypes

import numpy as np
import pytest

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po

pytestmark = pytest.mark.gpu


def _eahr_raw(cur, sparse):
    """eahr_topk through the C ABI, returning (status, n_out)."""
    sp = np.ascontiguousarray(sparse, dtype=np.int64)
    p = pvs._params(20, 60, pvs.EAHR_NUMERATOR, pvs.EAHR_POLICY_GEOMETRIC, 0, (1, 1))
    ids = np.full(20, -1, np.int64)
    F = np.zeros(20, np.float64)
    got = ctypes.c_int32(7)
    st = pvs.eahr_stats()
    rc = pvs._lib.eahr_topk(cur, sp.ctypes.data, sp.size, ctypes.byref(p), ids.ctypes.data,
                            F.ctypes.data, ctypes.byref(got), ctypes.byref(st))
    return rc, got.value, ids


def _exported(index, n, dim):
    codes = np.zeros((n, dim), np.int8)
    scale, vnorm, enorm = (np.zeros(n, np.float32) for _ in range(3))
    pvs._check(pvs._lib.pvs_index_export(index, 0, n, codes.ctypes.data, scale.ctypes.data,
                                         vnorm.ctypes.data, enorm.ctypes.data), "export")
    return codes, scale, vnorm, enorm


def test_imported_index_ranks_exactly_and_a_wrong_scale_fails_the_request():
    n, dim, r = 20_000, 128, 1234
    V = synth.unit_normal(n, dim, seed=71).numpy()
    rng = np.random.default_rng(72)
    q = V[r] + 0.05 * rng.standard_normal(dim).astype(np.float32)
    q = (q / np.linalg.norm(q)).astype(np.float32)
    ref_ids, ref_sc = po.dense_ranking(q, V)
    assert ref_ids[0] == r
    built = pvs.pvs_build(V)
    try:
        codes, scale, vnorm, enorm = _exported(built, n, dim)
    finally:
        pvs.pvs_index_free(built)
    # the parameters as exported: the imported index ranks exactly
    good = pvs.pvs_index_import(V, codes, scale, vnorm, enorm)
    try:
        cur = pvs.pvs_cursor_open(good, q)
        try:
            ids, sc, _ = pvs.pvs_next(cur, 200)
        finally:
            pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(good)
    assert np.array_equal(ids, ref_ids[:200])
    assert np.array_equal(sc.view(np.uint32), ref_sc[:200].view(np.uint32))
    # row r's scale 1.5x too large: its interval sits around 1.5 x its
    # score, above the exact value, and r is the first row refined
    bad_scale = scale.copy()
    bad_scale[r] *= np.float32(1.5)
    bad = pvs.pvs_index_import(V, codes, bad_scale, vnorm, enorm)
    try:
        cur = pvs.pvs_cursor_open(bad, q)
        try:
            lo, hi = pvs.pvs_cursor_bounds(cur, r, 1)
            assert lo[0] > ref_sc[0]                   # the interval misses the score
            with pytest.raises(pvs.PvsError) as e:
                pvs.pvs_next(cur, 20)
            assert e.value.status == pvs.PVS_ERR_INTERVAL
            with pytest.raises(pvs.PvsError) as e:     # Failed for good
                pvs.pvs_next(cur, 20)
            assert e.value.status == pvs.PVS_ERR_FAILED
            assert pvs.pvs_cursor_stats(cur)["state"] == pvs.PVS_ERR_INTERVAL
        finally:
            pvs.pvs_cursor_close(cur)
        # EAHR over such a cursor returns the failure and no partial result
        cur = pvs.pvs_cursor_open(bad, q)
        try:
            rc, n_out, ids = _eahr_raw(cur, np.arange(n)[::-1])
        finally:
            pvs.pvs_cursor_close(cur)
        assert rc == pvs.PVS_ERR_INTERVAL and n_out == 0
    finally:
        pvs.pvs_index_free(bad)


def test_import_rejects_what_the_kernels_rely_on():
    V = synth.unit_normal(8, 16, seed=73).numpy()
    codes = np.zeros((8, 16), np.int8)
    ones = np.ones(8, np.float32)
    for args, code in (
            ((V, np.full((8, 16), -128, np.int8), ones, ones, ones), pvs.PVS_ERR_INVALID),
            ((V, codes, np.zeros(8, np.float32), ones, ones), pvs.PVS_ERR_INVALID),
            ((V, codes, ones, -ones, ones), pvs.PVS_ERR_INVALID),
            ((V, codes, ones, ones, np.full(8, np.inf, np.float32)), pvs.PVS_ERR_INVALID),
            ((np.where(np.eye(8, 16) > 0, np.nan, V).astype(np.float32), codes, ones, ones,
              ones), pvs.PVS_ERR_NONFINITE)):
        with pytest.raises(pvs.PvsError) as e:
            pvs.pvs_index_import(*args)
        assert e.value.status == code


def test_device_wait_timeout_fails_the_cursor_and_the_index_recovers():
    n, dim = 400_000, 256
    V = synth.unit_normal(n, dim, seed=74, device="cuda")
    q = synth.unit_normal(1, dim, seed=75).numpy()[0]
    index = pvs.pvs_build(V)
    try:
        with pytest.raises(pvs.PvsError) as e:
            pvs.pvs_index_set_wait_limit(index, -1)
        assert e.value.status == pvs.PVS_ERR_INVALID
        pvs.pvs_index_set_wait_limit(index, 0)
        cur = pvs.pvs_cursor_open(index, q)
        try:
            with pytest.raises(pvs.PvsError) as e:
                pvs.pvs_next(cur, 20)
            assert e.value.status == pvs.PVS_ERR_TIMEOUT
            with pytest.raises(pvs.PvsError) as e:
                pvs.pvs_next(cur, 20)
            assert e.value.status == pvs.PVS_ERR_FAILED
            assert pvs.pvs_cursor_stats(cur)["state"] == pvs.PVS_ERR_TIMEOUT
        finally:
            pvs.pvs_cursor_close(cur)
        cur = pvs.pvs_cursor_open(index, q)
        try:
            rc, n_out, _ = _eahr_raw(cur, np.arange(n))
        finally:
            pvs.pvs_cursor_close(cur)
        assert rc == pvs.PVS_ERR_TIMEOUT and n_out == 0
        # the context is intact: restore the limit, open a fresh cursor
        pvs.pvs_index_set_wait_limit(index, 2_000_000_000)
        cur = pvs.pvs_cursor_open(index, q)
        try:
            ids, sc, _ = pvs.pvs_next(cur, 100)
        finally:
            pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)
    ref_ids, ref_sc = po.dense_ranking(q, V.cpu().numpy())
    assert np.array_equal(ids, ref_ids[:100])
    assert np.array_equal(sc.view(np.uint32), ref_sc[:100].view(np.uint32))
