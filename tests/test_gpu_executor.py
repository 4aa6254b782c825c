"""Native request executor through the C ABI (include/executor.h): requests
paged through the host path (arXiv 2608.07152 Sec. 2.1) over PVS cursors
(Sec. 2.3) equal the oracle's complete ranking, request by request, in ids
and in the bits of the authoritative scores."""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po

pytestmark = pytest.mark.gpu


def _mixture(n, m, nq, seed, comps=32):
    centres = synth.mixture_centres(comps, m, seed=seed, device="cpu")
    V = synth.mixture_rows(n, centres, 0.35, seed=seed + 1).numpy()
    Q = synth.mixture_queries(nq, centres, 0.5, seed=seed + 2).numpy()
    return V, Q


def _check_rows(V, Q, ids, sc, n_out, ranks, visible=None, rows=None):
    for i in (range(Q.shape[0]) if rows is None else rows):
        ref_ids, ref_sc = po.dense_ranking(Q[i], V, visible)
        k = min(ranks, ref_ids.size)
        assert n_out[i] == k, i
        assert np.array_equal(ids[i, :k], ref_ids[:k]), i
        assert np.array_equal(sc[i, :k].view(np.uint32), ref_sc[:k].view(np.uint32)), i
        assert np.all(ids[i, k:] == -1) and np.all(np.isnan(sc[i, k:])), i


@pytest.mark.parametrize("workers,ranks,page", [(4, 300, 20), (3, 101, 7), (8, 64, 64), (1, 50, 13)])
def test_requests_equal_the_oracle_ranking(workers, ranks, page):
    V, Q = _mixture(9_001, 96, 23, seed=workers * 100 + page)
    index = pvs.pvs_build(V)
    try:
        ex = pvs.pvs_executor_create(index, workers)
        try:
            ids, sc, n_out, status, rc = pvs.pvs_executor_run(ex, Q, ranks, page)
            st = pvs.pvs_executor_stats(ex)
        finally:
            pvs.pvs_executor_destroy(ex)
    finally:
        pvs.pvs_index_free(index)
    assert rc == pvs.PVS_OK and np.all(status == pvs.PVS_OK)
    _check_rows(V, Q, ids, sc, n_out, ranks)
    pages_per_request = -(-ranks // page)
    assert st["requests"] == 23 and st["failed"] == 0 and st["workers"] == workers
    assert st["pages"] == 23 * pages_per_request and st["ranks"] == 23 * ranks


def test_pinned_buffers_repeated_runs_and_exhaustion():
    V, Q = _mixture(61, 32, 17, seed=5, comps=4)
    index = pvs.pvs_build(V)
    try:
        ex = pvs.pvs_executor_create(index, 5)
        try:
            q = torch.from_numpy(Q).pin_memory()
            ids = torch.empty((17, 80), dtype=torch.int64).pin_memory()
            sc = torch.empty((17, 80), dtype=torch.float32).pin_memory()
            for _ in range(3):   # one executor, several runs into the same buffers
                _, _, n_out, status, rc = pvs.pvs_executor_run(ex, q, 80, 9, ids=ids, scores=sc)
                assert rc == pvs.PVS_OK
                assert np.all(status == pvs.PVS_EXHAUSTED) and np.all(n_out == 61)
                _check_rows(V, Q, ids.numpy(), sc.numpy(), n_out, 80)
            st = pvs.pvs_executor_stats(ex)
            assert st["requests"] == 51 and st["ranks"] == 51 * 61
            # no requests
            out = pvs.pvs_executor_run(ex, np.zeros((0, 32), np.float32), 10, 5)
            assert out[4] == pvs.PVS_OK and out[0].shape == (0, 10)
        finally:
            pvs.pvs_executor_destroy(ex)
    finally:
        pvs.pvs_index_free(index)


def test_a_failed_request_leaves_the_others_exact():
    V, Q = _mixture(4_000, 64, 12, seed=7)
    Q[5, 3] = np.nan
    index = pvs.pvs_build(V)
    try:
        ex = pvs.pvs_executor_create(index, 4)
        try:
            ids, sc, n_out, status, rc = pvs.pvs_executor_run(ex, Q, 120, 20)
            st = pvs.pvs_executor_stats(ex)
        finally:
            pvs.pvs_executor_destroy(ex)
    finally:
        pvs.pvs_index_free(index)
    assert status[5] == pvs.PVS_ERR_NONFINITE and rc == pvs.PVS_ERR_NONFINITE
    assert n_out[5] == 0 and np.all(ids[5] == -1)
    assert st["failed"] == 1
    _check_rows(V, Q, ids, sc, n_out, 120, rows=[i for i in range(12) if i != 5])


def test_snapshots_and_appends_order_with_the_executor():
    V, Q = _mixture(6_000, 64, 9, seed=9)
    W = synth.mixture_rows(2_000, synth.mixture_centres(32, 64, seed=9, device="cpu"), 0.35,
                           seed=99).numpy()
    index = pvs.pvs_build(V)
    snap = None
    try:
        rng = np.random.default_rng(4)
        dead = rng.choice(6_000, 300, replace=False)
        pvs.pvs_tombstone(index, dead)
        snap = pvs.pvs_snapshot_create(index)
        ex = pvs.pvs_executor_create(index, 3)
        try:
            pvs.pvs_append(index, W)            # after the snapshot, before the run
            ids, sc, n_out, status, rc = pvs.pvs_executor_run(ex, Q, 150, 25, snap=snap)
            assert rc == pvs.PVS_OK
            vis = np.ones(6_000, bool)
            vis[dead] = False
            _check_rows(V, Q, ids, sc, n_out, 150, visible=vis)
            # the current visible set includes the appended rows
            ids, sc, n_out, status, rc = pvs.pvs_executor_run(ex, Q, 150, 25)
            assert rc == pvs.PVS_OK
            full = np.concatenate([V, W])
            vis_all = np.ones(8_000, bool)
            vis_all[dead] = False
            _check_rows(full, Q, ids, sc, n_out, 150, visible=vis_all)
        finally:
            pvs.pvs_executor_destroy(ex)
    finally:
        if snap is not None:
            pvs.pvs_snapshot_free(snap)
        pvs.pvs_index_free(index)


def test_executor_argument_errors():
    V, Q = _mixture(500, 16, 3, seed=11, comps=4)
    index = pvs.pvs_build(V)
    other = pvs.pvs_build(V)
    try:
        with pytest.raises(pvs.PvsError):
            pvs.pvs_executor_create(index, 0)
        with pytest.raises(pvs.PvsError):
            pvs.pvs_executor_create(index, 65)
        ex = pvs.pvs_executor_create(index, 2)
        snap = pvs.pvs_snapshot_create(other)
        try:
            for ranks, page in ((0, 1), (10, 0), (10, 11)):
                with pytest.raises(pvs.PvsError):
                    pvs.pvs_executor_run(ex, Q, ranks, page)
            with pytest.raises(pvs.PvsError):   # a snapshot of another index
                pvs.pvs_executor_run(ex, Q, 10, 5, snap=snap)
            assert pvs.pvs_executor_stats(ex)["requests"] == 0
        finally:
            pvs.pvs_snapshot_free(snap)
            pvs.pvs_executor_destroy(ex)
    finally:
        pvs.pvs_index_free(other)
        pvs.pvs_index_free(index)


@pytest.mark.parametrize("group,workers", [(8, 3), (3, 2), (5, 1)])
def test_grouped_requests_equal_the_oracle_ranking(group, workers):
    """Requests served `group` at a time share one pass over the codes
    (pvs_cursor_open_group) and one batched pull per page; every request's
    ranks are still the oracle's."""
    V, Q = _mixture(9_001, 96, 23, seed=300 + group)
    index = pvs.pvs_build(V)
    try:
        ex = pvs.pvs_executor_create(index, workers)
        try:
            pvs.pvs_executor_set_group(ex, group)
            ids, sc, n_out, status, rc = pvs.pvs_executor_run(ex, Q, 300, 20)
            st = pvs.pvs_executor_stats(ex)
        finally:
            pvs.pvs_executor_destroy(ex)
    finally:
        pvs.pvs_index_free(index)
    assert rc == pvs.PVS_OK and np.all(status == pvs.PVS_OK)
    _check_rows(V, Q, ids, sc, n_out, 300)
    assert st["group"] == group and st["interval_passes"] == -(-23 // group)
    assert st["requests"] == 23 and st["failed"] == 0 and st["ranks"] == 23 * 300
    assert st["interval_ms"] > 0 and st["refined"] >= 23 * 300


@pytest.mark.parametrize("group", [1, 8])
def test_device_buffers_grouped_and_not(group):
    V, Q = _mixture(12_345, 128, 19, seed=400 + group)
    index = pvs.pvs_build(V)
    try:
        ex = pvs.pvs_executor_create(index, 4)
        try:
            pvs.pvs_executor_set_group(ex, group)
            q = torch.from_numpy(Q).cuda()
            ids = torch.zeros((19, 250), dtype=torch.int64, device="cuda")
            sc = torch.zeros((19, 250), dtype=torch.float32, device="cuda")
            n_out, status, rc = pvs.pvs_executor_run_device(ex, q, 250, 20, ids, sc)
        finally:
            pvs.pvs_executor_destroy(ex)
    finally:
        pvs.pvs_index_free(index)
    assert rc == pvs.PVS_OK and np.all(status == pvs.PVS_OK)
    _check_rows(V, Q, ids.cpu().numpy(), sc.cpu().numpy(), n_out, 250)


def test_grouped_requests_with_exhaustion_and_a_failed_query():
    V, Q = _mixture(61, 32, 17, seed=15, comps=4)
    index = pvs.pvs_build(V)
    try:
        ex = pvs.pvs_executor_create(index, 2)
        try:
            pvs.pvs_executor_set_group(ex, 8)
            _, _, n_out, status, rc = pvs.pvs_executor_run(ex, Q, 80, 9)
            assert rc == pvs.PVS_OK and np.all(status == pvs.PVS_EXHAUSTED)
            ids, sc, n_out, status, rc = pvs.pvs_executor_run(ex, Q, 80, 9)
            _check_rows(V, Q, ids, sc, n_out, 80)
            bad = Q.copy()
            bad[9, 1] = np.inf        # the second group's open fails; its others go on
            ids, sc, n_out, status, rc = pvs.pvs_executor_run(ex, bad, 80, 9)
            assert status[9] == pvs.PVS_ERR_NONFINITE and rc == pvs.PVS_ERR_NONFINITE
            assert n_out[9] == 0 and np.all(ids[9] == -1)
            _check_rows(V, Q, ids, sc, n_out, 80, rows=[i for i in range(17) if i != 9])
            with pytest.raises(pvs.PvsError):
                pvs.pvs_executor_set_group(ex, pvs.PVS_GROUP_MAX + 1)
        finally:
            pvs.pvs_executor_destroy(ex)
    finally:
        pvs.pvs_index_free(index)
