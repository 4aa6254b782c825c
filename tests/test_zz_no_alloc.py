"""pvs_rank_exact_noalloc: exact ranking without any device allocation.

Some callers cannot allocate device memory where they need a ranking: code
that runs while a CUDA stream is being captured into a graph, where
cudaMalloc is not permitted, and services whose memory pool already owns the
device memory budget.  For them the library keeps the ranking's scratch in a
fixed static device array.  These tests check, through the C ABI, that two
calls in a row return exactly what the cursor path (pvs_cursor_open +
pvs_next) returns for the same rows and query.  The second call ranks fewer
rows than the first, so keys the first call left in the shared array must
not leak into its result.  The bar is the one every parity test here uses:
identical ids in identical order and bit-identical float32 scores.
"""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth

pytestmark = pytest.mark.gpu


def _cursor_ranking(vecs, q, top):
    index = pvs.pvs_build(vecs)
    try:
        cur = pvs.pvs_cursor_open(index, q)
        try:
            ids, scores, _ = pvs.pvs_next(cur, top)
        finally:
            pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)
    return ids, scores


def test_noalloc_matches_cursor_path_on_two_calls_in_a_row():
    torch.cuda.set_device(0)
    V = synth.unit_normal(6000, 96, seed=21, device="cuda")
    Q = synth.unit_normal(2, 96, seed=22, device="cuda")
    out_ids = torch.empty(pvs.PVS_NOALLOC_MAX_VECTORS, dtype=torch.int64, device="cuda")
    out_scores = torch.empty(pvs.PVS_NOALLOC_MAX_VECTORS, dtype=torch.float32, device="cuda")
    cases = [(Q[0].contiguous(), V, 500),
             (Q[1].contiguous(), V[:3000].contiguous(), 3000)]
    for q, vecs, top in cases:
        pvs.pvs_rank_exact_noalloc(q, vecs, top, out_ids, out_scores)
        torch.cuda.synchronize()
        got_ids = out_ids[:top].cpu().numpy()
        got_scores = out_scores[:top].cpu().numpy()
        ref_ids, ref_scores = _cursor_ranking(vecs, q, top)
        assert np.array_equal(got_ids, ref_ids)
        assert np.array_equal(got_scores.view(np.uint32), ref_scores.view(np.uint32))


def test_noalloc_rejects_sizes_beyond_its_scratch_and_bad_input():
    torch.cuda.set_device(0)
    out_ids = torch.empty(16, dtype=torch.int64, device="cuda")
    out_scores = torch.empty(16, dtype=torch.float32, device="cuda")
    q = torch.ones(16, device="cuda")
    too_many = torch.zeros((pvs.PVS_NOALLOC_MAX_VECTORS + 1, 16), device="cuda")
    with pytest.raises(pvs.PvsError) as e:
        pvs.pvs_rank_exact_noalloc(q, too_many, 10, out_ids, out_scores)
    assert e.value.status == pvs.PVS_ERR_INVALID
    bad = torch.ones((40, 16), device="cuda")
    bad[7, 3] = float("nan")
    with pytest.raises(pvs.PvsError) as e:
        pvs.pvs_rank_exact_noalloc(q, bad, 10, out_ids, out_scores)
    assert e.value.status == pvs.PVS_ERR_NONFINITE
