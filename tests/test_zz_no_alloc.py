"""pvs_rank_exact_noalloc: exact ranking without any device allocation.

Some callers cannot allocate device memory where they need a ranking:
services whose device memory belongs to a pool or budget of their own, where
an allocation outside it fails or breaks the pool's accounting, and
latency-critical callers, for whom cudaMalloc is slow and cudaFree waits for
the whole device.  For them the library keeps the ranking's scratch in a
fixed static device array.

These tests call it through the C ABI and compare it with the oracle's
complete dense ranking (Sec. 2.1: authoritative scores, ties by ascending
id): identical ids in identical order and bit-identical float32 scores, the
bar every parity test here uses.  Each case makes two calls in a row, and
the second ranks fewer rows than the first, so keys the first call left in
the shared array must not leak into its result.  This file is collected
last, so a run that stops at the first failure has run every other test.
"""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po

pytestmark = pytest.mark.gpu

MAX = pvs.PVS_NOALLOC_MAX_VECTORS


def _outs(k=MAX):
    return (torch.full((max(k, 1),), -7, dtype=torch.int64, device="cuda"),
            torch.full((max(k, 1),), float("nan"), dtype=torch.float32, device="cuda"))


def _check_against_oracle(q, V, top, out_ids, out_scores):
    pvs.pvs_rank_exact_noalloc(q, V, top, out_ids, out_scores)
    torch.cuda.synchronize()
    got_ids = out_ids[:top].cpu().numpy()
    got_scores = out_scores[:top].cpu().numpy()
    ref_ids, ref_scores = po.dense_ranking(q.cpu().numpy(), V.cpu().numpy())
    assert np.array_equal(got_ids, ref_ids[:top])
    assert np.array_equal(got_scores.view(np.uint32), ref_scores[:top].view(np.uint32))


def test_noalloc_matches_oracle_on_two_calls_in_a_row():
    torch.cuda.set_device(0)
    V = synth.unit_normal(MAX, 96, seed=21, device="cuda")
    Q = synth.unit_normal(3, 96, seed=22, device="cuda")
    out_ids, out_scores = _outs()
    # the full scratch (n = 8192, every rank), then fewer rows with top < n
    _check_against_oracle(Q[0].contiguous(), V, MAX, out_ids, out_scores)
    _check_against_oracle(Q[1].contiguous(), V[:3000].contiguous(), 500, out_ids, out_scores)
    # a ragged size that is no power of two, every rank
    _check_against_oracle(Q[2].contiguous(), V[:1237].contiguous(), 1237, out_ids, out_scores)


def test_noalloc_exact_ties_go_to_ascending_row_number():
    torch.cuda.set_device(0)
    base = synth.unit_normal(40, 32, seed=23, device="cuda")
    # every row appears three times: equal scores, ranked by row number
    V = base.repeat(3, 1).contiguous()
    q = synth.unit_normal(1, 32, seed=24, device="cuda")[0].contiguous()
    out_ids, out_scores = _outs(120)
    _check_against_oracle(q, V, 120, out_ids, out_scores)
    _check_against_oracle(q, V[:50].contiguous(), 17, out_ids, out_scores)


def test_noalloc_empty_input_and_top_zero_write_nothing():
    torch.cuda.set_device(0)
    q = synth.unit_normal(1, 16, seed=25, device="cuda")[0].contiguous()
    out_ids, out_scores = _outs(8)
    empty = torch.zeros((0, 16), device="cuda")
    assert pvs.pvs_rank_exact_noalloc(q, empty, 0, out_ids, out_scores) == pvs.PVS_OK
    V = synth.unit_normal(64, 16, seed=26, device="cuda")
    assert pvs.pvs_rank_exact_noalloc(q, V, 0, out_ids, out_scores) == pvs.PVS_OK
    torch.cuda.synchronize()
    assert (out_ids.cpu() == -7).all() and torch.isnan(out_scores.cpu()).all()
    # and the array works again afterwards
    _check_against_oracle(q, V, 64, *_outs(64))


def test_noalloc_rejects_sizes_beyond_its_scratch_and_bad_input():
    torch.cuda.set_device(0)
    out_ids, out_scores = _outs(16)
    q = torch.ones(16, device="cuda")
    too_many = torch.zeros((MAX + 1, 16), device="cuda")
    with pytest.raises(pvs.PvsError) as e:
        pvs.pvs_rank_exact_noalloc(q, too_many, 10, out_ids, out_scores)
    assert e.value.status == pvs.PVS_ERR_INVALID
    bad = torch.ones((40, 16), device="cuda")
    bad[7, 3] = float("nan")
    with pytest.raises(pvs.PvsError) as e:
        pvs.pvs_rank_exact_noalloc(q, bad, 10, out_ids, out_scores)
    assert e.value.status == pvs.PVS_ERR_NONFINITE
    good = torch.ones((40, 16), device="cuda")
    qbad = torch.ones(16, device="cuda")
    qbad[5] = float("inf")
    with pytest.raises(pvs.PvsError) as e:
        pvs.pvs_rank_exact_noalloc(qbad, good, 10, out_ids, out_scores)
    assert e.value.status == pvs.PVS_ERR_NONFINITE
    # shape and type errors the library cannot see through raw pointers
    with pytest.raises(ValueError):
        pvs.pvs_rank_exact_noalloc(torch.ones(15, device="cuda"), good, 10, out_ids, out_scores)
    with pytest.raises(ValueError):
        pvs.pvs_rank_exact_noalloc(q, good, 17, out_ids, out_scores)
    with pytest.raises(ValueError):
        pvs.pvs_rank_exact_noalloc(q, good, 41, *_outs(64))
    with pytest.raises(TypeError):
        pvs.pvs_rank_exact_noalloc(q.double(), good, 10, out_ids, out_scores)
    with pytest.raises(TypeError):
        pvs.pvs_rank_exact_noalloc(q, good, 10, out_ids.int(), out_scores)
    # a good call right after the failures still matches the oracle
    V = synth.unit_normal(40, 16, seed=27, device="cuda")
    _check_against_oracle(q, V, 40, *_outs(40))
