"""Parity at full size and in deep pulls, through the C ABI.

* Passage scale (8,841,823 x 768, the mixture corpus of the benchmark), in
  the launch configuration the benchmark times -- the native executor with
  four workers, eight queries per grouped pass over the codes, 50 batched
  pulls of 20 ranks into device buffers -- and for a lone cursor on its own
  stream (the latency figures' path).  The oracle cannot rank 8.8M rows
  in a test, so it checks what it can compute one by one and what holds at
  any size (Sec. 2.1, 2.3.1, App. A.1):
    - every emitted score equals the oracle's exact score of that row;
    - the emitted order is (score desc, id asc);
    - no row of a 100,000-row sample outside the emitted set beats the last
      emitted rank;
    - the intervals of a sample of rows (including every emitted row) are
      bit-identical to the oracle's and contain the exact scores.
* EAHR with lists that are read deep or to the end (Sec. 2.2): the dense
  cursor serves pulls of up to 131,072 ranks (the multi-kernel path with the
  device radix sort) and the result equals complete-list fusion.
"""
import numpy as np
import pytest
import torch

import paper_2608_07152_gb300 as pvs
import synth
from oracle import pvs_oracle as po
from oracle import rrf_oracle as ro

pytestmark = pytest.mark.gpu

N_PASSAGE = 8_841_823
DIM = 768


@pytest.fixture(scope="module")
def passage():
    dev = torch.device("cuda")
    centres = synth.mixture_centres(4096, DIM, seed=2, device=dev)
    rows = torch.empty((N_PASSAGE, DIM), dtype=torch.float32, device=dev)
    for r in range(0, N_PASSAGE, 1 << 20):
        c = min(1 << 20, N_PASSAGE - r)
        rows[r:r + c] = synth.mixture_rows(c, centres, 0.35, seed=2, first=r)
    index = pvs.pvs_build(rows)
    try:
        yield dev, centres, rows, index
    finally:
        pvs.pvs_index_free(index)


def _check_prefix(rows, dev, qh, ids, sc, sample):
    """The three checks of a first-1,000 prefix that the oracle can make at
    this size: exact scores of the emitted rows, (score desc, id asc) order,
    and nothing of a row sample outside the prefix ahead of its last rank."""
    V_ids = rows[torch.from_numpy(ids).to(dev)].cpu().numpy()
    ref = np.array([po.exact_score_one(qh, v) for v in V_ids], np.float32)
    assert np.array_equal(sc.view(np.uint32), ref.view(np.uint32))
    key = list(zip((-sc.astype(np.float64)).tolist(), ids.tolist()))
    assert key == sorted(key)
    assert len(set(ids.tolist())) == ids.size
    Vs = rows[torch.from_numpy(sample).to(dev)].cpu().numpy()
    s_sample = po.exact_scores(qh, Vs)
    emitted = set(ids.tolist())
    last_s, last_id = float(sc[-1]), int(ids[-1])
    for i, s in zip(sample.tolist(), s_sample.tolist()):
        if i not in emitted:
            assert s < last_s or (s == last_s and i > last_id), i
    return s_sample


def test_passage_scale_grouped_executor_in_the_benchmark_configuration(passage):
    dev, centres, rows, index = passage
    Q = synth.mixture_queries(16, centres, 0.5, seed=3).contiguous()
    ids_t = torch.empty((16, 1000), dtype=torch.int64, device=dev)
    sc_t = torch.empty((16, 1000), dtype=torch.float32, device=dev)
    ex = pvs.pvs_executor_create(index, 4)
    try:
        pvs.pvs_executor_set_group(ex, 8)
        n_out, status, rc = pvs.pvs_executor_run_device(ex, Q, 1000, 20, ids_t, sc_t)
        st = pvs.pvs_executor_stats(ex)
    finally:
        pvs.pvs_executor_destroy(ex)
    assert rc == pvs.PVS_OK and np.all(n_out == 1000)
    assert st["interval_passes"] == 2          # two groups of eight, one pass each
    ids_all, sc_all = ids_t.cpu().numpy(), sc_t.cpu().numpy()
    Qh = Q.cpu().numpy()
    rng = np.random.default_rng(6)
    base = rng.integers(0, N_PASSAGE, 50_000)
    for i in range(16):
        sample = np.unique(np.concatenate([base, ids_all[i]]))
        _check_prefix(rows, dev, Qh[i], ids_all[i], sc_all[i], sample)
    # the grouped pass's bounds of a row sample: the oracle's, for each query
    first = np.unique(rng.integers(0, N_PASSAGE, 3000))
    Qs = po.quantize(rows[torch.from_numpy(first).to(dev)].cpu().numpy())
    curs = pvs.pvs_cursor_open_group(index, Q[:8])
    try:
        for i, cur in enumerate(curs):
            lo = np.empty(first.size, np.float32)
            hi = np.empty(first.size, np.float32)
            for k, r in enumerate(first.tolist()):
                l, h = pvs.pvs_cursor_bounds(cur, int(r), 1)
                lo[k], hi[k] = l[0], h[0]
            ref_lo, ref_hi = po.intervals(po.encode_query(Qh[i]), Qs, DIM)
            assert np.array_equal(lo.view(np.uint32), ref_lo.view(np.uint32))
            assert np.array_equal(hi.view(np.uint32), ref_hi.view(np.uint32))
    finally:
        for cur in curs:
            pvs.pvs_cursor_close(cur)


def test_passage_scale_lone_cursor(passage):
    dev, centres, rows, index = passage
    q = synth.mixture_queries(1, centres, 0.5, seed=3)[0].contiguous()
    side = torch.cuda.Stream()
    ids_t = torch.empty(1000, dtype=torch.int64, device=dev)
    sc_t = torch.empty(1000, dtype=torch.float32, device=dev)
    cur = pvs.pvs_cursor_open(index, q)
    pvs.pvs_cursor_set_stream(cur, side)
    try:
        for p in range(50):
            n_out, _ = pvs.pvs_next_device(cur, 20, ids_t[20 * p:], sc_t[20 * p:])
            assert n_out == 20
        assert pvs.pvs_cursor_sync(cur) >= 0
        side.synchronize()
        ids = ids_t.cpu().numpy()
        sc = sc_t.cpu().numpy()
        rng = np.random.default_rng(5)
        sample = np.unique(np.concatenate([rng.integers(0, N_PASSAGE, 100_000), ids]))
        lo, hi = [], []
        for i in sample[:4096]:      # bounds of a sample (ids sorted; contiguous reads)
            l, h = pvs.pvs_cursor_bounds(cur, int(i), 1)
            lo.append(l[0])
            hi.append(h[0])
    finally:
        pvs.pvs_cursor_close(cur)
    qh = q.cpu().numpy()
    # 1-3. exact scores, order, completeness on a sample
    s_sample = _check_prefix(rows, dev, qh, ids, sc, sample)
    emitted = set(ids.tolist())
    # 4. intervals of sampled rows: the oracle's (or, for a row already
    # refined, lo == hi == its exact score; -inf once delivered), and sound
    qe = po.encode_query(qh)
    first = sample[:4096]
    Qs = po.quantize(rows[torch.from_numpy(first).to(dev)].cpu().numpy())
    ref_lo, ref_hi = po.intervals(qe, Qs, DIM)
    lo = np.array(lo, np.float32)
    hi = np.array(hi, np.float32)
    s_first = s_sample[np.searchsorted(sample, first)]
    last_s, last_id = float(sc[-1]), int(ids[-1])
    for k, i in enumerate(first.tolist()):
        if i in emitted:
            assert lo[k] == -np.inf and hi[k] == -np.inf
        elif lo[k] == -np.inf:
            # computed ahead of the caller: it ranks right after the prefix
            s = float(s_first[k])
            assert hi[k] == -np.inf and (s < last_s or (s == last_s and i > last_id))
        elif lo[k] == hi[k]:
            assert lo[k].view(np.uint32) == s_first[k].view(np.uint32)
        else:
            assert lo[k].view(np.uint32) == ref_lo[k].view(np.uint32)
            assert hi[k].view(np.uint32) == ref_hi[k].view(np.uint32)
    assert np.all(ref_lo <= s_first) and np.all(s_first <= ref_hi)


@pytest.mark.parametrize("tau", [0.0, -0.5])
def test_eahr_with_deep_pulls_matches_complete_list_fusion(tau):
    m = 256
    n = 200_003
    centres = synth.mixture_centres(256, m, seed=70, device="cpu")
    V = synth.mixture_rows(n, centres, 0.35, seed=71).numpy()
    q = synth.mixture_queries(1, centres, 0.5, seed=72).numpy()[0]
    index = pvs.pvs_build(V)
    try:
        dense_ids, dense_sc = po.dense_ranking(q, V)
        proxy = torch.from_numpy(dense_sc[np.argsort(dense_ids)].astype(np.float64))
        sparse = synth.copula_ranking(proxy, tau, seed=73).numpy()
        cur = pvs.pvs_cursor_open(index, q)
        try:
            ids, F, st = pvs.eahr_topk(cur, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR)
        finally:
            pvs.pvs_cursor_close(cur)
        assert st["depth"][0] > 100_000        # the deep-pull path was exercised
        T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
        assert ids.tolist() == [x for x, _ in T]
        for (x, f), got in zip(T, F):
            if not np.isnan(got):
                assert got == ro.as_float(f)
    finally:
        pvs.pvs_index_free(index)


def _oracle_check_ranks(q, V, ids, sc, visible=None):
    """The oracle's complete ranking (Sec. 2.1) agrees with the delivered
    prefix id by id and in the bits of every authoritative score."""
    ref_ids, ref_sc = po.dense_ranking(q, V, visible)
    k = ids.size
    assert np.array_equal(ids, ref_ids[:k])
    assert np.array_equal(sc.view(np.uint32), ref_sc[:k].view(np.uint32))


def test_batched_configuration_at_full_size():
    """1,000,000 x 768 (1,024 mixture components), one batch of 256 queries
    opened together (tensor-core filter pass, horizon 200), then 4 batched
    pulls of 50 ranks into device buffers on the batch's stream: the
    benchmark's launch configuration.  Sampled queries are checked against
    the oracle's complete ranking."""
    dev = torch.device("cuda")
    n = 1_000_000
    centres = synth.mixture_centres(1024, DIM, seed=4, device=dev)
    rows = torch.empty((n, DIM), dtype=torch.float32, device=dev)
    for r in range(0, n, 1 << 20):
        c = min(1 << 20, n - r)
        rows[r:r + c] = synth.mixture_rows(c, centres, 0.35, seed=4, first=r)
    index = pvs.pvs_build(rows)
    Q = synth.mixture_queries(256, centres, 0.5, seed=5).contiguous()
    st = torch.cuda.Stream()
    ids_t = torch.empty((256, 50), dtype=torch.int64, device=dev)
    sc_t = torch.empty((256, 50), dtype=torch.float32, device=dev)
    got_ids, got_sc = [], []
    try:
        curs = pvs.pvs_cursor_open_batch(index, Q, horizon=200, stream=st)
        try:
            for _ in range(4):
                n_out = pvs.pvs_next_batch(curs, 50, ids_t, sc_t)
                assert all(n_out == 50)
                st.synchronize()
                got_ids.append(ids_t.cpu().numpy().copy())
                got_sc.append(sc_t.cpu().numpy().copy())
            assert all(s >= 0 for s in pvs.pvs_cursor_sync_batch(curs))
        finally:
            pvs.pvs_cursor_close_batch(curs)
        V = rows.cpu().numpy()
        Qh = Q.cpu().numpy()
        for i in (0, 97, 255):
            _oracle_check_ranks(Qh[i], V, np.concatenate([g[i] for g in got_ids]),
                                np.concatenate([g[i] for g in got_sc]))
    finally:
        pvs.pvs_index_free(index)


def test_snapshot_configuration_at_full_size():
    """2,000,000 x 1,024 with 20 % near-duplicates (copies + N(0, 1e-4^2),
    normalised); snapshot 1, then 200,000 appended rows and 2 % of the live
    rows tombstoned, snapshot 2 (Sec. 2.4).  Per snapshot, sampled queries:
    the first 1,000 dense ranks equal the oracle's over the snapshot's
    visible rows, and EAHR Top-20 against a tau = 0.2 copula ranking of the
    visible ids equals complete-list fusion (Sec. 2.1, 2.2)."""
    dev = torch.device("cuda")
    n0, d, add = 2_000_000, 1024, 200_000
    centres = synth.mixture_centres(4096, d, seed=5, device=dev)
    rows = torch.empty((n0 + add, d), dtype=torch.float32, device=dev)
    n_mix = n0 - n0 // 5
    rows[:n_mix] = synth.mixture_rows(n_mix, centres, 0.35, seed=5)
    g = torch.Generator(device=dev)
    g.manual_seed(55)
    src = torch.randint(0, n_mix, (n0 - n_mix,), generator=g, device=dev)
    rows[n_mix:n0] = synth.near_duplicate_rows(rows[src], 1e-4, seed=56)
    rows[n0:] = synth.mixture_rows(add, centres, 0.35, seed=61)
    index = pvs.pvs_build(rows[:n0])
    Q = synth.mixture_queries(4, centres, 0.5, seed=58)
    snaps = []
    try:
        snaps.append(pvs.pvs_snapshot_create(index))
        pvs.pvs_append(index, rows[n0:])
        rng = np.random.default_rng(57)
        dead = rng.choice(n0 + add, int(0.02 * (n0 + add)), replace=False)
        pvs.pvs_tombstone(index, dead)
        snaps.append(pvs.pvs_snapshot_create(index))
        vis = [np.zeros(n0 + add, bool), np.ones(n0 + add, bool)]
        vis[0][:n0] = True
        vis[1][dead] = False
        V = rows.cpu().numpy()
        for s, snap in enumerate(snaps):
            vis_ids = torch.from_numpy(np.nonzero(vis[s])[0]).to(dev)
            for j in (2 * s, 2 * s + 1):
                q = Q[j].contiguous()
                cur = pvs.pvs_cursor_open(index, q, snap)
                ids, sc, _ = pvs.pvs_next(cur, 1000)
                pvs.pvs_cursor_close(cur)
                qh = q.cpu().numpy()
                ref_ids, ref_sc = po.dense_ranking(qh, V, vis[s])
                assert np.array_equal(ids, ref_ids[:1000])
                assert np.array_equal(sc.view(np.uint32), ref_sc[:1000].view(np.uint32))
                proxy = rows[vis_ids] @ q
                sparse = vis_ids[synth.copula_ranking(proxy, 0.2, 900 + j)].cpu().numpy()
                cur = pvs.pvs_cursor_open(index, q, snap)
                got, F, _ = pvs.eahr_topk(cur, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR)
                pvs.pvs_cursor_close(cur)
                T = ro.target_topk_large([ref_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
                assert got.tolist() == [x for x, _ in T]
                for (x, f), v in zip(T, F):
                    if not np.isnan(v):
                        assert v == ro.as_float(f)
    finally:
        for snap in snaps:
            pvs.pvs_snapshot_free(snap)
        pvs.pvs_index_free(index)


@pytest.mark.parametrize("tau", [0.5, 0.0, -0.5])
def test_eahr_adaptive_policy_equals_complete_list_fusion(tau):
    """EAHR_POLICY_ADAPTIVE (Sec. 2.2, last paragraph): geometric reading,
    then an exact finish on the device; the ordered Top-K and its F equal
    the oracle's complete-list fusion."""
    m, n = 256, 200_003
    centres = synth.mixture_centres(256, m, seed=74, device="cpu")
    V = synth.mixture_rows(n, centres, 0.35, seed=75).numpy()
    q = synth.mixture_queries(1, centres, 0.5, seed=76).numpy()[0]
    dense_ids, dense_sc = po.dense_ranking(q, V)
    proxy = torch.from_numpy(dense_sc[np.argsort(dense_ids)].astype(np.float64))
    sparse = synth.copula_ranking(proxy, tau, seed=77).numpy()
    T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
    index = pvs.pvs_build(V)
    try:
        for policy in (pvs.EAHR_POLICY_ADAPTIVE, pvs.EAHR_POLICY_GEOMETRIC):
            cur = pvs.pvs_cursor_open(index, q)
            try:
                ids, F, st = pvs.eahr_topk(cur, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR,
                                           policy=policy)
            finally:
                pvs.pvs_cursor_close(cur)
            assert ids.tolist() == [x for x, _ in T]
            for (x, f), got in zip(T, F):
                if not np.isnan(got):
                    assert got == ro.as_float(f)
            if policy == pvs.EAHR_POLICY_ADAPTIVE:
                # the exact rank queries finish whenever reading cannot
                assert st["complete"] in ((2, 3) if tau <= 0 else (0, 2, 3))
        # a finish that needs sparse ranks reads the whole sparse list
        if tau <= 0:
            bad = sparse.copy()
            bad[-1] = bad[0]                      # a repeated id, far down the list
            cur = pvs.pvs_cursor_open(index, q)
            try:
                with pytest.raises(pvs.PvsError) as e:
                    pvs.eahr_topk(cur, bad, K=20, k=60, form=pvs.EAHR_NUMERATOR,
                                  policy=pvs.EAHR_POLICY_ADAPTIVE)
                assert e.value.status == pvs.PVS_ERR_INVALID
            finally:
                pvs.pvs_cursor_close(cur)
    finally:
        pvs.pvs_index_free(index)


def test_eahr_at_passage_scale_equals_complete_list_fusion(passage):
    """The EAHR configuration at full size (8,841,823 x 768, K = 20,
    w / (60 + r)): one query per Kendall-tau level, a Gaussian-copula sparse
    ranking of every id, both scheduling policies, against complete-list
    fusion of the oracle's complete dense ranking (scored in row chunks)."""
    dev, centres, rows, index = passage
    Q = synth.mixture_queries(3, centres, 0.5, seed=1003)
    Qh = Q.cpu().numpy()
    scores = [[] for _ in range(3)]
    for r in range(0, N_PASSAGE, 1 << 20):
        Vh = rows[r:r + (1 << 20)].cpu().numpy()
        for i in range(3):
            scores[i].append(po.exact_scores(Qh[i], Vh))
    ids_all = np.arange(N_PASSAGE, dtype=np.int64)
    for i, tau in enumerate((0.5, 0.0, -0.5)):
        s = np.concatenate(scores[i])
        dense_ids = np.lexsort((ids_all, -s.astype(np.float64))).astype(np.int64)
        sparse = synth.copula_ranking(torch.from_numpy(s.astype(np.float64)), tau,
                                      seed=2003 + i).numpy()
        T = ro.target_topk_large([dense_ids, sparse], [1, 1], 60, 20, ro.NUMERATOR)
        for policy in (pvs.EAHR_POLICY_ADAPTIVE, pvs.EAHR_POLICY_GEOMETRIC):
            cur = pvs.pvs_cursor_open(index, Q[i].contiguous())
            try:
                ids, F, st = pvs.eahr_topk(cur, sparse, K=20, k=60, form=pvs.EAHR_NUMERATOR,
                                           policy=policy)
            finally:
                pvs.pvs_cursor_close(cur)
            assert ids.tolist() == [x for x, _ in T], (tau, policy)
            for (x, f), got in zip(T, F):
                if not np.isnan(got):
                    assert got == ro.as_float(f)
