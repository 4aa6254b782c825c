"""Benchmark: PVS resumable exact dense ranking on one GB300 (per rank).

Workload (the passage-scale single-query configuration): a corpus of
N = 8,841,823 vectors of d = 768 drawn from a 4,096-component Gaussian
mixture (standard-normal centres, within-component std 0.35, L2-normalised);
queries are perturbed mixture centres (noise std 0.5, normalised).  One step
= a batch of queries; per query a cursor delivers the first 1,000 exact ranks
in chunks of 20 (open, 50 pulls, close).  The corpus codes (6.9 GB per
interval pass) are far larger than the 129 MB L2, so no L2 flush is needed.

Both legs run through the library's native request executor
(pvs_executor_run_ex): WORKERS native threads, each serving GROUP queries
at a time from one grouped interval pass over the codes
(pvs_cursor_open_group) and pulling every 20-rank page of the group's
cursors in one batched launch; every query still gets its own pages.
`value` (exact dense ranks/s) has the queries resident in HBM and the ranks
written to device buffers, timed with CUDA events; `e2e` is the same
through host buffers (pinned queries in, every page on the host before the
next is requested), the copies inside the timed region.
`roofline` reports the grouped interval pass (the dominant kernel):
algorithmic bytes N * (m_pad + 12) read plus 8 * N * GROUP bytes of bounds
written per pass, over its CUDA-event duration (the library's events on the
pass's stream), against the measured HBM copy bandwidth.

`--impl reference` times the oracle (a plain CPU implementation, run as it
stands) on a bounded sample of the same workload.  Under torchrun every rank
ranks its own queries against its own copy of the index (no collective).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

N_CORPUS = 8_841_823
DIM = 768
COMPONENTS = 4096
WITHIN_STD = 0.35
QUERY_NOISE = 0.5
RANKS_PER_QUERY = 1000
CHUNK = 20
METRIC = "exact dense ranks/sec"
UNIT = "ranks/s"
WORKLOAD = ("passage-scale single-query ranking: N=8,841,823 x d=768 Gaussian mixture "
            "(4,096 components, within std 0.35, L2-normalised), first 1,000 exact ranks "
            "per query in chunks of 20")


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=60)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="pvs", choices=["pvs", "reference"])
    p.add_argument("--queries", type=int, default=64, help="queries per step")
    p.add_argument("--group", type=int, default=8,
                   help="passage: queries per grouped pass over the codes (1: one pass each)")
    p.add_argument("--n", type=int, default=N_CORPUS, help="corpus rows (default: full)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--workload", default="passage",
                   choices=["passage", "batched", "eahr", "snapshots", "sparse", "hybrid",
                            "ablation", "segments"],
                   help="passage: single-query ranking (default); batched: 256-query "
                        "tensor-core batches; eahr: EAHR Top-20 fusion over the passage "
                        "corpus and copula sparse rankings; snapshots: near-duplicate "
                        "corpus, five snapshots, EAHR Top-20; sparse: PBM sparse ranks "
                        "over a synthetic BM25 corpus; hybrid: EAHR Top-20 over PVS and PBM "
                        "on the same items; ablation: PVS vs scalar-quantization intervals "
                        "vs full scan; segments: EAHR over 8 merged Segments")
    p.add_argument("--eahr-queries", type=int, default=200,
                   help="queries per correlation level (tau = +0.5, 0)")
    p.add_argument("--eahr-exhaust-queries", type=int, default=200,
                   help="queries at tau = -0.5 (both lists are read to the end)")
    p.add_argument("--snap-queries", type=int, default=100, help="queries per snapshot")
    p.add_argument("--eahr-levels", default="0.5,0,-0.5",
                   help="Kendall tau levels of --workload eahr (comma-separated)")
    p.add_argument("--eahr-policy", default="adaptive",
                   choices=["adaptive", "geometric", "frozen", "equal"],
                   help="EAHR scheduling policy (adaptive: geometric reading, then an exact finish "
                        "on the device: ranks of the remaining candidates, else complete-list "
                        "fusion)")
    p.add_argument("--no-eahr", action="store_true",
                   help="passage: leave out the EAHR Top-20 record of the default line")
    p.add_argument("--ablation-queries", type=int, default=30,
                   help="queries per generator in --workload ablation")
    p.add_argument("--pipeline", type=int, default=0,
                   help="executor workers (passage), batches in flight (batched) or serving "
                        "threads (sparse); 0: the default")
    p.add_argument("--oracle-check", action="store_true",
                   help="snapshots: compare the first query's first 1,000 dense ranks of every "
                        "snapshot with the oracle and count near-tie swaps")
    return p.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def query_seed(base: int, rank: int) -> int:
    """Every rank draws its own queries (weak scaling: the work is sharded by
    query, each rank against its own replica of the index)."""
    return base + 7919 * rank


def slowest(pg, seconds: float, device) -> float:
    """The job's time: the maximum over ranks (no-op without a process group)."""
    if pg is None:
        return seconds
    import torch
    t = torch.tensor([seconds], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank: float, world: int, seconds: float) -> float:
    """Whole-job throughput: every rank's units over the slowest rank's time."""
    return units_per_rank * world / seconds


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def interval_traffic(n_rows: int, record="interval_pass_kernel_passage_8.8Mx768_traffic.json"):
    """DRAM bytes per pass from a committed ncu capture, scaled by rows; None
    when the kernel source changed since the capture."""
    import hashlib
    path = os.path.join(ROOT, "profiles", record)
    try:
        with open(path) as f:
            d = json.load(f)
        with open(os.path.join(ROOT, d["source"]), "rb") as f:
            if hashlib.sha256(f.read()).hexdigest() != d["source_sha256"]:
                return None
        per_row = (d["captured_dram_bytes_read"] + d["captured_dram_bytes_write"]) / d["captured_rows"]
        return per_row * n_rows
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region.

    The sampler is started, and its first sample awaited, before the region
    begins; a reader thread stamps every sample on arrival, and the summary
    keeps the samples that arrived between the region's start and one
    sampling period after its end."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    PERIOD_MS = 100

    def __init__(self, gpu: int):
        self.gpu = gpu
        self.proc = None
        self.rows = []
        self.t0 = self.t1 = 0.0

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append((time.monotonic(), line))

    def __enter__(self):
        import threading
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", str(self.PERIOD_MS)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.reader = threading.Thread(target=self._read, daemon=True)
            self.reader.start()
            deadline = time.monotonic() + 5.0
            while not self.rows and time.monotonic() < deadline and self.proc.poll() is None:
                time.sleep(0.01)
        except Exception:
            self.proc = None
        self.t0 = time.monotonic()
        return self

    def __exit__(self, *exc):
        self.t1 = time.monotonic()
        if self.proc is not None:
            time.sleep(self.PERIOD_MS / 1e3)   # the sample taken at the end
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.reader.join(timeout=5)
        return False

    def summary(self):
        late = self.t1 + self.PERIOD_MS / 1e3
        rows = [r.split(",") for t, r in self.rows if self.t0 <= t <= late and r.strip()]
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax.append(float(r[2]))
            except ValueError:
                continue
            for name, val in zip(names, r[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "reasons": sorted(reasons), "samples": len(sm)}


def build_corpus_index(pvs, synth, torch, n, stream, device, components=COMPONENTS, seed=2):
    """Generate the mixture corpus chunk by chunk straight into the index."""
    centres = synth.mixture_centres(components, DIM, seed=seed, device=device)
    index = None
    chunk = 1 << 20
    t0 = time.perf_counter()
    for r in range(0, n, chunk):
        c = min(chunk, n - r)
        rows = synth.mixture_rows(c, centres, WITHIN_STD, seed=seed, first=r)
        if index is None:
            index = pvs.pvs_build(rows, stream=stream)
        else:
            pvs.pvs_append(index, rows)
        del rows
    torch.cuda.synchronize()
    return index, centres, time.perf_counter() - t0


PIPELINE = 8   # passage: executor worker threads, each with a group of queries in flight
SPARSE_WORKERS = 16   # sparse: host threads serving PBM queries, a stream each


def _finish(pvs, cur, stats_acc):
    st = pvs.pvs_cursor_sync(cur)
    s = pvs.pvs_cursor_stats(cur)
    pvs.pvs_cursor_close(cur)
    if st < 0:
        raise RuntimeError(f"cursor failed: {st}")
    if stats_acc is not None:
        stats_acc.append(s)


def single_pass_record(stats, n, m_pad, peak):
    """The lone queries' interval pass (interval_pass_kernel, one query per
    read of the codes), timed by the library's CUDA events on each cursor's
    stream: N (m_pad + 12) B read + 8 N B written per pass."""
    ms = [s["interval_ms"] for s in stats if s.get("interval_ms", 0) > 0]
    if not ms:
        return None
    med = float(statistics.median(ms))
    gbps = (n * (m_pad + 12) + 8 * n) / (med / 1e3) / 1e9
    return {"kernel": "interval_pass_kernel", "ms_p50": med, "GBps": gbps, "frac": gbps / peak,
            "passes": len(ms)}


def measure_latency(pvs, torch, index, queries, out_ids, out_scores, stream, count,
                    stats=None):
    """Latency to the first 20 and first 1,000 ranks, one query at a time
    (each cursor's statistics appended to `stats` when given)."""
    lat20, lat1000 = [], []
    for qi in range(count):
        t_open = torch.cuda.Event(enable_timing=True)
        t_20 = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_open.record(stream)
        cur = pvs.pvs_cursor_open(index, queries[qi])
        for p in range(RANKS_PER_QUERY // CHUNK):
            off = p * CHUNK
            pvs.pvs_next_device(cur, CHUNK, out_ids[0, off:], out_scores[0, off:])
            if p == 0:
                t_20.record(stream)
        t_end.record(stream)
        _finish(pvs, cur, stats)
        stream.synchronize()
        lat20.append(t_open.elapsed_time(t_20))
        lat1000.append(t_open.elapsed_time(t_end))
    return lat20, lat1000


def cpu_baseline(synth, torch, centres_dev, queries_host, n_full, seconds_budget=20.0):
    """The oracle (as it stands) on a bounded sample: the first `rows` corpus
    rows, for as many queries as fit the budget; ranks/s scaled to the full N
    (the oracle's cost is linear in the rows it scores)."""
    import numpy as np
    from oracle import pvs_oracle as po
    rows = 1 << 20
    V = synth.mixture_rows(rows, centres_dev, WITHIN_STD, seed=2, first=0).cpu().numpy()
    t0 = time.perf_counter()
    c0 = time.process_time()
    done = 0
    while done < len(queries_host):
        ids, sc = po.dense_ranking(queries_host[done], V)
        _ = ids[:RANKS_PER_QUERY]
        done += 1
        if time.perf_counter() - t0 > seconds_budget:
            break
    dt = time.perf_counter() - t0
    cores = (time.process_time() - c0) / dt   # the cores it kept busy on average
    per_query_full = dt / done * (n_full / rows)
    return {"value": RANKS_PER_QUERY / per_query_full, "unit": UNIT,
            "cores": round(cores, 1), "host_cores": os.cpu_count(), "kind": "oracle",
            "projected": True,
            "sample": f"{done} queries x first {RANKS_PER_QUERY} exact ranks over the first "
                      f"{rows:,} corpus rows (oracle: binary64 scoring by numpy's BLAS, "
                      f"exact fallback in Python, full sort; cores = process CPU time / wall "
                      f"time); projected to N by scaling the time by N/{rows:,}"}


def reference_arm(args):
    rank, world, local = dist_env()
    if rank != 0:
        return
    import numpy as np
    import torch
    import synth
    from oracle import pvs_oracle as po
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    centres = synth.mixture_centres(COMPONENTS, DIM, seed=2, device=dev)
    rows = 1 << 19
    V = synth.mixture_rows(rows, centres, WITHIN_STD, seed=2, first=0).cpu().numpy()
    Q = synth.mixture_queries(args.warmup + args.steps, centres, QUERY_NOISE, seed=3).cpu().numpy()
    for w in range(args.warmup):
        po.dense_ranking(Q[w], V)
    t0 = time.perf_counter()
    c0 = time.process_time()
    for s in range(args.steps):
        po.dense_ranking(Q[args.warmup + s], V)
    wall = time.perf_counter() - t0
    cores = (time.process_time() - c0) / wall   # the cores it kept busy on average
    dt = wall / args.steps * (args.n / rows)
    value = RANKS_PER_QUERY / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "N": args.n, "d": DIM,
                       "step": "1 query, first 1,000 ranks"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": round(cores, 1),
                             "host_cores": os.cpu_count(), "kind": "oracle", "projected": True,
                             "sample": f"1 query per step over the first {rows:,} rows; "
                                       f"projected to N by scaling the time by N/{rows:,}"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


BATCH_N = 1_000_000
BATCH_COMPONENTS = 1024
BATCH_Q = 256
BATCH_RANKS = 200
BATCH_CHUNK = 50
BATCH_PIPELINE = 4   # batches in flight, each driven by its own host thread and stream
BATCH_WORKLOAD = ("batched queries: N=1,000,000 x d=768 Gaussian mixture (1,024 components, "
                  "within std 0.35), 256 concurrent queries per batch, first 200 exact ranks "
                  "per query in chunks of 50")


def bf16_peak():
    """The filter pass is timed inside a long run of batches: the sustained
    (power-capped) bf16 figure is its denominator."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["bf16_tflops_sustained"]), "measured sustained"
    except Exception:
        return 1700.0, "fallback sustained"


def _run_threads(worker, nthreads):
    import threading
    errors = []

    def guarded(k):
        try:
            worker(k)
        except Exception as e:  # surfaced below
            errors.append(e)

    threads = [threading.Thread(target=guarded, args=(k,)) for k in range(nthreads)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    if errors:
        raise errors[0]


def main_batched(args, pvs, synth, torch, np, rank, world, local, dev, pg):
    """Batched workload: one step = one batch of 256 queries opened together
    (one tensor-core interval pass), then 4 batched pulls of 50 ranks.
    BATCH_PIPELINE host threads drive alternate batches on their own streams,
    so one batch's pulls overlap the next batch's open."""
    stream = torch.cuda.Stream(device=dev)
    n = BATCH_N if args.n == N_CORPUS else args.n
    index, centres, build_s = build_corpus_index(pvs, synth, torch, n, stream.cuda_stream, dev,
                                                 components=BATCH_COMPONENTS, seed=4)
    # every host thread warms up on its own batches (the cursor pool and the
    # scratch pool grow to what four batches in flight hold)
    warm = max(args.warmup, 2 * BATCH_PIPELINE)
    nb = warm + args.steps
    queries = synth.mixture_queries(nb * BATCH_Q, centres, QUERY_NOISE, seed=query_seed(5, rank))
    queries = queries.reshape(nb, BATCH_Q, DIM).contiguous()
    streams = [torch.cuda.Stream(device=dev) for _ in range(BATCH_PIPELINE)]
    ids_t = torch.empty((BATCH_PIPELINE, BATCH_Q, BATCH_CHUNK), dtype=torch.int64, device=dev)
    sc_t = torch.empty((BATCH_PIPELINE, BATCH_Q, BATCH_CHUNK), dtype=torch.float32, device=dev)
    torch.cuda.synchronize()

    def step(qb, slot, pass_ms, stats=None):
        curs = pvs.pvs_cursor_open_batch(index, qb, horizon=BATCH_RANKS, stream=streams[slot])
        for _ in range(BATCH_RANKS // BATCH_CHUNK):
            pvs.pvs_next_batch(curs, BATCH_CHUNK, ids_t[slot], sc_t[slot])
        if stats is None:
            states = pvs.pvs_cursor_sync_batch(curs)   # one wait for every cursor's status
        else:
            st = pvs.pvs_cursor_stats_batch(curs)
            stats.extend(st)
            states = [x["state"] for x in st]
        if any(x < 0 for x in states):
            raise RuntimeError("cursor failed")
        if pass_ms is not None:   # device time of this batch's filter pass (CUDA events)
            pass_ms.append(pvs.pvs_cursor_stats(curs[0])["batch_ms"])
        pvs.pvs_cursor_close_batch(curs)

    def run(batches, pass_ms):
        def worker(k):
            torch.cuda.set_device(dev)
            for b in batches[k::BATCH_PIPELINE]:
                step(queries[b], k, pass_ms)
        _run_threads(worker, BATCH_PIPELINE)

    run(list(range(warm)), None)
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    pass_ms = []
    launches0 = pvs.pvs_launch_count()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        start.record(stream)
        for s_ in streams:
            s_.wait_event(start)
        run(list(range(warm, nb)), pass_ms)
        for s_ in streams:                      # join every stream's work
            done = torch.cuda.Event()
            done.record(s_)
            stream.wait_event(done)
        end.record(stream)
        stream.synchronize()
    launches = pvs.pvs_launch_count() - launches0
    stats = []   # per-query counters from one more (untimed) batch of the same queries
    step(queries[warm], 0, None, stats)
    elapsed = start.elapsed_time(end) / 1e3
    elapsed = slowest(pg, elapsed, dev)
    ranks_total = args.steps * BATCH_Q * BATCH_RANKS * world
    value = job_rate(args.steps * BATCH_Q * BATCH_RANKS, world, elapsed)

    # e2e: host queries, host outputs, the same threads and streams
    qh = [np.ascontiguousarray(queries[b].cpu().numpy()) for b in range(nb)]
    torch.cuda.synchronize()

    def e2e_worker(k):
        torch.cuda.set_device(dev)
        for b in range(warm + k, nb, BATCH_PIPELINE):
            curs = pvs.pvs_cursor_open_batch(index, qh[b], horizon=BATCH_RANKS,
                                             stream=streams[k])
            for _ in range(BATCH_RANKS // BATCH_CHUNK):
                pvs.pvs_next_batch(curs, BATCH_CHUNK)
            pvs.pvs_cursor_close_batch(curs)

    t0 = time.perf_counter()
    _run_threads(e2e_worker, BATCH_PIPELINE)
    e2e_elapsed = time.perf_counter() - t0
    e2e_value = ranks_total / e2e_elapsed

    batch_ms = statistics.mean(pass_ms)   # one filter pass per batch
    flops = 2.0 * BATCH_Q * n * DIM
    achieved = flops / (batch_ms / 1e3) / 1e12
    peak, peak_kind = bf16_peak()
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": warm, "ms_per_step": elapsed / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": BATCH_WORKLOAD, "N": n, "d": DIM, "queries_per_batch": BATCH_Q,
                   "ranks_per_query": BATCH_RANKS, "chunk": BATCH_CHUNK,
                   "batches_in_flight": BATCH_PIPELINE,
                   "l2": "no flush: each batch pass streams 1.5 GB of bf16 codes (> 129 MB L2)",
                   "parallelism": f"replicas x{world}"},
        "e2e": {"value": e2e_value, "unit": UNIT,
                "h2d_bytes_per_step": BATCH_Q * DIM * 4,
                "d2h_bytes_per_step": BATCH_Q * BATCH_RANKS * (8 + 4)},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak,
                     "traffic": interval_traffic(n, "batch_interval_kernel_traffic.json"),
                     "peak_kind": peak_kind, "kernel": "batch_interval_kernel (filter pass)"},
        "gpu_launches": launches,
        "batch_pass_ms": batch_ms,
        "per_query": {"refined_mean": statistics.mean(s["refined"] for s in stats),
                      "single_query_passes": sum(s["interval_passes"] for s in stats)},
        "build_s": build_s,
        "clocks": clk.summary(),
    }
    pvs.pvs_index_free(index)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


EAHR_K = 20
EAHR_RRF_K = 60   # the build target's w / (60 + rank), w_d = w_s = 1
EAHR_LEVELS = (0.5, 0.0, -0.5)


def eahr_levels(pvs, synth, torch, np, index, rows, queries, policy, counts, rank, dev,
                warmup=2, comparator_queries=None):
    """EAHR Top-20 per Kendall-tau level: per query a Gaussian-copula sparse
    ranking of every id (an fp32 torch product of the corpus with the query is
    the copula's proxy: input generation only), then, timed on the host,
    cursor open + eahr_topk (dense pulls through the library, sparse ids from
    host memory) + close.  Beside it, the exhaustive comparator: fp32 scores
    of every row, a full sort and complete-list fusion in plain torch (for the
    first `comparator_queries` queries of a level; all when None).
    counts: {tau: queries}.  Returns (levels, latencies)."""
    n = rows.shape[0]

    def sparse_for(q, tau, seed):
        proxy = rows @ q
        return synth.copula_ranking(proxy, tau, seed).cpu().numpy(), proxy

    def comparator(q, sparse_dev):
        """Exhaustive fp32 scoring + full sort + complete-list fusion, ms."""
        torch.cuda.synchronize()
        t = time.perf_counter()
        sc = rows @ q
        order = torch.argsort(sc, descending=True, stable=True)
        rd = torch.empty(n, dtype=torch.float64, device=dev)
        rd[order] = torch.arange(1, n + 1, dtype=torch.float64, device=dev)
        rs = torch.empty(n, dtype=torch.float64, device=dev)
        rs[sparse_dev] = torch.arange(1, n + 1, dtype=torch.float64, device=dev)
        fused = 1.0 / (EAHR_RRF_K + rd) + 1.0 / (EAHR_RRF_K + rs)
        top = torch.topk(fused, EAHR_K).indices
        top.cpu()
        return (time.perf_counter() - t) * 1e3

    qi = 0
    for w in range(warmup):   # library paths, torch kernels
        sp, _ = sparse_for(queries[qi], 0.5, 7 + w)
        cur = pvs.pvs_cursor_open(index, queries[qi])
        pvs.eahr_topk(cur, sp, K=EAHR_K, k=EAHR_RRF_K, form=pvs.EAHR_NUMERATOR, policy=policy)
        pvs.pvs_cursor_close(cur)
        comparator(queries[qi], torch.from_numpy(sp).to(dev))
        qi += 1
    levels, lat_all = {}, []
    for tau, count in counts.items():
        lat, cmp_ms, dd, ds, ex, pulls = [], [], [], [], 0, []
        finish = {0: 0, 1: 0, 2: 0, 3: 0}
        ktau = None
        for j in range(count):
            q = queries[qi]
            qi += 1
            sp, proxy = sparse_for(q, tau, query_seed(1000, rank) + qi)
            if j == 0:   # realised Kendall tau of the generated channel
                dense_order = torch.argsort(proxy, descending=True, stable=True).cpu().numpy()
                ktau = synth.kendall_tau_sample(dense_order, sp, 200_000, seed=qi)
            torch.cuda.synchronize()
            t = time.perf_counter()
            cur = pvs.pvs_cursor_open(index, q)
            ids, F, st = pvs.eahr_topk(cur, sp, K=EAHR_K, k=EAHR_RRF_K,
                                       form=pvs.EAHR_NUMERATOR, policy=policy)
            pvs.pvs_cursor_close(cur)
            lat.append((time.perf_counter() - t) * 1e3)
            if len(ids) != EAHR_K:
                raise RuntimeError("EAHR returned a short list")
            dd.append(st["depth"][0])
            ds.append(st["depth"][1])
            ex += int(st["exhausted"][0] and st["exhausted"][1])
            finish[int(st.get("complete", 0))] += 1
            pulls.append(st["pulls"][0])
            if comparator_queries is None or j < comparator_queries:
                cmp_ms.append(comparator(q, torch.from_numpy(sp).to(dev)))
        lat_all.extend(lat)
        levels[f"{tau:+.1f}"] = {
            "queries": count, "kendall_tau_realised": ktau,
            "latency_ms_p50": float(np.median(lat)), "latency_ms_p95": float(np.percentile(lat, 95)),
            "exhaustive_fp32_ms_p50": float(np.median(cmp_ms)) if cmp_ms else None,
            "dense_depth_p50": float(np.median(dd)), "dense_depth_mean": float(np.mean(dd)),
            "sparse_depth_p50": float(np.median(ds)), "both_exhausted": ex,
            "finished_by": {"reading": finish[0], "rank_intervals": finish[2],
                            "exact_ranks": finish[3], "complete_list_fusion": finish[1]},
            "dense_pulls_p50": float(np.median(pulls))}
    return levels, lat_all


def eahr_policy(args, pvs):
    return {"geometric": pvs.EAHR_POLICY_GEOMETRIC, "frozen": pvs.EAHR_POLICY_FROZEN,
            "equal": pvs.EAHR_POLICY_EQUAL_DEPTH,
            "adaptive": pvs.EAHR_POLICY_ADAPTIVE}[args.eahr_policy]


def main_eahr(args, pvs, synth, torch, np, rank, world, local, dev, pg):
    """EAHR end to end over the passage corpus: per query a sparse channel that
    is a complete ranking of all N ids, a Gaussian-copula permutation of the
    dense order with Kendall tau ~ +0.5, 0, -0.5 (an fp32 torch product of the
    corpus with the query is the copula's proxy: input generation only).  Timed
    per query: cursor open + eahr_topk (dense pulls through pvs_next, sparse
    ids read from host memory) + close.  Beside it, the exhaustive comparator:
    fp32 scores of every row, a full sort and complete-list fusion on the GPU
    (plain torch)."""
    n = args.n
    stream = torch.cuda.Stream(device=dev)
    centres = synth.mixture_centres(COMPONENTS, DIM, seed=2, device=dev)
    t0 = time.perf_counter()
    rows = torch.empty((n, DIM), dtype=torch.float32, device=dev)
    chunk = 1 << 20
    for r in range(0, n, chunk):
        c = min(chunk, n - r)
        rows[r:r + c] = synth.mixture_rows(c, centres, WITHIN_STD, seed=2, first=r)
    index = pvs.pvs_build(rows, stream=stream.cuda_stream)
    torch.cuda.synchronize()
    build_s = time.perf_counter() - t0
    counts = {t: (args.eahr_exhaust_queries if t < 0 else args.eahr_queries)
              for t in [float(x) for x in args.eahr_levels.split(",")]}
    total_q = sum(counts.values()) + 2
    queries = synth.mixture_queries(total_q, centres, QUERY_NOISE, seed=query_seed(3, rank))
    policy = eahr_policy(args, pvs)

    if pg:
        pg.barrier()
    launches0 = pvs.pvs_launch_count()
    with ClockSampler(local) as clk:
        levels, lat_all = eahr_levels(pvs, synth, torch, np, index, rows, queries, policy, counts,
                                      rank, dev, warmup=2)
    launches = pvs.pvs_launch_count() - launches0
    head = levels.get("+0.5", next(iter(levels.values())))
    line = {
        "metric": "EAHR Top-20 latency (p50, tau=+0.5)", "value": head["latency_ms_p50"],
        "unit": "ms", "n_gpus": world, "steps": sum(v["queries"] for v in levels.values()),
        "warmup": 2, "ms_per_step": float(np.mean(lat_all)), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "int8", "data": "synthetic",
        "config": {"workload": "EAHR end-to-end fusion: passage corpus N=8,841,823 x d=768 "
                               "(or --n), sparse channel a complete copula ranking of all N ids "
                               "(Kendall tau +0.5 / 0 / -0.5), weighted RRF 1/(60+rank), K=20",
                   "N": n, "d": DIM, "K": EAHR_K, "rrf_k": EAHR_RRF_K,
                   "policy": args.eahr_policy,
                   "l2": "no flush: every query's interval pass streams 6.9 GB of codes",
                   "parallelism": f"replicas x{world}"},
        "e2e": {"value": head["latency_ms_p50"], "unit": "ms",
                "h2d_bytes_per_step": DIM * 4, "d2h_bytes_per_step": EAHR_K * (8 + 8)},
        "levels": levels,
        "gpu_launches": launches,
        "build_s": build_s,
        "clocks": clk.summary(),
    }
    pvs.pvs_index_free(index)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


SPARSE_TERMS = 500_000      # vocabulary of the synthetic BM25 corpus
SPARSE_TOKENS = 40.0        # mean tokens per item (Poisson)
SPARSE_QUERY_TERMS = 5.0    # mean distinct terms per query
SPARSE_RANKS = 1000
SPARSE_CHUNK = 20


def build_sparse_index(pvs, synth, torch, n, dev, seed):
    """Synthetic BM25 postings generated on the device and the PBM index."""
    t0 = time.perf_counter()
    off, docs, imps = synth.bm25_postings(n, SPARSE_TERMS, SPARSE_TOKENS, seed=seed, device=dev)
    torch.cuda.synchronize()
    t1 = time.perf_counter()
    index = pvs.pbm_build(off, docs, imps, n)
    torch.cuda.synchronize()
    return index, (off, docs, imps), t1 - t0, time.perf_counter() - t1


def sparse_complete(torch, n, post, terms, weights, dev):
    """The complete sparse ranking in plain torch (the comparator): every
    query term's postings scattered into a score per item, then a full stable
    sort; returns the first SPARSE_RANKS ids of the positive-score support
    (host) and the time in ms."""
    off, docs, imps = post
    torch.cuda.synchronize()
    t = time.perf_counter()
    sc = torch.zeros(n, dtype=torch.float32, device=dev)
    for term, w in zip(terms.tolist(), weights.tolist()):
        a, b = int(off[term]), int(off[term + 1])
        sc.index_put_((docs[a:b].long(),), imps[a:b] * w, accumulate=True)
    order = torch.argsort(sc, descending=True, stable=True)
    head = order[:SPARSE_RANKS]
    head = head[sc[head] > 0].cpu()
    return head, (time.perf_counter() - t) * 1e3


def main_sparse(args, pvs, synth, torch, np, rank, world, local, dev, pg):
    """PBM sparse ranking over a passage-scale synthetic BM25 corpus: per
    query, open a cursor and pull the first 1,000 exact sparse ranks in
    chunks of 20 (host outputs).  The timed queries are served by
    SPARSE_WORKERS host threads, each cursor on its thread's stream; the
    latency of a lone query is measured after, one query at a time.  Each
    rank drives its own index replica.  Beside it, the complete sparse
    ranking in plain torch (score every posting of the query terms, sort all
    N)."""
    n = args.n
    index, post, gen_s, build_s = build_sparse_index(pvs, synth, torch, n, dev, seed=8)
    off_h = post[0].cpu()
    nqs = args.warmup + args.steps
    queries = synth.sparse_queries(nqs, off_h, seed=query_seed(9, rank),
                                   mean_terms=SPARSE_QUERY_TERMS, min_df=2)

    def one(terms, weights, stream=None):
        t0 = time.perf_counter()
        cur = pvs.pbm_cursor_open(index, terms, weights, stream=stream)
        first = None
        got = []
        for c in range(SPARSE_RANKS // SPARSE_CHUNK):
            ids, _, st = pvs.pbm_next(cur, SPARSE_CHUNK)
            got.append(ids)
            if c == 0:
                first = time.perf_counter() - t0
        total = time.perf_counter() - t0
        stats = pvs.pbm_cursor_stats(cur)
        pvs.pbm_cursor_close(cur)
        return total, first, stats, np.concatenate(got)

    for w in range(args.warmup):
        one(*queries[w])
        sparse_complete(torch, n, post, queries[w][0], queries[w][1], dev)
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    launches0 = pvs.pvs_launch_count()
    workers = SPARSE_WORKERS
    streams = [torch.cuda.Stream(device=dev) for _ in range(workers)]
    st_all = []

    def serve(k):
        torch.cuda.set_device(dev)
        for j in range(args.warmup + k, nqs, workers):
            _, _, stats, _ = one(*queries[j], stream=streams[k])
            st_all.append(stats)
    for k in range(workers):   # every thread's stream and the cursor pool warm
        one(*queries[k % max(args.warmup, 1)], stream=streams[k])
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:   # sampling runs before t0 and after the region
        t0 = time.perf_counter()
        _run_threads(serve, workers)
        torch.cuda.synchronize()
        elapsed = time.perf_counter() - t0
    elapsed = slowest(pg, elapsed, dev)
    launches = pvs.pvs_launch_count() - launches0
    lat, first = [], []   # a lone query at a time
    for j in range(args.warmup, min(nqs, args.warmup + 20)):
        total, f, _, _ = one(*queries[j])
        lat.append(total)
        first.append(f)
    cmp_ms, mismatches = [], 0
    for j in range(args.warmup, min(nqs, args.warmup + 20)):
        head, ms = sparse_complete(torch, n, post, queries[j][0], queries[j][1], dev)
        cmp_ms.append(ms)
    check = None
    if args.oracle_check:
        from oracle import pbm_oracle as po
        o, d, i = (x.cpu().numpy() for x in post)
        check = {"queries": 0, "mismatches": 0}
        for j in range(args.warmup, min(nqs, args.warmup + 3)):
            _, _, _, ids = one(*queries[j])
            ref, _ = po.sparse_ranking(queries[j][0], queries[j][1], o, d, i, n)
            check["queries"] += 1
            check["mismatches"] += int(not np.array_equal(ids, ref[:SPARSE_RANKS]))
    value = job_rate(args.steps * SPARSE_RANKS, world, elapsed)
    med = lambda k: float(np.median([s[k] for s in st_all]))
    line = {
        "metric": "exact sparse ranks/sec (PBM)", "value": value, "unit": "ranks/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": elapsed * 1e3 / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "PBM sparse ranking: synthetic BM25 impact postings over "
                               f"N={n:,} items (vocabulary {SPARSE_TERMS:,}, Zipf terms, "
                               f"Poisson({SPARSE_TOKENS:g}) tokens per item, k1=0.9 b=0.4), "
                               f"queries of 1+Poisson({SPARSE_QUERY_TERMS - 1:g}) terms, "
                               f"first {SPARSE_RANKS} ranks in chunks of {SPARSE_CHUNK}",
                   "N": n, "ranks_per_query": SPARSE_RANKS, "chunk": SPARSE_CHUNK,
                   "postings": int(post[1].numel()), "block": 128,
                   "l2": "no flush: queries run back to back on one index",
                   "host_threads": workers,
                   "parallelism": f"replicas x{world}"},
        "e2e": {"value": value, "unit": "ranks/s",
                "h2d_bytes_per_step": int(np.mean([8 * len(q[0]) for q in queries])),
                "d2h_bytes_per_step": SPARSE_RANKS * 12},
        "latency_ms": {"first_20_p50": float(np.median(first)) * 1e3,
                       "first_1000_p50": float(np.median(lat)) * 1e3,
                       "first_1000_p95": float(np.percentile(lat, 95)) * 1e3,
                       "note": "a lone query at a time, after the timed region"},
        "per_query": {"ranges_expanded_p50": med("ranges_expanded"), "ranges": st_all[0]["ranges"],
                      "postings_visited_p50": med("postings_visited"),
                      "rounds_p50": med("rounds"),
                      "pulls_from_window_p50": med("pulls_from_window")},
        "complete_sparse_ranking_ms_p50": float(np.median(cmp_ms)) if cmp_ms else None,
        "oracle_check": check,
        "gpu_launches": launches,
        "generate_s": gen_s, "build_s": build_s,
        "clocks": clk.summary(),
    }
    pvs.pbm_index_free(index)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


def main_ablation(args, pvs, synth, torch, np, rank, world, local, dev, pg):
    """Rank-generator ablation (the analogue of the paper's Table 1, dense
    side) over the passage corpus: the same queries through PVS, scalar-
    quantization intervals (an index with one scale for the corpus) and
    exhaustive float32 scanning.  Per generator and query: (1) the first
    1,000 ranks in chunks of 20 into host buffers; (2) EAHR Top-20 against a
    tau = +0.5 copula sparse ranking (as --workload eahr).  Reported: paired
    geometric-mean latency ratios to PVS and float32 evaluations per query."""
    n = args.n
    stream = torch.cuda.Stream(device=dev)
    centres = synth.mixture_centres(COMPONENTS, DIM, seed=2, device=dev)
    rows = torch.empty((n, DIM), dtype=torch.float32, device=dev)
    chunk = 1 << 20
    for r in range(0, n, chunk):
        c = min(chunk, n - r)
        rows[r:r + c] = synth.mixture_rows(c, centres, WITHIN_STD, seed=2, first=r)
    t0 = time.perf_counter()
    idx_pvs = pvs.pvs_build(rows, stream=stream.cuda_stream)
    torch.cuda.synchronize()
    t1 = time.perf_counter()
    idx_sq = pvs.pvs_build(rows, stream=stream.cuda_stream, quantization=pvs.PVS_QUANT_GLOBAL)
    torch.cuda.synchronize()
    t2 = time.perf_counter()
    nq = 2 + args.ablation_queries
    queries = synth.mixture_queries(nq, centres, QUERY_NOISE, seed=query_seed(14, rank))
    gens = {"pvs": (idx_pvs, pvs.PVS_GEN_INTERVALS),
            "scalar": (idx_sq, pvs.PVS_GEN_INTERVALS),
            "scan": (idx_pvs, pvs.PVS_GEN_FULL_SCAN)}

    def ranks(name, q):
        index, gen = gens[name]
        torch.cuda.synchronize()
        t = time.perf_counter()
        cur = pvs.pvs_cursor_open(index, q)
        pvs.pvs_cursor_set_generator(cur, gen)
        for _ in range(RANKS_PER_QUERY // CHUNK):
            pvs.pvs_next(cur, CHUNK)
        ev = pvs.pvs_cursor_stats(cur)["refined"]
        pvs.pvs_cursor_close(cur)
        return (time.perf_counter() - t) * 1e3, ev

    def fused(name, q, sp):
        index, gen = gens[name]
        torch.cuda.synchronize()
        t = time.perf_counter()
        cur = pvs.pvs_cursor_open(index, q)
        pvs.pvs_cursor_set_generator(cur, gen)
        ids, F, st = pvs.eahr_topk(cur, sp, K=EAHR_K, k=EAHR_RRF_K, form=pvs.EAHR_NUMERATOR)
        ev = pvs.pvs_cursor_stats(cur)["refined"]
        pvs.pvs_cursor_close(cur)
        return (time.perf_counter() - t) * 1e3, ev, ids

    def sparse_for(q, seed):
        return synth.copula_ranking(rows @ q, 0.5, seed).cpu().numpy()

    for w in range(2):   # warm-up
        sp = sparse_for(queries[w], 900 + w)
        for name in gens:
            ranks(name, queries[w])
            fused(name, queries[w], sp)
    launches0 = pvs.pvs_launch_count()
    res = {name: {"ranks_ms": [], "ranks_evals": [], "eahr_ms": [], "eahr_evals": []}
           for name in gens}
    mismatch = 0
    with ClockSampler(local) as clk:
        for i in range(2, nq):
            q = queries[i]
            sp = sparse_for(q, 900 + i)
            top = None
            for name in gens:   # the same query through every generator
                ms, ev = ranks(name, q)
                res[name]["ranks_ms"].append(ms)
                res[name]["ranks_evals"].append(ev)
                ms, ev, ids = fused(name, q, sp)
                res[name]["eahr_ms"].append(ms)
                res[name]["eahr_evals"].append(ev)
                if top is None:
                    top = ids.tolist()
                mismatch += int(ids.tolist() != top)
    launches = pvs.pvs_launch_count() - launches0

    def gmean_ratio(a, b):
        return float(np.exp(np.mean(np.log(np.asarray(a) / np.asarray(b)))))

    table = {}
    for name, r in res.items():
        table[name] = {
            "first_1000_ms_p50": float(np.median(r["ranks_ms"])),
            "first_1000_f32_evals_p50": float(np.median(r["ranks_evals"])),
            "eahr_top20_ms_p50": float(np.median(r["eahr_ms"])),
            "eahr_f32_evals_p50": float(np.median(r["eahr_evals"])),
            "first_1000_ratio_to_pvs": gmean_ratio(r["ranks_ms"], res["pvs"]["ranks_ms"]),
            "eahr_ratio_to_pvs": gmean_ratio(r["eahr_ms"], res["pvs"]["eahr_ms"]),
        }
    line = {
        "metric": "rank-generator ablation: EAHR Top-20 latency ratio scalar/PVS, scan/PVS",
        "value": table["scan"]["eahr_ratio_to_pvs"], "unit": "x (paired geometric mean)",
        "n_gpus": world, "steps": nq - 2, "warmup": 2,
        "ms_per_step": float(np.mean(res["pvs"]["eahr_ms"])), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int8", "data": "synthetic",
        "config": {"workload": f"passage mixture N={n:,} x d={DIM}; generators: PVS (per-vector "
                               "scales), scalar-quantization intervals (one scale for the "
                               "corpus), exhaustive float32 scan; first 1,000 ranks in chunks "
                               f"of {CHUNK}, and EAHR Top-{EAHR_K} against a tau=+0.5 copula "
                               "sparse ranking",
                   "N": n, "d": DIM, "parallelism": f"replicas x{world}"},
        "e2e": {"value": table["scan"]["eahr_ratio_to_pvs"], "unit": "x",
                "h2d_bytes_per_step": DIM * 4, "d2h_bytes_per_step": EAHR_K * 16},
        "generators": table,
        "eahr_results_differ": mismatch,
        "gpu_launches": launches,
        "build_s": {"pvs": t1 - t0, "scalar": t2 - t1},
        "clocks": clk.summary(),
    }
    pvs.pvs_index_free(idx_sq)
    pvs.pvs_index_free(idx_pvs)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


SEGMENTS = 8   # one Shard of eight immutable Segments, as the paper's TREC-DL setup


def main_segments(args, pvs, synth, torch, np, rank, world, local, dev, pg):
    """Hierarchical merging at passage scale: the C2 corpus and the topical
    BM25 corpus of --workload hybrid, each cut into 8 Segments of
    consecutive ids (one Shard).  Per query, the same request twice:
    unsegmented (one PVS index, one PBM index, eahr_topk_pbm) and segmented
    (8 PVS and 8 PBM segment cursors under two merge cursors,
    eahr_topk_merge); plus the first 1,000 dense ranks through one index and
    through the merge.  The two Top-20 results must agree."""
    n = args.n
    stream = torch.cuda.Stream(device=dev)
    centres = synth.mixture_centres(COMPONENTS, DIM, seed=2, device=dev)
    rows = torch.empty((n, DIM), dtype=torch.float32, device=dev)
    chunk = 1 << 20
    for r in range(0, n, chunk):
        c = min(chunk, n - r)
        rows[r:r + c] = synth.mixture_rows(c, centres, WITHIN_STD, seed=2, first=r)
    bounds = [(n * i // SEGMENTS, n * (i + 1) // SEGMENTS) for i in range(SEGMENTS)]
    t0 = time.perf_counter()
    d_full = pvs.pvs_build(rows, stream=stream.cuda_stream)
    # each Segment index gets a stream of its own (the library creates it),
    # so the merge's concurrent refills of Segment cursors overlap on the GPU
    d_seg = [pvs.pvs_build(rows[a:b]) for a, b in bounds]
    del rows
    torch.cuda.synchronize()
    comps = synth.mixture_components(n, COMPONENTS, seed=2, device=dev)
    off, docs, imps = synth.bm25_postings(n, SPARSE_TERMS, SPARSE_TOKENS, seed=10, device=dev,
                                          topic_of=comps, topic_terms=HYBRID_TOPIC_TERMS,
                                          topic_share=HYBRID_TOPIC_SHARE)
    del comps
    s_full = pvs.pbm_build(off, docs, imps, n)
    term_of = torch.repeat_interleave(torch.arange(off.numel() - 1, device=dev),
                                      off[1:] - off[:-1])
    s_seg = []
    for a, b in bounds:   # the postings of items a .. b-1, renumbered from 0
        sel = torch.nonzero((docs >= a) & (docs < b)).squeeze(1)
        cnt = torch.bincount(term_of[sel], minlength=off.numel() - 1)
        o = torch.zeros(off.numel(), dtype=torch.int64, device=dev)
        o[1:] = torch.cumsum(cnt, 0)
        s_seg.append(pvs.pbm_build(o, (docs[sel] - a).to(torch.int32), imps[sel], b - a))
    del term_of
    torch.cuda.synchronize()
    build_s = time.perf_counter() - t0
    nq = 2 + args.eahr_queries
    dq = synth.mixture_queries(nq, centres, QUERY_NOISE, seed=query_seed(15, rank))
    qc = synth.mixture_query_components(nq, COMPONENTS, seed=query_seed(15, rank), device=dev)
    sq = synth.topical_queries(qc, off, SPARSE_TERMS, HYBRID_TOPIC_TERMS,
                               seed=query_seed(16, rank))

    def unsegmented(i):
        torch.cuda.synchronize()
        t = time.perf_counter()
        dc = pvs.pvs_cursor_open(d_full, dq[i])
        sc = pvs.pbm_cursor_open(s_full, *sq[i])
        ids, _, _ = pvs.eahr_topk_pbm(dc, sc, K=EAHR_K, k=EAHR_RRF_K, form=pvs.EAHR_NUMERATOR)
        pvs.pbm_cursor_close(sc)
        pvs.pvs_cursor_close(dc)
        return (time.perf_counter() - t) * 1e3, ids

    def segmented(i):
        torch.cuda.synchronize()
        t = time.perf_counter()
        dcs = [pvs.pvs_cursor_open(x, dq[i]) for x in d_seg]
        scs = [pvs.pbm_cursor_open(x, *sq[i]) for x in s_seg]
        dm = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, a) for c, (a, _) in zip(dcs, bounds)])
        sm = pvs.pvs_merge_open([(pvs.PVS_CHILD_SPARSE, c, a) for c, (a, _) in zip(scs, bounds)])
        ids, _, _ = pvs.eahr_topk_merge(dm, sm, K=EAHR_K, k=EAHR_RRF_K, form=pvs.EAHR_NUMERATOR)
        st = pvs.pvs_merge_stats(dm)
        pvs.pvs_merge_close(dm)
        pvs.pvs_merge_close(sm)
        for c in dcs:
            pvs.pvs_cursor_close(c)
        for c in scs:
            pvs.pbm_cursor_close(c)
        return (time.perf_counter() - t) * 1e3, ids, st

    def ranks_single(i):
        torch.cuda.synchronize()
        t = time.perf_counter()
        c = pvs.pvs_cursor_open(d_full, dq[i])
        out = [pvs.pvs_next(c, CHUNK)[0] for _ in range(RANKS_PER_QUERY // CHUNK)]
        pvs.pvs_cursor_close(c)
        return (time.perf_counter() - t) * 1e3, np.concatenate(out)

    def ranks_merged(i):
        torch.cuda.synchronize()
        t = time.perf_counter()
        dcs = [pvs.pvs_cursor_open(x, dq[i]) for x in d_seg]
        dm = pvs.pvs_merge_open([(pvs.PVS_CHILD_DENSE, c, a) for c, (a, _) in zip(dcs, bounds)])
        out = [pvs.pvs_merge_next(dm, CHUNK)[0] for _ in range(RANKS_PER_QUERY // CHUNK)]
        pvs.pvs_merge_close(dm)
        for c in dcs:
            pvs.pvs_cursor_close(c)
        return (time.perf_counter() - t) * 1e3, np.concatenate(out)

    for w in range(2):
        unsegmented(w)
        segmented(w)
        ranks_single(w)
        ranks_merged(w)
    launches0 = pvs.pvs_launch_count()
    lat_u, lat_s, lat_r1, lat_rm, differ, depth = [], [], [], [], 0, []
    with ClockSampler(local) as clk:
        for i in range(2, nq):
            ms_u, ids_u = unsegmented(i)
            ms_s, ids_s, st = segmented(i)
            ms_1, r1 = ranks_single(i)
            ms_m, rm = ranks_merged(i)
            lat_u.append(ms_u)
            lat_s.append(ms_s)
            lat_r1.append(ms_1)
            lat_rm.append(ms_m)
            depth.append(st["emitted"])
            differ += int(ids_u.tolist() != ids_s.tolist()) + int(not np.array_equal(r1, rm))
    launches = pvs.pvs_launch_count() - launches0
    line = {
        "metric": "EAHR Top-20 latency over 8 Segments, PVS + PBM (p50)",
        "value": float(np.median(lat_s)), "unit": "ms", "n_gpus": world, "steps": len(lat_s),
        "warmup": 2, "ms_per_step": float(np.mean(lat_s)), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "int8", "data": "synthetic",
        "config": {"workload": f"one Shard of {SEGMENTS} Segments of consecutive ids over the "
                               f"passage mixture (N={n:,} x d={DIM}) and the topical BM25 "
                               "corpus of --workload hybrid; EAHR Top-20 over two merge "
                               "cursors vs one index per channel",
                   "N": n, "segments": SEGMENTS, "K": EAHR_K, "rrf_k": EAHR_RRF_K,
                   "parallelism": f"replicas x{world}"},
        "e2e": {"value": float(np.median(lat_s)), "unit": "ms",
                "h2d_bytes_per_step": SEGMENTS * DIM * 4, "d2h_bytes_per_step": EAHR_K * 16},
        "eahr_ms": {"segmented_p50": float(np.median(lat_s)),
                    "segmented_p95": float(np.percentile(lat_s, 95)),
                    "unsegmented_p50": float(np.median(lat_u)),
                    "unsegmented_p95": float(np.percentile(lat_u, 95))},
        "first_1000_dense_ms": {"merged_8_p50": float(np.median(lat_rm)),
                                "single_index_p50": float(np.median(lat_r1))},
        "dense_merge_depth_p50": float(np.median(depth)),
        "results_differ": differ,
        "gpu_launches": launches, "build_s": build_s,
        "clocks": clk.summary(),
    }
    for x in d_seg + [d_full]:
        pvs.pvs_index_free(x)
    for x in s_seg + [s_full]:
        pvs.pbm_index_free(x)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


HYBRID_TOPIC_TERMS = 64     # topic block per mixture component
HYBRID_TOPIC_SHARE = 0.3    # share of an item's tokens drawn from its topic block


def main_hybrid(args, pvs, synth, torch, np, rank, world, local, dev, pg):
    """EAHR end to end with both generators on the GPU: PVS over the passage
    mixture corpus (dense) and PBM over a topical synthetic BM25 corpus of
    the same items (sparse: a share of every item's tokens comes from its
    mixture component's term block, and each query draws terms from its own
    component's block, so the two rankings agree in part).  Timed per query:
    both cursors opened, eahr_topk_pbm, both closed.  Beside it, the
    exhaustive comparator in plain torch: fp32 dense scores of every row and a
    full sort, the complete sparse ranking, and complete-list fusion."""
    n = args.n
    stream = torch.cuda.Stream(device=dev)
    centres = synth.mixture_centres(COMPONENTS, DIM, seed=2, device=dev)
    t0 = time.perf_counter()
    rows = torch.empty((n, DIM), dtype=torch.float32, device=dev)
    chunk = 1 << 20
    for r in range(0, n, chunk):
        c = min(chunk, n - r)
        rows[r:r + c] = synth.mixture_rows(c, centres, WITHIN_STD, seed=2, first=r)
    index = pvs.pvs_build(rows, stream=stream.cuda_stream)
    torch.cuda.synchronize()
    dense_build_s = time.perf_counter() - t0
    t0 = time.perf_counter()
    comps = synth.mixture_components(n, COMPONENTS, seed=2, device=dev)
    off, docs, imps = synth.bm25_postings(n, SPARSE_TERMS, SPARSE_TOKENS, seed=10, device=dev,
                                          topic_of=comps, topic_terms=HYBRID_TOPIC_TERMS,
                                          topic_share=HYBRID_TOPIC_SHARE)
    del comps
    sindex = pvs.pbm_build(off, docs, imps, n)
    torch.cuda.synchronize()
    sparse_build_s = time.perf_counter() - t0
    nq = 2 + args.eahr_queries
    dq = synth.mixture_queries(nq, centres, QUERY_NOISE, seed=query_seed(12, rank))
    qc = synth.mixture_query_components(nq, COMPONENTS, seed=query_seed(12, rank), device=dev)
    sq = synth.topical_queries(qc, off, SPARSE_TERMS, HYBRID_TOPIC_TERMS,
                               seed=query_seed(13, rank))

    def one(i):
        torch.cuda.synchronize()
        t = time.perf_counter()
        dcur = pvs.pvs_cursor_open(index, dq[i])
        scur = pvs.pbm_cursor_open(sindex, *sq[i])
        ids, F, st = pvs.eahr_topk_pbm(dcur, scur, K=EAHR_K, k=EAHR_RRF_K,
                                       form=pvs.EAHR_NUMERATOR, policy=eahr_policy(args, pvs))
        ps = pvs.pbm_cursor_stats(scur)
        pvs.pbm_cursor_close(scur)
        pvs.pvs_cursor_close(dcur)
        ms = (time.perf_counter() - t) * 1e3
        if len(ids) != EAHR_K:
            raise RuntimeError("EAHR returned a short list")
        return ms, st, ps

    def full_orders(i):
        sc = rows @ dq[i]
        dorder = torch.argsort(sc, descending=True, stable=True)
        ss = torch.zeros(n, dtype=torch.float32, device=dev)
        for term, w in zip(sq[i][0].tolist(), sq[i][1].tolist()):
            a, b = int(off[term]), int(off[term + 1])
            ss.index_put_((docs[a:b].long(),), imps[a:b] * w, accumulate=True)
        sorder = torch.argsort(ss, descending=True, stable=True)
        return dorder, sorder, ss

    def comparator(i):
        torch.cuda.synchronize()
        t = time.perf_counter()
        dorder, sorder, ss = full_orders(i)
        ar = torch.arange(1, n + 1, dtype=torch.float64, device=dev)
        rd = torch.empty(n, dtype=torch.float64, device=dev)
        rd[dorder] = ar
        rs = torch.empty(n, dtype=torch.float64, device=dev)
        rs[sorder] = ar
        # the sparse list is the positive-score support (Sec. 2.1)
        fused = 1.0 / (EAHR_RRF_K + rd) + torch.where(ss > 0, 1.0 / (EAHR_RRF_K + rs), 0.0)
        torch.topk(fused, EAHR_K).indices.cpu()
        return (time.perf_counter() - t) * 1e3

    for w in range(2):
        one(w)
        comparator(w)
    dorder, sorder, _ = full_orders(2)
    ktau = synth.kendall_tau_sample(dorder.cpu().numpy(), sorder.cpu().numpy(), 200_000, seed=5)
    del dorder, sorder
    if pg:
        pg.barrier()
    launches0 = pvs.pvs_launch_count()
    lat, dd, ds, ex, rexp = [], [], [], 0, []
    finish = {0: 0, 1: 0, 2: 0, 3: 0}
    with ClockSampler(local) as clk:
        for i in range(2, nq):
            ms, st, ps = one(i)
            lat.append(ms)
            dd.append(st["depth"][0])
            ds.append(st["depth"][1])
            ex += int(st["exhausted"][0] and st["exhausted"][1])
            rexp.append(ps["ranges_expanded"])
            finish[int(st.get("complete", 0))] += 1
    launches = pvs.pvs_launch_count() - launches0
    cmp_ms = [comparator(i) for i in range(2, min(nq, 22))]
    line = {
        "metric": "EAHR Top-20 latency, PVS dense + PBM sparse (p50)",
        "value": float(np.median(lat)), "unit": "ms", "n_gpus": world, "steps": len(lat),
        "warmup": 2, "ms_per_step": float(np.mean(lat)), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "int8", "data": "synthetic",
        "config": {"workload": f"EAHR over PVS (passage mixture N={n:,} x d={DIM}) and PBM "
                               f"(topical synthetic BM25 over the same items: vocabulary "
                               f"{SPARSE_TERMS:,} + {COMPONENTS} x {HYBRID_TOPIC_TERMS} topic "
                               f"terms, topic share {HYBRID_TOPIC_SHARE}), weighted RRF "
                               f"1/(60+rank), K={EAHR_K}",
                   "N": n, "d": DIM, "K": EAHR_K, "rrf_k": EAHR_RRF_K,
                   "policy": args.eahr_policy, "postings": int(docs.numel()),
                   "l2": "no flush: every query's interval pass streams 6.9 GB of codes",
                   "parallelism": f"replicas x{world}"},
        "e2e": {"value": float(np.median(lat)), "unit": "ms",
                "h2d_bytes_per_step": DIM * 4 + int(np.mean([8 * len(q[0]) for q in sq])),
                "d2h_bytes_per_step": EAHR_K * 16},
        "latency_ms": {"p50": float(np.median(lat)), "p95": float(np.percentile(lat, 95)),
                       "p99": float(np.percentile(lat, 99))},
        "kendall_tau_dense_sparse": ktau,
        "dense_depth_p50": float(np.median(dd)), "sparse_depth_p50": float(np.median(ds)),
        "both_exhausted": ex, "pbm_ranges_expanded_p50": float(np.median(rexp)),
        "finished_by": {"reading": finish[0], "rank_intervals": finish[2],
                        "exact_ranks": finish[3]},
        "pbm_ranges": pvs.pbm_index_ranges(sindex),
        "exhaustive_torch_ms_p50": float(np.median(cmp_ms)),
        "gpu_launches": launches,
        "dense_build_s": dense_build_s, "sparse_build_s": sparse_build_s,
        "clocks": clk.summary(),
    }
    pvs.pbm_index_free(sindex)
    pvs.pvs_index_free(index)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


SNAP_N = 2_000_000
SNAP_DIM = 1024
SNAP_DUP = 0.2          # near-duplicate share of the base corpus
SNAP_DUP_STD = 1e-4     # their noise (standard deviation)
SNAP_STEPS = 5
SNAP_APPEND = 0.1       # of the base size, per snapshot
SNAP_TOMB = 0.02        # of the live rows, per snapshot
SNAP_TAU = 0.2


def main_snapshots(args, pvs, synth, torch, np, rank, world, local, dev, pg):
    """Adversarial ties and snapshots: a 2,000,000 x 1,024 mixture corpus whose
    last 20 % are near-duplicates of earlier rows (copies + N(0, 1e-4^2),
    normalised); snapshot 1 is that corpus, every later snapshot appends 10 %
    new mixture rows and tombstones 2 % of the live rows.  Per snapshot, 100
    queries run EAHR Top-20 with a sparse channel that is a Gaussian-copula
    ranking (Kendall tau 0.2) of the snapshot's visible ids."""
    n0 = SNAP_N if args.n == N_CORPUS else args.n
    d = SNAP_DIM
    stream = torch.cuda.Stream(device=dev)
    centres = synth.mixture_centres(COMPONENTS, d, seed=5, device=dev)
    total = n0 + (SNAP_STEPS - 1) * int(SNAP_APPEND * n0)
    rows = torch.empty((total, d), dtype=torch.float32, device=dev)
    n_mix = n0 - int(SNAP_DUP * n0)
    t0 = time.perf_counter()
    rows[:n_mix] = synth.mixture_rows(n_mix, centres, WITHIN_STD, seed=5)
    g = torch.Generator(device=dev)
    g.manual_seed(55)
    src = torch.randint(0, n_mix, (n0 - n_mix,), generator=g, device=dev)
    rows[n_mix:n0] = synth.near_duplicate_rows(rows[src], SNAP_DUP_STD, seed=56)
    index = pvs.pvs_build(rows[:n0], stream=stream.cuda_stream)
    torch.cuda.synchronize()
    build_s = time.perf_counter() - t0
    visible = torch.ones(total, dtype=torch.bool, device=dev)
    visible[n0:] = False
    rng = np.random.default_rng(57 + rank)
    queries = synth.mixture_queries(SNAP_STEPS * args.snap_queries + 2, centres, QUERY_NOISE,
                                    seed=query_seed(58, rank))
    launches0 = pvs.pvs_launch_count()
    per_snap = []
    size = n0
    qi = 0
    lat_all = []
    with ClockSampler(local) as clk:
        for step in range(SNAP_STEPS):
            if step > 0:   # grow and delete, then freeze
                add = int(SNAP_APPEND * n0)
                rows[size:size + add] = synth.mixture_rows(add, centres, WITHIN_STD,
                                                           seed=60 + step)
                pvs.pvs_append(index, rows[size:size + add])
                visible[size:size + add] = True
                size += add
                live = torch.nonzero(visible[:size]).squeeze(1).cpu().numpy()
                dead = rng.choice(live, int(SNAP_TOMB * live.size), replace=False)
                pvs.pvs_tombstone(index, dead)
                visible[torch.from_numpy(dead).to(dev)] = False
            snap = pvs.pvs_snapshot_create(index)
            vis_ids = torch.nonzero(visible[:size]).squeeze(1)
            lat, depth, ex_any, ex_both, near_ties, swaps = [], [], 0, 0, None, None
            finish = {0: 0, 1: 0, 2: 0, 3: 0}
            for j in range(args.snap_queries):
                q = queries[qi]
                qi += 1
                proxy = rows[vis_ids] @ q
                sparse = vis_ids[synth.copula_ranking(proxy, SNAP_TAU, 900 + qi)].cpu().numpy()
                torch.cuda.synchronize()
                t = time.perf_counter()
                cur = pvs.pvs_cursor_open(index, q, snap)
                ids, F, st = pvs.eahr_topk(cur, sparse, K=EAHR_K, k=EAHR_RRF_K,
                                           form=pvs.EAHR_NUMERATOR,
                                           policy=eahr_policy(args, pvs))
                pvs.pvs_cursor_close(cur)
                lat.append((time.perf_counter() - t) * 1e3)
                depth.append(st["depth"][0])
                finish[int(st.get("complete", 0))] += 1
                ex_any += int(st["exhausted"][0] or st["exhausted"][1])
                ex_both += int(st["exhausted"][0] and st["exhausted"][1])
                if j == 0:   # near ties among the first 1,000 dense ranks of this snapshot
                    cur = pvs.pvs_cursor_open(index, q, snap)
                    d_ids, d_sc, _ = pvs.pvs_next(cur, 1000)
                    pvs.pvs_cursor_close(cur)
                    a = d_sc[:-1].astype(np.float64)
                    b = d_sc[1:].astype(np.float64)
                    near_ties = int(np.sum(np.abs(a - b) < 2.0 ** -20 *
                                           np.maximum(np.abs(a), np.abs(b))))
                    if args.oracle_check:
                        from oracle import pvs_oracle as po
                        vis_host = visible[:size].cpu().numpy()
                        ref_ids, _ = po.dense_ranking(q.cpu().numpy(),
                                                      rows[:size].cpu().numpy(), vis_host)
                        swaps = int(np.sum(ref_ids[:len(d_ids)] != d_ids))
            pvs.pvs_snapshot_free(snap)
            lat_all.extend(lat)
            per_snap.append({
                "snapshot": step + 1, "rows": size, "visible": int(vis_ids.numel()),
                "queries": args.snap_queries,
                "latency_ms_p50": float(np.median(lat)), "latency_ms_p95": float(np.percentile(lat, 95)),
                "dense_depth_p50": float(np.median(depth)),
                "exhaustion_rate_any": ex_any / args.snap_queries,
                "exhaustion_rate_both": ex_both / args.snap_queries,
                "near_tie_pairs_first_1000": near_ties,
                "oracle_mismatches_first_1000": swaps,
                "finished_by": {"reading": finish[0], "rank_intervals": finish[2],
                                "exact_ranks": finish[3], "complete_list_fusion": finish[1]}})
    launches = pvs.pvs_launch_count() - launches0
    p50 = float(np.median(lat_all))
    line = {
        "metric": "EAHR Top-20 latency (p50 over five snapshots)", "value": p50, "unit": "ms",
        "n_gpus": world, "steps": len(lat_all), "warmup": 0, "ms_per_step": float(np.mean(lat_all)),
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "int8",
        "data": "synthetic",
        "config": {"workload": "adversarial ties + snapshots: N=2,000,000 x d=1,024 mixture with "
                               "20% near-duplicates (std 1e-4), +10% appended and 2% tombstoned "
                               "per snapshot, 5 snapshots, EAHR Top-20, sparse Kendall tau 0.2",
                   "N": n0, "d": d, "K": EAHR_K, "rrf_k": EAHR_RRF_K, "policy": args.eahr_policy,
                   "l2": "no flush: every query's interval pass streams >= 2 GB of codes",
                   "parallelism": f"replicas x{world}"},
        "e2e": {"value": p50, "unit": "ms", "h2d_bytes_per_step": d * 4,
                "d2h_bytes_per_step": EAHR_K * (8 + 8)},
        "snapshots": per_snap,
        "gpu_launches": launches,
        "build_s": build_s,
        "clocks": clk.summary(),
    }
    pvs.pvs_index_free(index)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


def eahr_record(args, pvs, synth, torch, np, index, centres, n, rank, dev):
    """The EAHR Top-20 configuration on the passage index (K = 20, weighted
    RRF 1 / (60 + rank), a Gaussian-copula sparse ranking of every id per
    query at Kendall tau +0.5 / 0 / -0.5, the adaptive policy): per-level
    latency, depth and the exhaustive comparator, for the default line."""
    rows = torch.empty((n, DIM), dtype=torch.float32, device=dev)   # the copula's proxy
    for r in range(0, n, 1 << 20):
        c = min(1 << 20, n - r)
        rows[r:r + c] = synth.mixture_rows(c, centres, WITHIN_STD, seed=2, first=r)
    counts = {0.5: args.eahr_queries, 0.0: args.eahr_queries, -0.5: args.eahr_exhaust_queries}
    queries = synth.mixture_queries(sum(counts.values()) + 2, centres, QUERY_NOISE,
                                    seed=query_seed(5003, rank))
    levels, _ = eahr_levels(pvs, synth, torch, np, index, rows, queries,
                            pvs.EAHR_POLICY_ADAPTIVE, counts, rank, dev, warmup=2,
                            comparator_queries=20)
    del rows
    torch.cuda.empty_cache()
    return {"metric": "EAHR Top-20 latency", "unit": "ms", "higher_is_better": False,
            "K": EAHR_K, "rrf": "1/(60+rank), w_d = w_s = 1", "policy": "adaptive",
            "timed": "cursor open + eahr_topk + close per query, host clock, sparse ids in "
                     "host memory",
            "comparator": "exhaustive fp32 scoring + full sort + complete-list fusion in plain "
                          "torch, first 20 queries of each level",
            "levels": levels}


def main_passage(args, pvs, synth, torch, np, rank, world, local, dev, pg):
    """The passage workload (the default): the queries of a step served by
    the native executor, GROUP at a time from one grouped pass over the
    codes, every 20-rank page of a group's cursors in one batched pull."""
    stream = torch.cuda.Stream(device=dev)
    n = args.n
    group = max(1, min(args.group, pvs.PVS_GROUP_MAX))
    index, centres, build_s = build_corpus_index(pvs, synth, torch, n, stream.cuda_stream, dev)
    nq = args.queries
    total_q = (args.warmup + args.steps) * nq
    queries = synth.mixture_queries(total_q, centres, QUERY_NOISE, seed=query_seed(3, rank))
    queries = queries.reshape(total_q, DIM).contiguous()
    warm_q = queries[:args.warmup * nq]
    timed_q = queries[args.warmup * nq:]
    n_timed = timed_q.shape[0]
    n_buf = max(n_timed, warm_q.shape[0])   # the warm-up may hold more queries than the timed steps
    ids_buf = torch.empty((n_buf, RANKS_PER_QUERY), dtype=torch.int64, device=dev)
    scores_buf = torch.empty((n_buf, RANKS_PER_QUERY), dtype=torch.float32, device=dev)
    ids, scores = ids_buf[:n_timed], scores_buf[:n_timed]
    executor = pvs.pvs_executor_create(index, PIPELINE)
    try:
        pvs.pvs_executor_set_group(executor, group)
        if warm_q.shape[0]:
            pvs.pvs_executor_run_device(executor, warm_q, RANKS_PER_QUERY, CHUNK,
                                        ids_buf[:warm_q.shape[0]], scores_buf[:warm_q.shape[0]])
        st0 = pvs.pvs_executor_stats(executor)

        # ---- timed region: device-resident queries and outputs ----
        if pg:
            pg.barrier()
        torch.cuda.synchronize()
        launches0 = pvs.pvs_launch_count()
        start = torch.cuda.Event(enable_timing=True)
        end = torch.cuda.Event(enable_timing=True)
        with ClockSampler(local) as clk:
            start.record(stream)
            n_out, status, rc = pvs.pvs_executor_run_device(executor, timed_q, RANKS_PER_QUERY,
                                                            CHUNK, ids, scores)
            end.record(stream)
            stream.synchronize()
        torch.cuda.synchronize()
        launches = pvs.pvs_launch_count() - launches0
        st1 = pvs.pvs_executor_stats(executor)
        if rc != pvs.PVS_OK or int(n_out.min()) != RANKS_PER_QUERY:
            raise RuntimeError(f"executor run failed: {rc}")
        elapsed = start.elapsed_time(end) / 1e3
        elapsed = slowest(pg, elapsed, dev)
        ranks_total = n_timed * RANKS_PER_QUERY * world
        value = job_rate(n_timed * RANKS_PER_QUERY, world, elapsed)

        # ---- e2e: pinned host queries and outputs through the same executor ----
        qh = timed_q.cpu().pin_memory()
        h_ids = torch.empty((n_timed, RANKS_PER_QUERY), dtype=torch.int64).pin_memory()
        h_sc = torch.empty((n_timed, RANKS_PER_QUERY), dtype=torch.float32).pin_memory()
        if pg:
            pg.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        _, _, n_got, _, rc = pvs.pvs_executor_run(executor, qh, RANKS_PER_QUERY, CHUNK,
                                                  ids=h_ids, scores=h_sc)
        torch.cuda.synchronize()
        e2e_elapsed = time.perf_counter() - t0
        if rc != pvs.PVS_OK or int(n_got.min()) != RANKS_PER_QUERY:
            raise RuntimeError(f"executor run failed: {rc}")
        # the two legs deliver the same ranks
        same = bool(torch.equal(h_ids, ids.cpu()))
    finally:
        pvs.pvs_executor_destroy(executor)

    # ---- latency of a lone query (its own cursor and pass), one at a time ----
    out_ids = torch.empty((1, RANKS_PER_QUERY), dtype=torch.int64, device=dev)
    out_scores = torch.empty((1, RANKS_PER_QUERY), dtype=torch.float32, device=dev)
    lone = []
    lat20, lat1000 = measure_latency(pvs, torch, index, timed_q, out_ids, out_scores, stream,
                                     min(n_timed, 20), lone)
    e2e_elapsed = slowest(pg, e2e_elapsed, dev)
    e2e_value = ranks_total / e2e_elapsed

    # ---- roofline of the grouped interval pass ----
    m_pad = ((DIM + 63) // 64) * 64
    passes = st1["interval_passes"] - st0["interval_passes"]
    pass_ms = (st1["interval_ms"] - st0["interval_ms"]) / max(passes, 1)
    read_bytes = n * (m_pad + 12)
    # bounds (lo, hi) of every row per query, and with groups the largest
    # upper bound of each 16-row block per query
    write_bytes = 8 * n * group + (4 * ((n + 15) // 16) * group if group > 1 else 0)
    alg_bytes = read_bytes + write_bytes
    achieved = alg_bytes / (pass_ms / 1e3) / 1e9
    peak, peak_kind = measured_peaks()
    kernel = "interval_group_kernel" if group > 1 else "interval_pass_kernel"
    traffic = (interval_traffic(n, "interval_group_kernel_passage_traffic.json") if group > 1
               else interval_traffic(n))

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": elapsed / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int8", "data": "synthetic",
        "config": {"workload": WORKLOAD, "N": n, "d": DIM, "queries_per_step": nq,
                   "ranks_per_query": RANKS_PER_QUERY, "chunk": CHUNK,
                   "queries_per_pass": group, "executor_workers": PIPELINE,
                   "l2": "no flush: each interval pass streams 6.9 GB of codes (> 129 MB L2)",
                   "parallelism": f"replicas x{world} (queries sharded, no collective)"},
        "e2e": {"value": e2e_value, "unit": UNIT,
                "h2d_bytes_per_step": nq * DIM * 4,
                "d2h_bytes_per_step": nq * RANKS_PER_QUERY * (8 + 4),
                "path": f"pvs_executor_run: {PIPELINE} native workers, {group} queries per "
                        f"pass, pages of {CHUNK} through batched pulls, pinned host queries and "
                        "outputs",
                "same_ranks_as_value_leg": same},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "peak_kind": peak_kind, "kernel": kernel,
                     "frac_of_8tbs_nominal": achieved / 8000.0,
                     "algorithmic_bytes": {"codes_and_params_read": read_bytes,
                                           "bounds_written": write_bytes}},
        "gpu_launches": launches,
        "latency_ms": {"first_20_p50": statistics.median(lat20),
                       "first_1000_p50": statistics.median(lat1000),
                       "first_1000_p95": sorted(lat1000)[int(0.95 * (len(lat1000) - 1))],
                       "note": "a lone query with its own cursor and single-query pass"},
        "interval_pass": {"ms": pass_ms, "GBps": achieved, "queries_per_pass": group,
                          "ms_per_query": pass_ms / group, "passes_timed": passes},
        "single_query_pass": single_pass_record(lone, n, m_pad, peak),
        "per_query": {"refined_mean": (st1["refined"] - st0["refined"]) / n_timed},
        "build_s": build_s,
        "clocks": clk.summary(),
    }
    if rank == 0 and not args.no_eahr:
        line["eahr"] = eahr_record(args, pvs, synth, torch, np, index, centres, n, rank, dev)
    if rank == 0 and not args.no_cpu_baseline:
        qb = timed_q[:64].cpu().numpy()
        line["cpu_baseline"] = cpu_baseline(synth, torch, centres, qb, n)
    pvs.pvs_index_free(index)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


def main():
    global PIPELINE, BATCH_PIPELINE, SPARSE_WORKERS
    args = parse()
    if args.pipeline > 0:
        PIPELINE = BATCH_PIPELINE = SPARSE_WORKERS = args.pipeline
    if args.impl == "reference":
        reference_arm(args)
        return
    import numpy as np
    import torch
    import paper_2608_07152_gb300 as pvs
    import synth

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    if args.workload == "batched":
        main_batched(args, pvs, synth, torch, np, rank, world, local, dev, pg)
        return
    if args.workload == "eahr":
        main_eahr(args, pvs, synth, torch, np, rank, world, local, dev, pg)
        return
    if args.workload == "snapshots":
        main_snapshots(args, pvs, synth, torch, np, rank, world, local, dev, pg)
        return
    if args.workload == "sparse":
        main_sparse(args, pvs, synth, torch, np, rank, world, local, dev, pg)
        return
    if args.workload == "hybrid":
        main_hybrid(args, pvs, synth, torch, np, rank, world, local, dev, pg)
        return
    if args.workload == "ablation":
        main_ablation(args, pvs, synth, torch, np, rank, world, local, dev, pg)
        return
    if args.workload == "segments":
        main_segments(args, pvs, synth, torch, np, rank, world, local, dev, pg)
        return

    main_passage(args, pvs, synth, torch, np, rank, world, local, dev, pg)


if __name__ == "__main__":
    main()
