// Native request executor (include/executor.h): arXiv 2608.07152 Sec. 2.1
// (ranked lists read page by page as a stable, only-extended prefix) over
// the PVS cursors of Sec. 2.3.
//
// A fixed pool of worker threads, each bound to the index's device with its
// own non-blocking stream.  A run publishes one job and bumps a generation
// counter; the workers take request indexes from an atomic counter.  For a
// request a worker opens the cursor on its own stream, reads the pages one
// after another through pvs_next straight into the request's rows of the
// caller's buffers, and closes the cursor.  With a group size G >= 2 a
// worker takes G requests at a time: one grouped open (one pass over the
// codes for all G queries, pvs_cursor_open_group), then every page of the G
// cursors in one batched pull.  No lock is held across a device wait; the
// job lock is taken only at the start and end of a run.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <condition_variable>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include "../../include/executor.h"
#include "runtime.h"

namespace {

constexpr int32_t kMaxWorkers = 64;

struct Job {
    const pvs_snapshot* snap = nullptr;
    const float* queries = nullptr;
    int32_t nq = 0, ranks = 0, page = 0;
    int32_t on_device = 0;              // queries, ids and scores in device memory
    int64_t* ids = nullptr;
    float* scores = nullptr;
    int32_t* n_out = nullptr;
    int32_t* status = nullptr;
};

}  // namespace

struct pvs_executor {
    pvs_index* index = nullptr;
    std::vector<std::thread> threads;
    std::vector<cudaStream_t> streams;
    std::mutex m;                       // job, generation, busy, stop
    std::condition_variable work_cv, done_cv;
    Job job;
    uint64_t generation = 0;
    int busy = 0;                       // workers not yet done with the job
    bool stop = false;
    std::atomic<int32_t> next{0};       // next request index to hand out
    std::mutex run_mutex;               // one run at a time
    int32_t group = 1;                  // requests per grouped open
    std::atomic<int64_t> requests{0}, failed{0}, pages{0}, ranks{0};
    std::atomic<int64_t> passes{0}, refined{0};
    std::mutex ms_mutex;
    double interval_ms = 0.0;           // device time of the passes over the codes
};

namespace {

// Ranks [from, ranks) of request i's row: -1 / NaN (device rows: all bits
// set, which is -1 as an int64 and a NaN as a float32).
void fill_rest(const Job& j, cudaStream_t st, int32_t i, int32_t from) {
    if (from >= j.ranks) return;
    int64_t* ids = j.ids + (size_t)i * j.ranks;
    float* sc = j.scores + (size_t)i * j.ranks;
    if (j.on_device) {
        cudaMemsetAsync(ids + from, 0xff, (size_t)(j.ranks - from) * sizeof(int64_t), st);
        cudaMemsetAsync(sc + from, 0xff, (size_t)(j.ranks - from) * sizeof(float), st);
        return;
    }
    for (int32_t k = from; k < j.ranks; ++k) {
        ids[k] = -1;
        sc[k] = NAN;
    }
}

void count_request(pvs_executor* ex, pvs_status s, int64_t pages, int32_t total) {
    ex->requests.fetch_add(1, std::memory_order_relaxed);
    if (s < 0) ex->failed.fetch_add(1, std::memory_order_relaxed);
    ex->pages.fetch_add(pages, std::memory_order_relaxed);
    ex->ranks.fetch_add(total, std::memory_order_relaxed);
}

// The pass counters of a closed group: the interval time of its cursors'
// passes (a grouped pass is counted once) and their exact evaluations.
void count_passes(pvs_executor* ex, pvs_cursor* const* cs, int n, bool grouped) {
    double ms = 0.0;
    int64_t passes = 0, refined = 0;
    for (int i = 0; i < n; ++i) {
        pvs_stats st;
        if (pvs_cursor_stats(cs[i], &st) != PVS_OK) continue;
        refined += st.refined;
        if (!grouped || i == 0) {
            ms += st.interval_ms;
            passes += st.interval_passes;
        }
    }
    ex->passes.fetch_add(passes, std::memory_order_relaxed);
    ex->refined.fetch_add(refined, std::memory_order_relaxed);
    std::lock_guard<std::mutex> lk(ex->ms_mutex);
    ex->interval_ms += ms;
}

// One request on its own cursor: open, read the pages, close.  Returns the
// request's status.
pvs_status serve_one(pvs_executor* ex, const Job& j, cudaStream_t st, int32_t i,
                     pvs_cursor* c, int32_t total) {
    int64_t* ids = j.ids + (size_t)i * j.ranks;
    float* sc = j.scores + (size_t)i * j.ranks;
    int64_t pages = 0;
    pvs_status s = PVS_OK;
    const bool own = c == nullptr;   // a cursor handed over was counted with its group
    if (!c) {
        const int32_t dim = ex->index->m;
        s = pvs::cursor_open_on(ex->index, j.snap, j.queries + (size_t)i * dim, j.on_device, st,
                                &c);
    }
    if (s == PVS_OK && c) {
        while (total < j.ranks) {
            int32_t got = 0;
            const int32_t n = std::min(j.page, j.ranks - total);
            s = j.on_device ? pvs_next_device(c, n, ids + total, sc + total, &got)
                            : pvs_next(c, n, ids + total, sc + total, &got);
            ++pages;
            if (s < 0) break;
            total += got;
            if (s == PVS_EXHAUSTED || got < n) break;
        }
        if (s >= 0 && j.on_device) s = pvs_cursor_sync(c);   // device work done, status read
    }
    if (c) {
        if (own) count_passes(ex, &c, 1, false);
        pvs_cursor_close(c);
    }
    fill_rest(j, st, i, total);
    if (j.on_device) cudaStreamSynchronize(st);
    j.n_out[i] = total;
    count_request(ex, s < 0 ? s : PVS_OK, pages, total);
    return s == PVS_EXHAUSTED ? PVS_EXHAUSTED : (s < 0 ? s : PVS_OK);
}

// Requests first .. first+count-1 (2 <= count <= PVS_GROUP_MAX) from one
// grouped open; each page of every cursor in one batched pull.  A failed
// open (a bad query) serves the group's requests one by one instead; a
// failure of the batched pull leaves the failed cursors' requests with
// their error and the others continuing one by one.
void serve_group(pvs_executor* ex, const Job& j, cudaStream_t st, int32_t first, int32_t count) {
    const int32_t dim = ex->index->m;
    pvs_cursor* cs[PVS_GROUP_MAX] = {nullptr};
    pvs_status s = pvs::cursor_open_group(ex->index, j.snap, j.queries + (size_t)first * dim,
                                          count, j.on_device, st, nullptr, cs);
    if (s != PVS_OK) {   // e.g. one non-finite query: the others go on alone
        for (int32_t i = 0; i < count; ++i)
            j.status[first + i] = serve_one(ex, j, st, first + i, nullptr, 0);
        return;
    }
    int32_t got[PVS_GROUP_MAX] = {0};
    int32_t n_out[PVS_GROUP_MAX] = {0};
    int64_t* id_rows[PVS_GROUP_MAX];
    float* sc_rows[PVS_GROUP_MAX];
    int64_t pages = 0;
    int32_t total = 0;
    bool batch_ok = true;
    while (total < j.ranks) {
        const int32_t n = std::min(j.page, j.ranks - total);
        for (int32_t i = 0; i < count; ++i) {
            id_rows[i] = j.ids + (size_t)(first + i) * j.ranks + got[i];
            sc_rows[i] = j.scores + (size_t)(first + i) * j.ranks + got[i];
        }
        s = pvs::next_batch_rows(cs, count, n, j.on_device, id_rows, sc_rows, n_out);
        ++pages;
        if (s < 0) {
            batch_ok = false;
            break;
        }
        bool more = false;
        for (int32_t i = 0; i < count; ++i) {
            got[i] += n_out[i];
            more = more || n_out[i] == n;
        }
        total += n;
        if (!more) break;
    }
    int states[PVS_GROUP_MAX] = {0};
    if (batch_ok && pvs_cursor_sync_batch(cs, count, states) != PVS_OK)
        for (int32_t i = 0; i < count; ++i) states[i] = PVS_ERR_CUDA;
    count_passes(ex, cs, count, true);
    for (int32_t i = 0; i < count; ++i) {
        const int32_t r = first + i;
        if (!batch_ok) {
            pvs_stats st_i;
            const bool failed = pvs_cursor_stats(cs[i], &st_i) != PVS_OK || st_i.state < 0;
            if (failed) {
                fill_rest(j, st, r, got[i]);
                j.n_out[r] = got[i];
                j.status[r] = st_i.state < 0 ? (pvs_status)st_i.state : s;
                count_request(ex, (pvs_status)j.status[r], pages, got[i]);
                pvs_cursor_close(cs[i]);
            } else {   // continue this request on its own
                j.status[r] = serve_one(ex, j, st, r, cs[i], got[i]);
            }
            continue;
        }
        fill_rest(j, st, r, got[i]);
        j.n_out[r] = got[i];
        j.status[r] = states[i] < 0 ? (pvs_status)states[i]
                                    : (got[i] < j.ranks ? PVS_EXHAUSTED : PVS_OK);
        count_request(ex, (pvs_status)j.status[r], pages, got[i]);
        pvs_cursor_close(cs[i]);
    }
    if (j.on_device) cudaStreamSynchronize(st);
}

void worker_main(pvs_executor* ex, int w) {
    cudaSetDevice(ex->index->device);
    const cudaStream_t st = ex->streams[(size_t)w];
    uint64_t seen = 0;
    for (;;) {
        Job j;
        {
            std::unique_lock<std::mutex> lk(ex->m);
            ex->work_cv.wait(lk, [&] { return ex->stop || ex->generation != seen; });
            if (ex->stop) return;
            seen = ex->generation;
            j = ex->job;
        }
        const int32_t G = ex->group;
        for (;;) {
            const int32_t i = ex->next.fetch_add(G, std::memory_order_relaxed);
            if (i >= j.nq) break;
            const int32_t count = std::min(G, j.nq - i);
            if (count == 1)
                j.status[i] = serve_one(ex, j, st, i, nullptr, 0);
            else
                serve_group(ex, j, st, i, count);
        }
        std::lock_guard<std::mutex> lk(ex->m);
        if (--ex->busy == 0) ex->done_cv.notify_all();
    }
}

void shutdown(pvs_executor* ex) {
    {
        std::lock_guard<std::mutex> lk(ex->m);
        ex->stop = true;
    }
    ex->work_cv.notify_all();
    for (auto& t : ex->threads)
        if (t.joinable()) t.join();
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(ex->index->device);
    for (cudaStream_t s : ex->streams) cudaStreamDestroy(s);
    if (prev >= 0) cudaSetDevice(prev);
}

}  // namespace

extern "C" {

pvs_status pvs_executor_create(pvs_index* index, int32_t workers, pvs_executor** out) {
    if (!out) return PVS_ERR_INVALID;
    *out = nullptr;
    if (!index || workers < 1 || workers > kMaxWorkers) return PVS_ERR_INVALID;
    pvs_executor* ex = new (std::nothrow) pvs_executor();
    if (!ex) return PVS_ERR_OOM;
    ex->index = index;
    int prev = -1;
    cudaGetDevice(&prev);
    cudaError_t e = cudaSetDevice(index->device);
    for (int32_t w = 0; w < workers && e == cudaSuccess; ++w) {
        cudaStream_t s = nullptr;
        e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
        if (e == cudaSuccess) ex->streams.push_back(s);
    }
    if (prev >= 0) cudaSetDevice(prev);
    if (e != cudaSuccess) {
        cudaGetLastError();
        shutdown(ex);
        delete ex;
        return PVS_ERR_CUDA;
    }
    try {
        for (int32_t w = 0; w < workers; ++w) ex->threads.emplace_back(worker_main, ex, (int)w);
    } catch (...) {
        shutdown(ex);
        delete ex;
        return PVS_ERR_OOM;
    }
    *out = ex;
    return PVS_OK;
}

pvs_status pvs_executor_set_group(pvs_executor* ex, int32_t group) {
    if (!ex || group < 1 || group > PVS_GROUP_MAX) return PVS_ERR_INVALID;
    std::lock_guard<std::mutex> run(ex->run_mutex);   // not during a run
    ex->group = group;
    return PVS_OK;
}

pvs_status pvs_executor_run(pvs_executor* ex, const pvs_snapshot* snap, const float* queries,
                            int32_t nq, int32_t ranks, int32_t page, int64_t* ids, float* scores,
                            int32_t* n_out, int32_t* status) {
    return pvs_executor_run_ex(ex, snap, queries, nq, ranks, page, 0, ids, scores, n_out, status);
}

pvs_status pvs_executor_run_ex(pvs_executor* ex, const pvs_snapshot* snap, const float* queries,
                               int32_t nq, int32_t ranks, int32_t page, int32_t buffers_on_device,
                               int64_t* ids, float* scores, int32_t* n_out, int32_t* status) {
    if (!ex || nq < 0 || ranks < 1 || page < 1 || page > ranks) return PVS_ERR_INVALID;
    if (snap && snap->index != ex->index) return PVS_ERR_INVALID;
    if (nq == 0) return PVS_OK;
    if (!queries || !ids || !scores || !n_out) return PVS_ERR_INVALID;
    std::vector<int32_t> own;
    if (!status) {
        own.assign((size_t)nq, 0);
        status = own.data();
    }
    std::lock_guard<std::mutex> run(ex->run_mutex);
    {
        std::lock_guard<std::mutex> lk(ex->m);
        ex->job = Job{snap, queries, nq, ranks, page, buffers_on_device ? 1 : 0, ids, scores,
                      n_out, status};
        ex->next.store(0, std::memory_order_relaxed);
        ex->busy = (int)ex->threads.size();
        ++ex->generation;
    }
    ex->work_cv.notify_all();
    {
        std::unique_lock<std::mutex> lk(ex->m);
        ex->done_cv.wait(lk, [&] { return ex->busy == 0; });
    }
    for (int32_t i = 0; i < nq; ++i)
        if (status[i] < 0) return (pvs_status)status[i];
    return PVS_OK;
}

pvs_status pvs_executor_stats_get(pvs_executor* ex, pvs_executor_stats* out) {
    if (!ex || !out) return PVS_ERR_INVALID;
    out->requests = ex->requests.load();
    out->failed = ex->failed.load();
    out->pages = ex->pages.load();
    out->ranks = ex->ranks.load();
    out->workers = (int32_t)ex->threads.size();
    out->group = ex->group;
    out->interval_passes = ex->passes.load();
    out->refined = ex->refined.load();
    {
        std::lock_guard<std::mutex> lk(ex->ms_mutex);
        out->interval_ms = ex->interval_ms;
    }
    return PVS_OK;
}

void pvs_executor_destroy(pvs_executor* ex) {
    if (!ex) return;
    {
        std::lock_guard<std::mutex> run(ex->run_mutex);   // after a run in progress
    }
    shutdown(ex);
    delete ex;
}

}  // extern "C"
