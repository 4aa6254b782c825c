// Native request executor (include/executor.h): arXiv 2608.07152 Sec. 2.1
// (ranked lists read page by page as a stable, only-extended prefix) over
// the PVS cursors of Sec. 2.3.
//
// A fixed pool of worker threads, each bound to the index's device with its
// own non-blocking stream.  A run publishes one job and bumps a generation
// counter; the workers take request indexes from an atomic counter.  For a
// request a worker opens the cursor on its own stream, reads the pages one
// after another through pvs_next straight into the request's rows of the
// caller's buffers, and closes the cursor.  No lock is held across a device
// wait; the job lock is taken only at the start and end of a run.
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
    std::atomic<int64_t> requests{0}, failed{0}, pages{0}, ranks{0};
};

namespace {

// One request: open, read the pages, close.  Returns the request's status.
pvs_status serve(pvs_executor* ex, const Job& j, cudaStream_t st, int32_t i) {
    const int32_t dim = ex->index->m;
    int64_t* ids = j.ids + (size_t)i * j.ranks;
    float* sc = j.scores + (size_t)i * j.ranks;
    int32_t total = 0;
    int64_t pages = 0;
    pvs_cursor* c = nullptr;
    pvs_status s = pvs::cursor_open_on(ex->index, j.snap, j.queries + (size_t)i * dim, 0, st, &c);
    if (s == PVS_OK && c) {
        while (total < j.ranks) {
            int32_t got = 0;
            s = pvs_next(c, std::min(j.page, j.ranks - total), ids + total, sc + total, &got);
            ++pages;
            if (s < 0) break;
            total += got;
            if (s == PVS_EXHAUSTED) break;
        }
    }
    if (c) pvs_cursor_close(c);
    for (int32_t k = total; k < j.ranks; ++k) {
        ids[k] = -1;
        sc[k] = NAN;
    }
    j.n_out[i] = total;
    ex->requests.fetch_add(1, std::memory_order_relaxed);
    if (s < 0) ex->failed.fetch_add(1, std::memory_order_relaxed);
    ex->pages.fetch_add(pages, std::memory_order_relaxed);
    ex->ranks.fetch_add(total, std::memory_order_relaxed);
    return s;
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
        for (;;) {
            const int32_t i = ex->next.fetch_add(1, std::memory_order_relaxed);
            if (i >= j.nq) break;
            j.status[i] = serve(ex, j, st, i);
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

pvs_status pvs_executor_run(pvs_executor* ex, const pvs_snapshot* snap, const float* queries,
                            int32_t nq, int32_t ranks, int32_t page, int64_t* ids, float* scores,
                            int32_t* n_out, int32_t* status) {
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
        ex->job = Job{snap, queries, nq, ranks, page, ids, scores, n_out, status};
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
    out->reserved = 0;
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
