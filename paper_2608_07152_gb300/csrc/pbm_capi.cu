// C ABI of the PBM sparse rank generator (include/pbm.h): arXiv 2608.07152
// Sec. 2.3.2 and App. A.2; ranked-list contract of Sec. 2.1.
//
// The ranges' keys key(H(R), first id of R) are sorted once, descending, at
// open, and ranges are expanded in that order.  A pull repeats two device
// steps until the next ranks are certified:
//   1. K = the key of the first unexpanded range in that order (the largest
//      unexpanded key), and the number of scored items in the pool with
//      K < key < (last key emitted): those items precede every unexpanded
//      item, so they are the next ranks;
//   2. if fewer than asked are certified and ranges remain, expand the next E
//      ranges (E doubles every round and carries over between pulls).
// The certified items are then emitted in key order.  The pool is
// append-only: emission runs in strictly decreasing key order, so the items
// not yet emitted are exactly the pool keys below the last emitted key.
//
// The ranked list is the support U_s = {x : S(x) > 0} (Sec. 2.1), minus the
// items a snapshot deletes.  A range with H(R) = 0 holds no item of U_s
// (S <= H), so only the ranges with H > 0 -- a prefix of the sorted order --
// are ever expanded; zero-score and deleted items of an expanded range enter
// the pool with key 0, which no window takes.  The list is Exhausted once
// every range with H > 0 is expanded and the window below the last emitted
// key has been delivered.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include <cuda_runtime.h>

#include "../../include/pbm.h"
#include "kernels.h"
#include "pbm_kernels.h"
#include "pvs_common.cuh"
#include "runtime.h"

namespace {

constexpr int kDefaultBlock = 128;
constexpr uint64_t kCollectCap = 65536;   // smallest gather buffer (keys)

pvs_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return PVS_OK;
    if (e == cudaErrorMemoryAllocation) {
        cudaGetLastError();
        return PVS_ERR_OOM;
    }
    return PVS_ERR_CUDA;
}

#define PBM_CUDA(x)                                      \
    do {                                                 \
        cudaError_t _e = (x);                            \
        if (_e != cudaSuccess) return cuda_status(_e);   \
    } while (0)

template <typename T>
cudaError_t dalloc(T** p, size_t count) {
    *p = nullptr;
    return cudaMalloc(reinterpret_cast<void**>(p), (count ? count : 1) * sizeof(T));
}

template <typename T>
void dfree(T*& p) {
    if (p) cudaFree(p);
    p = nullptr;
}

struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        int cur = -1;
        if (dev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != dev &&
            cudaSetDevice(dev) == cudaSuccess)
            prev = cur;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

}  // namespace

struct pbm_index {
    int device = 0;
    int num_sms = 0;
    cudaStream_t stream = nullptr;
    bool own_stream = false;
    int64_t n_items = 0, n_postings = 0, nb = 0, n_ranges = 0, nchunk = 0;
    int32_t n_terms = 0;
    int block = kDefaultBlock;
    int64_t* term_off = nullptr;    // [n_terms + 1]
    int32_t* docs = nullptr;        // [n_postings]
    float* imps = nullptr;          // [n_postings]
    int32_t* blk_range = nullptr;   // [nb]
    int64_t* blk_pbeg = nullptr;    // [nb + 1]
    float* blk_max = nullptr;       // [nb]
    int64_t* blk_off = nullptr;     // [n_terms + 1]
    // closed cursors keep their device and pinned buffers here for the next
    // open (allocating them per query cost a cudaMalloc of n_items keys and a
    // cudaFree, which waits for the whole device)
    std::vector<pbm_cursor*> cursor_pool;
    std::mutex pool_mutex;
};

struct pbm_cursor {
    pbm_index* index = nullptr;
    cudaStream_t stream = nullptr;
    int nq = 0;
    int nq_cap = 0;                   // capacity of terms, weights, starts
    int32_t* terms = nullptr;
    float* weights = nullptr;
    int64_t* starts = nullptr;        // [nq][nchunk + 1]
    float* H = nullptr;               // [n_ranges], as computed at open
    uint64_t* rkeys = nullptr;        // [n_ranges] range keys, sorted descending at open
    uint64_t* pool = nullptr;         // [n_items] rank keys of scored items
    pvs::PbmCounters* ctr = nullptr;  // device
    pvs::PbmCounters* h_ctr = nullptr;   // pinned mirror
    unsigned long long* sel64 = nullptr;   // [258]
    uint64_t* buf = nullptr;          // gathered keys
    uint64_t* tmp = nullptr;
    size_t buf_cap = 0;
    void* sort_scratch = nullptr;
    int64_t* out_ids = nullptr;
    float* out_scores = nullptr;
    int64_t* h_ids = nullptr;         // pinned: the sorted window of the last pull served by
    float* h_scores = nullptr;        // the finish kernel
    // entries [ahead_pos, ahead_len) of that window are certified ranks not
    // yet delivered: the next ranks in order (their keys exceed the bound of
    // every range not expanded when the window was taken, and the window held
    // every scored item above that bound), served without device work
    int64_t ahead_pos = 0, ahead_len = 0;
    bool ahead_complete = false;      // that window held every remaining rank
    uint64_t last_key = ~0ull;
    int64_t n_pos = 0;                // ranges with H > 0: the only ones expanded
    std::shared_ptr<pvs::SnapData> snap;   // visible set (null: every item)
    int64_t next = 0;                 // ranges expanded (a prefix of the sorted order)
    uint64_t E = 64;                  // ranges to expand in the next round
    int64_t emitted = 0, pulls = 0, rounds = 0;
    int64_t served_ahead = 0;         // pulls served from the window without device work
    int state = PVS_OK;
};

namespace {

pvs_status fail(pbm_cursor* c, pvs_status s) {
    if (s < 0 && c->state >= 0) c->state = s;
    return s;
}

constexpr size_t kPbmCursorPool = 32;

void free_cursor(pbm_cursor* c) {
    if (!c) return;
    dfree(c->terms);
    dfree(c->weights);
    dfree(c->starts);
    dfree(c->H);
    dfree(c->rkeys);
    dfree(c->pool);
    dfree(c->ctr);
    if (c->h_ctr) cudaFreeHost(c->h_ctr);
    dfree(c->sel64);
    dfree(c->buf);
    dfree(c->tmp);
    if (c->sort_scratch) cudaFree(c->sort_scratch);
    dfree(c->out_ids);
    dfree(c->out_scores);
    if (c->h_ids) cudaFreeHost(c->h_ids);
    if (c->h_scores) cudaFreeHost(c->h_scores);
    delete c;
}

// Gather / sort buffers for at least `count` keys.
pvs_status ensure_buffers(pbm_cursor* c, uint64_t count) {
    const uint64_t need = std::max<uint64_t>(count, kCollectCap);
    if (c->buf_cap >= need) return PVS_OK;
    dfree(c->buf);
    dfree(c->tmp);
    if (c->sort_scratch) cudaFree(c->sort_scratch);
    c->sort_scratch = nullptr;
    dfree(c->out_ids);
    dfree(c->out_scores);
    c->buf_cap = 0;
    PBM_CUDA(dalloc(&c->buf, need));
    PBM_CUDA(dalloc(&c->tmp, need));
    PBM_CUDA(cudaMalloc(&c->sort_scratch, pvs::radix_sort_scratch_bytes((int64_t)need)));
    PBM_CUDA(dalloc(&c->out_ids, need));
    PBM_CUDA(dalloc(&c->out_scores, need));
    c->buf_cap = need;
    return PVS_OK;
}

pvs_status sort_desc(pbm_cursor* c, uint64_t count) {
    if (count <= 1) return PVS_OK;
    if (count <= (uint64_t)pvs::kBitonicMax)
        PBM_CUDA(pvs::launch_bitonic_desc(c->buf, (int)count, c->stream));
    else
        PBM_CUDA(pvs::launch_radix_sort_desc(c->buf, c->tmp, (int64_t)count, c->sort_scratch,
                                             c->stream));
    return PVS_OK;
}

pvs_status read_counters(pbm_cursor* c) {
    PBM_CUDA(cudaMemcpyAsync(c->h_ctr, c->ctr, sizeof(pvs::PbmCounters), cudaMemcpyDeviceToHost,
                             c->stream));
    PBM_CUDA(cudaStreamSynchronize(c->stream));
    if (c->h_ctr->status != 0) return (pvs_status)c->h_ctr->status;
    return PVS_OK;
}

}  // namespace

extern "C" {

pvs_status pbm_build(const int64_t* term_off, int32_t n_terms, const int32_t* docs,
                     const float* imps, int64_t n_postings, int64_t n_items, int32_t block,
                     int32_t on_device, void* cuda_stream, pbm_index** out) {
    if (!out) return PVS_ERR_INVALID;
    *out = nullptr;
    if (block == 0) block = kDefaultBlock;
    if (n_terms < 0 || n_items < 1 || n_items >= ((int64_t)1 << 31) || n_postings < 0 ||
        n_postings >= ((int64_t)1 << 32) - 1 || block < 1 || block > pvs::kPbmMaxBlock ||
        !term_off || (n_postings > 0 && (!docs || !imps)))
        return PVS_ERR_INVALID;
    // the offsets are small: check them on the host
    std::vector<int64_t> off((size_t)n_terms + 1);
    if (on_device) {
        if (cudaMemcpy(off.data(), term_off, off.size() * sizeof(int64_t),
                       cudaMemcpyDeviceToHost) != cudaSuccess)
            return PVS_ERR_CUDA;
    } else {
        std::memcpy(off.data(), term_off, off.size() * sizeof(int64_t));
    }
    if (off[0] != 0 || off[(size_t)n_terms] != n_postings) return PVS_ERR_INVALID;
    for (int32_t t = 0; t < n_terms; ++t)
        if (off[(size_t)t + 1] < off[(size_t)t]) return PVS_ERR_INVALID;

    pbm_index* x = new (std::nothrow) pbm_index();
    if (!x) return PVS_ERR_OOM;
    auto bail = [&](pvs_status s) {
        pbm_index_free(x);
        return s;
    };
    if (cudaGetDevice(&x->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&x->num_sms, cudaDevAttrMultiProcessorCount, x->device) !=
            cudaSuccess)
        return bail(PVS_ERR_CUDA);
    if (cuda_stream) {
        x->stream = static_cast<cudaStream_t>(cuda_stream);
    } else {
        if (cudaStreamCreateWithFlags(&x->stream, cudaStreamNonBlocking) != cudaSuccess)
            return bail(PVS_ERR_CUDA);
        x->own_stream = true;
    }
    x->n_items = n_items;
    x->n_terms = n_terms;
    x->n_postings = n_postings;
    x->block = block;
    x->n_ranges = (n_items + block - 1) / block;
    x->nchunk = (x->n_ranges + pvs::kPbmChunk - 1) / pvs::kPbmChunk;
    cudaStream_t st = x->stream;
    const cudaMemcpyKind kind = on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    if (dalloc(&x->term_off, off.size()) != cudaSuccess ||
        dalloc(&x->docs, (size_t)n_postings) != cudaSuccess ||
        dalloc(&x->imps, (size_t)n_postings) != cudaSuccess ||
        dalloc(&x->blk_off, (size_t)n_terms + 1) != cudaSuccess)
        return bail(PVS_ERR_OOM);
    if (cudaMemcpyAsync(x->term_off, off.data(), off.size() * sizeof(int64_t),
                        cudaMemcpyHostToDevice, st) != cudaSuccess ||
        (n_postings > 0 &&
         (cudaMemcpyAsync(x->docs, docs, (size_t)n_postings * sizeof(int32_t), kind, st) !=
              cudaSuccess ||
          cudaMemcpyAsync(x->imps, imps, (size_t)n_postings * sizeof(float), kind, st) !=
              cudaSuccess)))
        return bail(PVS_ERR_CUDA);

    // blocks: starts marked and counted, then written once their number is known
    uint8_t* flags = nullptr;
    unsigned int* scratch = nullptr;
    int* status = nullptr;
    unsigned long long* nb_dev = nullptr;
    auto free_tmp = [&]() {
        dfree(flags);
        dfree(scratch);
        dfree(status);
        dfree(nb_dev);
    };
    auto bail2 = [&](pvs_status s) {
        free_tmp();
        return bail(s);
    };
    if (dalloc(&flags, (size_t)n_postings) != cudaSuccess ||
        dalloc(&scratch, pvs::pbm_scan_scratch_elems(n_postings)) != cudaSuccess ||
        dalloc(&status, 1) != cudaSuccess || dalloc(&nb_dev, 1) != cudaSuccess)
        return bail2(PVS_ERR_OOM);
    if (cudaMemsetAsync(status, 0, sizeof(int), st) != cudaSuccess ||
        pvs::launch_pbm_mark(x->term_off, n_terms, x->docs, x->imps, n_postings, n_items, block,
                             flags, status, st) != cudaSuccess ||
        pvs::launch_pbm_count_blocks(flags, n_postings, scratch, nb_dev, st) != cudaSuccess)
        return bail2(PVS_ERR_CUDA);
    int h_status = 0;
    unsigned long long h_nb = 0;
    if (cudaMemcpyAsync(&h_status, status, sizeof(int), cudaMemcpyDeviceToHost, st) !=
            cudaSuccess ||
        cudaMemcpyAsync(&h_nb, nb_dev, sizeof(h_nb), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return bail2(PVS_ERR_CUDA);
    if (h_status != 0) return bail2((pvs_status)h_status);
    x->nb = (int64_t)h_nb;
    if (dalloc(&x->blk_range, (size_t)x->nb) != cudaSuccess ||
        dalloc(&x->blk_pbeg, (size_t)x->nb + 1) != cudaSuccess ||
        dalloc(&x->blk_max, (size_t)x->nb) != cudaSuccess)
        return bail2(PVS_ERR_OOM);
    const int64_t p_end = n_postings;
    if (pvs::launch_pbm_write_blocks(flags, x->docs, n_postings, block, scratch, x->blk_range,
                                     x->blk_pbeg, st) != cudaSuccess ||
        cudaMemcpyAsync(x->blk_pbeg + x->nb, &p_end, sizeof(int64_t), cudaMemcpyHostToDevice,
                        st) != cudaSuccess ||
        pvs::launch_pbm_block_max(x->blk_pbeg, x->imps, x->nb, x->blk_max, st) != cudaSuccess ||
        pvs::launch_pbm_term_blocks(x->term_off, n_terms, x->blk_pbeg, x->nb, x->blk_off, st) !=
            cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)
        return bail2(PVS_ERR_CUDA);
    free_tmp();
    *out = x;
    return PVS_OK;
}

int64_t pbm_index_items(const pbm_index* x) { return x ? x->n_items : 0; }
int64_t pbm_index_ranges(const pbm_index* x) { return x ? x->n_ranges : 0; }

void pbm_index_free(pbm_index* x) {
    if (!x) return;
    DeviceGuard device_guard(x->device);
    if (x->stream) cudaStreamSynchronize(x->stream);
    for (pbm_cursor* c : x->cursor_pool) free_cursor(c);
    x->cursor_pool.clear();
    dfree(x->term_off);
    dfree(x->docs);
    dfree(x->imps);
    dfree(x->blk_range);
    dfree(x->blk_pbeg);
    dfree(x->blk_max);
    dfree(x->blk_off);
    if (x->own_stream && x->stream) cudaStreamDestroy(x->stream);
    delete x;
}

}  // extern "C"

namespace {

pvs_status open_cursor(pbm_index* x, const std::shared_ptr<pvs::SnapData>& snap,
                       const int32_t* terms, const float* weights, int32_t nq,
                       cudaStream_t stream, pbm_cursor** out) {
    if (!out) return PVS_ERR_INVALID;
    *out = nullptr;
    if (!x || nq < 0 || nq > pvs::kPbmMaxTerms || (nq > 0 && (!terms || !weights)))
        return PVS_ERR_INVALID;
    if (snap && snap->rows != x->n_items) return PVS_ERR_INVALID;
    DeviceGuard device_guard(x->device);
    std::vector<int32_t> sorted(terms, terms + nq);
    std::sort(sorted.begin(), sorted.end());
    for (int i = 0; i < nq; ++i) {
        if (sorted[i] < 0 || sorted[i] >= x->n_terms) return PVS_ERR_INVALID;
        if (i > 0 && sorted[i] == sorted[i - 1]) return PVS_ERR_INVALID;   // Q is a set
    }
    for (int i = 0; i < nq; ++i) {
        if (!std::isfinite(weights[i])) return PVS_ERR_NONFINITE;
        if (weights[i] < 0.0f) return PVS_ERR_INVALID;
    }
    pbm_cursor* c = nullptr;
    {
        std::lock_guard<std::mutex> lock(x->pool_mutex);
        if (!x->cursor_pool.empty()) {
            c = x->cursor_pool.back();
            x->cursor_pool.pop_back();
        }
    }
    if (!c) c = new (std::nothrow) pbm_cursor();
    if (!c) return PVS_ERR_OOM;
    // the state of a fresh cursor; buffers of a pooled one are kept
    c->index = x;
    c->stream = stream ? stream : x->stream;
    c->nq = nq;
    c->snap.reset();
    if (snap && snap->d_tomb) c->snap = snap;   // deletions apply
    c->ahead_pos = c->ahead_len = 0;
    c->ahead_complete = false;
    c->last_key = ~0ull;
    c->n_pos = 0;
    c->next = 0;
    c->E = 64;
    c->emitted = c->pulls = c->rounds = c->served_ahead = 0;
    c->state = PVS_OK;
    auto bail = [&](pvs_status s) {
        free_cursor(c);
        return s;
    };
    if (nq > c->nq_cap) {
        dfree(c->terms);
        dfree(c->weights);
        dfree(c->starts);
        c->nq_cap = 0;
        const int cap = std::max(nq, 16);
        if (dalloc(&c->terms, (size_t)cap) != cudaSuccess ||
            dalloc(&c->weights, (size_t)cap) != cudaSuccess ||
            dalloc(&c->starts, (size_t)cap * (size_t)(x->nchunk + 1)) != cudaSuccess)
            return bail(PVS_ERR_OOM);
        c->nq_cap = cap;
    }
    if ((!c->H && dalloc(&c->H, (size_t)x->n_ranges) != cudaSuccess) ||
        (!c->rkeys && dalloc(&c->rkeys, (size_t)x->n_ranges) != cudaSuccess) ||
        (!c->pool && dalloc(&c->pool, (size_t)x->n_items) != cudaSuccess) ||
        (!c->ctr && dalloc(&c->ctr, 1) != cudaSuccess) ||
        (!c->sel64 && dalloc(&c->sel64, 258) != cudaSuccess) ||
        (!c->h_ctr && cudaMallocHost(reinterpret_cast<void**>(&c->h_ctr),
                                     sizeof(pvs::PbmCounters)) != cudaSuccess) ||
        (!c->h_ids && cudaMallocHost(reinterpret_cast<void**>(&c->h_ids),
                                     pvs::kPbmFastWindow * sizeof(int64_t)) != cudaSuccess) ||
        (!c->h_scores && cudaMallocHost(reinterpret_cast<void**>(&c->h_scores),
                                        pvs::kPbmFastWindow * sizeof(float)) != cudaSuccess))
        return bail(PVS_ERR_OOM);
    std::memset(c->h_ctr, 0, sizeof(pvs::PbmCounters));
    cudaStream_t st = c->stream;
    const pvs::PbmQuery q{c->terms, c->weights, nq};
    if ((nq > 0 &&
         (cudaMemcpyAsync(c->terms, terms, (size_t)nq * sizeof(int32_t), cudaMemcpyHostToDevice,
                          st) != cudaSuccess ||
          cudaMemcpyAsync(c->weights, weights, (size_t)nq * sizeof(float),
                          cudaMemcpyHostToDevice, st) != cudaSuccess)) ||
        cudaMemsetAsync(c->ctr, 0, sizeof(pvs::PbmCounters), st) != cudaSuccess ||
        pvs::launch_pbm_starts(q, x->blk_off, x->blk_range, x->nchunk, c->starts, st) !=
            cudaSuccess ||
        pvs::launch_pbm_bounds(q, c->starts, x->blk_range, x->blk_max, x->n_ranges, x->nchunk,
                               c->H, &c->ctr->status, &c->ctr->pos_ranges, st) != cudaSuccess ||
        pvs::launch_pbm_range_keys(c->H, x->n_ranges, x->block, c->rkeys, st) != cudaSuccess)
        return bail(PVS_ERR_CUDA);
    // the expansion order: range keys sorted descending (the sort's scratch is
    // the gather buffers, sized for at least n_ranges keys)
    if (ensure_buffers(c, (uint64_t)x->n_ranges) != PVS_OK) return bail(PVS_ERR_OOM);
    if (x->n_ranges > 1 &&
        ((uint64_t)x->n_ranges <= (uint64_t)pvs::kBitonicMax
             ? pvs::launch_bitonic_desc(c->rkeys, (int)x->n_ranges, st)
             : pvs::launch_radix_sort_desc(c->rkeys, c->tmp, x->n_ranges, c->sort_scratch, st)) !=
            cudaSuccess)
        return bail(PVS_ERR_CUDA);
    if (cudaMemcpyAsync(c->h_ctr, c->ctr, sizeof(pvs::PbmCounters), cudaMemcpyDeviceToHost,
                        st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess)   // query copies, the count of ranges
        return bail(PVS_ERR_CUDA);
    c->n_pos = (int64_t)c->h_ctr->pos_ranges;
    *out = c;
    return PVS_OK;
}

}  // namespace

namespace pvs {
const SnapData* pbm_cursor_snapshot(const pbm_cursor* c) { return c->snap.get(); }

// The complete sparse ranking of the cursor's query as a staged list: every
// item's S in the query's term order (the expand kernel's evaluation), the
// visible items with S > 0 sorted by key, their positions scattered into
// rank_of.  Runs on a stream of its own and waits for it once (for the
// member count), so the caller may be a helper thread.
pvs_status pbm_stage_ranks(pbm_cursor* c, pvs_index* owner, StagedList** out) {
    *out = nullptr;
    if (!c || !c->index || !owner || c->state < 0) return PVS_ERR_INVALID;
    pbm_index* x = c->index;
    if (cudaSetDevice(x->device) != cudaSuccess) {
        cudaGetLastError();
        return PVS_ERR_CUDA;
    }
    StagedList* s = new (std::nothrow) StagedList();
    if (!s) return PVS_ERR_OOM;
    s->index = owner;
    s->rows = x->n_items;
    const size_t n = (size_t)std::max<int64_t>(x->n_items, 1);
    const uint32_t* tomb = c->snap ? c->snap->d_tomb : nullptr;
    float* acc = nullptr;
    uint64_t* keys = nullptr;
    uint64_t* tmp = nullptr;
    void* scratch = nullptr;
    unsigned long long* count = nullptr;
    unsigned long long* h_count = nullptr;
    cudaError_t e = cudaStreamCreateWithFlags(&s->stream, cudaStreamNonBlocking);
    auto pool_alloc = [&](void** p, size_t bytes) {
        if (e == cudaSuccess)
            e = cudaMallocFromPoolAsync(p, std::max<size_t>(bytes, 16), owner->scratch_pool,
                                        s->stream);
    };
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&s->ready, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaMallocHost(&h_count, sizeof(unsigned long long));
    pool_alloc(reinterpret_cast<void**>(&s->rank_of), n * 4);
    pool_alloc(reinterpret_cast<void**>(&s->status), sizeof(int));
    pool_alloc(reinterpret_cast<void**>(&acc), n * 4);
    pool_alloc(reinterpret_cast<void**>(&keys), n * 8);
    pool_alloc(reinterpret_cast<void**>(&count), sizeof(unsigned long long));
    const int grid = std::max(1, x->num_sms) * 8;
    if (e == cudaSuccess) e = cudaMemsetAsync(s->rank_of, 0, n * 4, s->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(s->status, 0, sizeof(int), s->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(acc, 0, n * 4, s->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(count, 0, sizeof(unsigned long long), s->stream);
    if (e == cudaSuccess)
        e = launch_pbm_score_all(PbmQuery{c->terms, c->weights, c->nq}, x->term_off, x->docs,
                                 x->imps, acc, grid, s->stream);
    if (e == cudaSuccess)
        e = launch_pbm_member_keys(acc, x->n_items, tomb, keys, count, grid, s->stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h_count, count, sizeof(unsigned long long), cudaMemcpyDeviceToHost,
                            s->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s->stream);
    const int64_t m = e == cudaSuccess ? (int64_t)*h_count : 0;
    if (m > 1) {
        pool_alloc(reinterpret_cast<void**>(&tmp), (size_t)m * 8);
        pool_alloc(&scratch, radix_sort_scratch_bytes(m));
        if (e == cudaSuccess) e = launch_radix_sort_desc(keys, tmp, m, scratch, s->stream);
    }
    if (e == cudaSuccess) e = launch_pbm_rank_of(keys, m, s->rank_of, grid, s->stream);
    if (e == cudaSuccess) e = cudaEventRecord(s->ready, s->stream);
    for (void* p : {(void*)acc, (void*)keys, (void*)tmp, scratch, (void*)count})
        if (p) cudaFreeAsync(p, s->stream);
    if (h_count) cudaFreeHost(h_count);
    if (e != cudaSuccess) {
        cudaGetLastError();
        free_staged_list(s);
        return e == cudaErrorMemoryAllocation ? PVS_ERR_OOM : PVS_ERR_CUDA;
    }
    *out = s;
    return PVS_OK;
}
}  // namespace pvs

extern "C" {

pvs_status pbm_cursor_open(pbm_index* x, const int32_t* terms, const float* weights, int32_t nq,
                           pbm_cursor** out) {
    return open_cursor(x, nullptr, terms, weights, nq, nullptr, out);
}

pvs_status pbm_cursor_open_snapshot(pbm_index* x, const pvs_snapshot* snap, const int32_t* terms,
                                    const float* weights, int32_t nq, pbm_cursor** out) {
    return pbm_cursor_open_stream(x, snap, terms, weights, nq, nullptr, out);
}

pvs_status pbm_cursor_open_stream(pbm_index* x, const pvs_snapshot* snap, const int32_t* terms,
                                  const float* weights, int32_t nq, void* cuda_stream,
                                  pbm_cursor** out) {
    if (out) *out = nullptr;
    if (snap && (!x || !snap->index || snap->index->device != x->device)) return PVS_ERR_INVALID;
    return open_cursor(x, snap ? snap->data : nullptr, terms, weights, nq,
                       static_cast<cudaStream_t>(cuda_stream), out);
}

pvs_status pbm_next(pbm_cursor* c, int32_t n, int64_t* ids, float* scores, int32_t* n_out) {
    if (n_out) *n_out = 0;
    if (!c) return PVS_ERR_INVALID;
    if (c->state < 0) return PVS_ERR_FAILED;
    if (n < 1 || !ids || !scores || !n_out) return PVS_ERR_INVALID;
    if (c->state == PVS_EXHAUSTED) return PVS_EXHAUSTED;
    pbm_index* x = c->index;
    DeviceGuard device_guard(x->device);
    cudaStream_t st = c->stream;
    ++c->pulls;
    const uint64_t need = (uint64_t)std::min<int64_t>(n, x->n_items - c->emitted);
    if (need == 0) {   // every item was delivered: the support is the whole id space
        c->state = PVS_EXHAUSTED;
        return PVS_EXHAUSTED;
    }
    const uint64_t avail = (uint64_t)(c->ahead_len - c->ahead_pos);
    if (need > 0 && (avail >= need || (c->ahead_complete && avail > 0))) {
        // certified ranks already here (all that remain, when the window was complete)
        const uint64_t m = std::min(need, avail);
        std::memcpy(ids, c->h_ids + c->ahead_pos, m * sizeof(int64_t));
        std::memcpy(scores, c->h_scores + c->ahead_pos, m * sizeof(float));
        c->ahead_pos += (int64_t)m;
        c->last_key = pvs::rank_key(scores[m - 1], (uint32_t)ids[m - 1]);
        c->emitted += (int64_t)m;
        ++c->served_ahead;
        *n_out = (int32_t)m;
        if (c->ahead_complete && c->ahead_pos == c->ahead_len) {
            c->state = PVS_EXHAUSTED;
            return PVS_EXHAUSTED;
        }
        return PVS_OK;
    }
    // too few: the device gathers them again (they lie below last_key)
    c->ahead_pos = c->ahead_len = 0;
    c->ahead_complete = false;
    uint64_t E = std::max<uint64_t>(c->E, 2 * ((need + x->block - 1) / x->block));
    uint64_t window = 0;
    uint64_t last = 0;   // size of the last expansion of this pull
    bool served = false, complete = false;
    for (;;) {
        // the certified window, gathered; a window of at most kPbmFastWindow
        // keys that covers the pull (or holds every remaining rank) is sorted
        // and written to pinned memory in the same step (one synchronisation)
        complete = c->next >= c->n_pos;
        cudaError_t e = pvs::launch_pbm_window(c->rkeys, c->next, c->n_pos, c->pool, c->last_key,
                                               c->buf, c->buf_cap, c->ctr, st);
        if (e == cudaSuccess)
            e = pvs::launch_pbm_finish(c->buf, c->ctr, need, complete, c->h_ids, c->h_scores,
                                       c->h_ctr, st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(st);
        if (e != cudaSuccess) return fail(c, cuda_status(e));
        if (c->h_ctr->status != 0) return fail(c, (pvs_status)c->h_ctr->status);
        window = c->h_ctr->collected;
        if (window >= 1 && (window >= need || complete) &&
            window <= (uint64_t)pvs::kPbmFastWindow) {
            served = true;
            break;
        }
        if (window >= need || complete) break;
        // expand the next E ranges of the sorted order (ranges with H > 0 only)
        ++c->rounds;
        const uint64_t k = std::min(E, (uint64_t)(c->n_pos - c->next));
        pvs::PbmExpandArgs a{};
        a.ranges = c->rkeys + c->next;
        a.count = (int64_t)k;
        a.q = pvs::PbmQuery{c->terms, c->weights, c->nq};
        a.starts = c->starts;
        a.nchunk = x->nchunk;
        a.blk_range = x->blk_range;
        a.blk_pbeg = x->blk_pbeg;
        a.docs = x->docs;
        a.imps = x->imps;
        a.n_items = x->n_items;
        a.block = x->block;
        a.tomb = c->snap ? c->snap->d_tomb : nullptr;
        a.pool = c->pool;
        a.ctr = c->ctr;
        e = pvs::launch_pbm_expand(a, (int)std::min<uint64_t>(k, (uint64_t)x->num_sms * 4), st);
        if (e != cudaSuccess) return fail(c, cuda_status(e));
        c->next += (int64_t)k;
        last = k;
        E *= 2;
    }
    // the next pull starts from the size of the expansion that last sufficed
    if (last) c->E = std::max<uint64_t>(16, last);
    const uint64_t m = std::min<uint64_t>(need, window);
    if (served) {
        std::memcpy(ids, c->h_ids, m * sizeof(int64_t));
        std::memcpy(scores, c->h_scores, m * sizeof(float));
        c->ahead_pos = (int64_t)m;
        c->ahead_len = (int64_t)window;
        c->ahead_complete = complete;
    } else if (m > 0) {
        // large window: the m-th largest key first (or the whole window when
        // it fits the gather buffer), then a device sort of the m keys
        pvs_status s = ensure_buffers(c, m);
        if (s != PVS_OK) return fail(c, s);
        cudaError_t e = pvs::launch_pbm_select64(c->pool, c->ctr, c->last_key, m, c->sel64, st);
        if (e == cudaSuccess)
            e = pvs::launch_pbm_collect(c->pool, c->sel64, c->last_key, c->buf, c->buf_cap, c->ctr,
                                        st);
        if (e != cudaSuccess) return fail(c, cuda_status(e));
        s = sort_desc(c, m);
        if (s != PVS_OK) return fail(c, s);
        if (pvs::launch_pbm_emit(c->buf, (int)m, c->out_ids, c->out_scores, st) != cudaSuccess ||
            cudaMemcpyAsync(ids, c->out_ids, m * sizeof(int64_t), cudaMemcpyDeviceToHost, st) !=
                cudaSuccess ||
            cudaMemcpyAsync(scores, c->out_scores, m * sizeof(float), cudaMemcpyDeviceToHost,
                            st) != cudaSuccess)
            return fail(c, PVS_ERR_CUDA);
        s = read_counters(c);   // also waits for the outputs
        if (s != PVS_OK) return fail(c, s);
        if (c->h_ctr->collected != m) return fail(c, PVS_ERR_INVALID);   // internal invariant
    }
    if (m > 0) {
        c->last_key = pvs::rank_key(scores[m - 1], (uint32_t)ids[m - 1]);
        c->emitted += (int64_t)m;
    }
    *n_out = (int32_t)m;
    // with every range of positive bound expanded, the window held every
    // remaining rank: delivering all of it ends the list
    if (complete && m == window) {
        c->state = PVS_EXHAUSTED;
        return PVS_EXHAUSTED;
    }
    return PVS_OK;
}

pvs_status pbm_cursor_range_bounds(pbm_cursor* c, int64_t first, int64_t count, float* H) {
    if (!c || !H || first < 0 || count < 0 || first + count > c->index->n_ranges)
        return PVS_ERR_INVALID;
    DeviceGuard device_guard(c->index->device);
    if (count == 0) return PVS_OK;
    PBM_CUDA(cudaMemcpyAsync(H, c->H + first, (size_t)count * sizeof(float),
                             cudaMemcpyDeviceToHost, c->stream));
    PBM_CUDA(cudaStreamSynchronize(c->stream));
    return c->state < 0 ? (pvs_status)c->state : PVS_OK;
}

pvs_status pbm_cursor_stats(pbm_cursor* c, pbm_stats* out) {
    if (!c || !out) return PVS_ERR_INVALID;
    DeviceGuard device_guard(c->index->device);
    pvs_status s = read_counters(c);
    if (s != PVS_OK && c->state >= 0) c->state = s;
    out->items = c->index->n_items;
    out->emitted = c->emitted;
    out->ranges = c->index->n_ranges;
    out->ranges_expanded = (int64_t)c->h_ctr->ranges_expanded;
    out->postings_visited = (int64_t)c->h_ctr->postings;
    out->items_scored = (int64_t)c->h_ctr->items;
    out->pulls = c->pulls;
    out->rounds = c->rounds;
    out->pulls_from_window = c->served_ahead;
    out->state = c->state;
    out->reserved = 0;
    return PVS_OK;
}

void pbm_cursor_close(pbm_cursor* c) {
    if (!c) return;
    DeviceGuard device_guard(c->index ? c->index->device : -1);
    if (c->stream) cudaStreamSynchronize(c->stream);
    pbm_index* x = c->index;
    if (x) {   // the buffers serve the next open
        c->snap.reset();
        std::lock_guard<std::mutex> lock(x->pool_mutex);
        if (x->cursor_pool.size() < kPbmCursorPool) {
            x->cursor_pool.push_back(c);
            return;
        }
    }
    free_cursor(c);
}

}  // extern "C"
