// C ABI of libpvs.so: index build / append / tombstone, snapshots, cursors
// and the pull orchestration of PVS resumable exact ranking
// (arXiv 2608.07152, Sec. 2.1, 2.3.1, 2.4, App. A.1).
//
// Pull of n ranks (Sec. 2.3.1: candidates in decreasing interval upper
// bound, raw vectors read only where intervals do not decide):
//   1. first pull: one interval pass over the Int8 codes -> lo[i], hi[i];
//   2. working set W: tau_H = H-th largest lo among live rows, W = {live rows
//      with hi >= tau_H} in id order; W holds the next H ranks (every item
//      outside W is preceded by the >= H items with lo >= tau_H);
//   3. per pull: tau = n-th largest lo in W; candidates C = {hi >= tau}; score
//      the unresolved candidates exactly (lo = hi = s afterwards); C contains
//      the next n ranks, which are its n largest (score, -id) keys;
//   4. emit them in order and mark them emitted (lo = hi = -inf).
//   W is rebuilt with a doubled horizon when a pull would go past it.
#include <algorithm>
#include <cmath>
#include <atomic>
#include <chrono>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <thread>

#include "runtime.h"

using namespace pvs;

namespace pvs {

static std::atomic<long long> g_launches{0};
void count_launches(int k) { g_launches.fetch_add(k, std::memory_order_relaxed); }

SnapData::~SnapData() {
    if (d_tomb) cudaFree(d_tomb);
}

int64_t cursor_visible(const pvs_cursor* c) { return c->visible; }
int64_t cursor_emitted(const pvs_cursor* c) { return c->emitted - c->ahead; }
const SnapData* cursor_snapshot(const pvs_cursor* c) { return c->snap.get(); }

}  // namespace pvs

namespace {

constexpr size_t kStageBytes = size_t(1) << 30;   // host-input staging chunk

inline int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

pvs_status cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return PVS_OK;
    if (e == cudaErrorMemoryAllocation) {
        cudaGetLastError();
        return PVS_ERR_OOM;
    }
    return PVS_ERR_CUDA;
}

#define PVS_CUDA(x)                                      \
    do {                                                 \
        cudaError_t _e = (x);                            \
        if (_e != cudaSuccess) return cuda_status(_e);   \
    } while (0)

template <typename T>
cudaError_t dev_alloc(T** p, size_t count) {
    *p = nullptr;
    if (count == 0) count = 1;
    return cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T));
}

template <typename T>
void dev_free(T*& p) {
    if (p) cudaFree(p);
    p = nullptr;
}

bool is_device_ptr(const void* p) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

// Grow the index arrays to hold `need` rows.
pvs_status index_reserve(pvs_index* x, int64_t need) {
    if (need <= x->cap) return PVS_OK;
    int64_t cap = std::max<int64_t>(need, x->cap + x->cap / 2);
    cap = round_up(std::max<int64_t>(cap, 64), 64);
    int8_t* codes = nullptr;
    float *scale = nullptr, *vnorm = nullptr, *enorm = nullptr, *raw = nullptr;
    cudaError_t e = dev_alloc(&codes, (size_t)cap * x->m_pad);
    if (e == cudaSuccess) e = dev_alloc(&scale, (size_t)cap);
    if (e == cudaSuccess) e = dev_alloc(&vnorm, (size_t)cap);
    if (e == cudaSuccess) e = dev_alloc(&enorm, (size_t)cap);
    if (e == cudaSuccess) e = dev_alloc(&raw, (size_t)cap * x->m_raw);
    if (e == cudaSuccess) {
        // zero the tail so that tile copies past the last row read zeros
        e = cudaMemsetAsync(scale, 0, cap * sizeof(float), x->stream);
        if (e == cudaSuccess) e = cudaMemsetAsync(vnorm, 0, cap * sizeof(float), x->stream);
        if (e == cudaSuccess) e = cudaMemsetAsync(enorm, 0, cap * sizeof(float), x->stream);
    }
    if (e == cudaSuccess && x->size > 0) {
        e = cudaMemcpyAsync(codes, x->codes, (size_t)x->size * x->m_pad, cudaMemcpyDeviceToDevice,
                            x->stream);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(scale, x->scale, x->size * sizeof(float), cudaMemcpyDeviceToDevice,
                                x->stream);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(vnorm, x->vnorm, x->size * sizeof(float), cudaMemcpyDeviceToDevice,
                                x->stream);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(enorm, x->enorm, x->size * sizeof(float), cudaMemcpyDeviceToDevice,
                                x->stream);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(raw, x->raw, (size_t)x->size * x->m_raw * sizeof(float),
                                cudaMemcpyDeviceToDevice, x->stream);
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(x->stream);
    if (e != cudaSuccess) {
        dev_free(codes), dev_free(scale), dev_free(vnorm), dev_free(enorm), dev_free(raw);
        return cuda_status(e);
    }
    dev_free(x->codes), dev_free(x->scale), dev_free(x->vnorm), dev_free(x->enorm);
    dev_free(x->raw);
    dev_free(x->codes_bf16);   // rebuilt on demand at the new capacity
    x->bf16_rows = 0;
    dev_free(x->resid), dev_free(x->rparam);   // likewise
    x->resid_rows = 0;
    x->codes = codes, x->scale = scale, x->vnorm = vnorm, x->enorm = enorm, x->raw = raw;
    x->cap = cap;
    x->h_tomb.resize((size_t)(cap / 32), 0u);
    return PVS_OK;
}

// Quantize n rows into the index at row offset x->size (does not commit).
pvs_status index_fill(pvs_index* x, const float* vecs, int64_t n, bool on_device) {
    if (n == 0) return PVS_OK;
    PVS_CUDA(cudaMemsetAsync(x->d_status, 0, sizeof(int), x->stream));
    const int64_t row0 = x->size;
    if (on_device) {
        PVS_CUDA(launch_build(vecs, n, x->m, x->m_pad, x->m_raw, x->codes + row0 * x->m_pad,
                              x->scale + row0, x->vnorm + row0, x->enorm + row0,
                              x->raw + row0 * x->m_raw, x->d_status, x->stream, x->gscale));
    } else {
        const int64_t rows_per_chunk =
            std::max<int64_t>(1, (int64_t)(kStageBytes / sizeof(float)) / x->m);
        const int64_t chunk = std::min<int64_t>(rows_per_chunk, n);
        if (x->stage_floats < (size_t)(chunk * x->m)) {
            dev_free(x->d_stage);
            PVS_CUDA(dev_alloc(&x->d_stage, (size_t)(chunk * x->m)));
            x->stage_floats = (size_t)(chunk * x->m);
        }
        for (int64_t r = 0; r < n; r += chunk) {
            const int64_t c = std::min<int64_t>(chunk, n - r);
            PVS_CUDA(cudaMemcpyAsync(x->d_stage, vecs + r * x->m, (size_t)(c * x->m) * sizeof(float),
                                     cudaMemcpyHostToDevice, x->stream));
            const int64_t dr = row0 + r;
            PVS_CUDA(launch_build(x->d_stage, c, x->m, x->m_pad, x->m_raw,
                                  x->codes + dr * x->m_pad, x->scale + dr, x->vnorm + dr,
                                  x->enorm + dr, x->raw + dr * x->m_raw, x->d_status, x->stream,
                                  x->gscale));
        }
    }
    int st = 0;
    PVS_CUDA(cudaMemcpyAsync(&st, x->d_status, sizeof(int), cudaMemcpyDeviceToHost, x->stream));
    PVS_CUDA(cudaStreamSynchronize(x->stream));
    return (pvs_status)st;
}

// Corpus maxima of the norm bounds over rows [0, size); waits for them.
pvs_status refresh_norm_maxes(pvs_index* x) {
    if (!x->norm_maxes) PVS_CUDA(dev_alloc(&x->norm_maxes, 2));
    PVS_CUDA(launch_norm_max(x->vnorm, x->enorm, x->size, x->norm_maxes, x->stream));
    PVS_CUDA(cudaStreamSynchronize(x->stream));
    return PVS_OK;
}

std::shared_ptr<SnapData> make_snapdata(const pvs_index* x) {
    auto s = std::make_shared<SnapData>();
    s->rows = x->size;
    s->visible = x->live;
    if (x->tombstoned > 0) {
        const size_t words = (size_t)((x->size + 31) / 32);
        s->h_tomb.assign(x->h_tomb.begin(), x->h_tomb.begin() + words);
        if (cudaMalloc(&s->d_tomb, words * sizeof(uint32_t)) != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        if (cudaMemcpy(s->d_tomb, s->h_tomb.data(), words * sizeof(uint32_t),
                       cudaMemcpyHostToDevice) != cudaSuccess)
            return nullptr;
    }
    return s;
}

void cursor_free_device(pvs_cursor* c) {
    dev_free(c->zq), dev_free(c->qraw), dev_free(c->qs);
    dev_free(c->lo), dev_free(c->hi), dev_free(c->bmax);
    dev_free(c->w_id), dev_free(c->w_lo), dev_free(c->w_hi);
    dev_free(c->compact_scratch), dev_free(c->slot_top);
    c->slot_cap = 0;
    dev_free(c->cand), dev_free(c->keys), dev_free(c->keys_tmp), dev_free(c->front);
    if (c->sort_scratch) cudaFree(c->sort_scratch);
    c->sort_scratch = nullptr;
    dev_free(c->sel), dev_free(c->ctr), dev_free(c->d_status);
    dev_free(c->d_ids), dev_free(c->d_scores);
    if (c->h_ids) cudaFreeHost(c->h_ids);
    if (c->h_scores) cudaFreeHost(c->h_scores);
    if (c->h_small) cudaFreeHost(c->h_small);
    c->h_ids = nullptr, c->h_scores = nullptr, c->h_small = nullptr;
    if (c->rq_pinned) cudaFreeHost(c->rq_pinned);
    if (c->rq_stream) cudaStreamDestroy(c->rq_stream);
    if (c->rq_event) cudaEventDestroy(c->rq_event);
    c->rq_pinned = nullptr, c->rq_stream = nullptr, c->rq_event = nullptr;
    if (c->ev_begin) cudaEventDestroy(c->ev_begin);
    if (c->ev_end) cudaEventDestroy(c->ev_end);
    if (c->ev_order) cudaEventDestroy(c->ev_order);
    c->ev_begin = c->ev_end = c->ev_order = nullptr;
    dev_free(c->scan_keys), dev_free(c->scan_tmp);
    if (c->scan_scratch) cudaFree(c->scan_scratch);
    c->scan_scratch = nullptr;
    c->scan_cap = 0;
}

// Host-side state of a fresh cursor; device buffers are kept for reuse.
void cursor_reset(pvs_cursor* c) {
    c->index = nullptr;
    c->snap.reset();
    c->rows = c->visible = c->emitted = 0;
    c->state = PVS_OK;
    c->scanned = false;
    c->bmax_valid = false;
    c->batch_ws = false;
    c->fresh_ws = false;
    c->horizon = c->horizon_base = 0;
    c->pulls = c->interval_passes = c->horizon_builds = c->candidates = 0;
    c->code_bytes = 0;
    c->group_size = 1;
    c->ahead = c->ahead_pos = 0;
    c->ahead_host = false;
    c->readahead = 4;
    c->batch_passes = 0;
    c->batch_ms = 0.0;
    c->ev_pending = false;
    c->slot_fresh = false;
    c->slot_n = 0;
    c->interval_ms = 0.0;
    c->generator = PVS_GEN_INTERVALS;
    c->scan_ready = false;
}

// Closed cursors kept per index for reuse: at most kCursorPool of them and
// a quarter of the device's memory (at least kCursorPoolBytes) in device
// buffers.  Batched opens reuse hundreds of small cursors; single-query
// cursors hold buffers for every row (~460 MB at 8.8M rows), and grouped
// opens keep dozens of them in flight: a cursor that is not pooled frees its
// buffers, and cudaFree waits for the whole device.
constexpr size_t kCursorPool = 1024;
constexpr size_t kCursorPoolBytes = size_t(4) << 30;

size_t cursor_device_bytes(const pvs_cursor* c) {
    return (size_t)c->cap_rows * 12 + (size_t)c->cap_rows / 4 + (size_t)c->cap_w * 40 + 4096 +
           kFrontCap * 4 +
           (size_t)c->scan_cap * 20;
}

// Allocate the per-row state of a cursor (first pull); a pooled cursor keeps
// buffers that are large enough.
// Bounds of every row of the snapshot (single-query interval pass).
pvs_status cursor_alloc_full(pvs_cursor* c) {
    if (c->lo && c->cap_rows >= c->rows) return PVS_OK;
    dev_free(c->lo), dev_free(c->hi), dev_free(c->bmax), dev_free(c->compact_scratch);
    c->cap_rows = 0;
    c->bmax_valid = false;
    const size_t n = (size_t)std::max<int64_t>(c->rows, 1);
    PVS_CUDA(dev_alloc(&c->lo, n));
    PVS_CUDA(dev_alloc(&c->hi, n));
    PVS_CUDA(dev_alloc(&c->bmax, (n + kBmaxRows - 1) / kBmaxRows));
    PVS_CUDA(dev_alloc(&c->compact_scratch, compact_scratch_elems((int64_t)n)));
    c->cap_rows = (int64_t)n;
    return PVS_OK;
}

// Working-set arrays and pull scratch for up to `cap` entries (contents are
// not preserved when they grow).
pvs_status cursor_alloc_ws(pvs_cursor* c, int64_t cap) {
    cap = std::max<int64_t>(cap, 1);
    if (!c->front) PVS_CUDA(dev_alloc(&c->front, (size_t)kFrontCap));
    if (c->w_id && c->cap_w >= cap) return PVS_OK;
    dev_free(c->w_id), dev_free(c->w_lo), dev_free(c->w_hi);
    dev_free(c->cand), dev_free(c->keys), dev_free(c->keys_tmp);
    if (c->sort_scratch) cudaFree(c->sort_scratch);
    c->sort_scratch = nullptr;
    c->cap_w = 0;
    const size_t n = (size_t)cap;
    PVS_CUDA(dev_alloc(&c->w_id, n));
    PVS_CUDA(dev_alloc(&c->w_lo, n));
    PVS_CUDA(dev_alloc(&c->w_hi, n));
    PVS_CUDA(dev_alloc(&c->cand, n));
    PVS_CUDA(dev_alloc(&c->keys, n));
    PVS_CUDA(dev_alloc(&c->keys_tmp, n));
    PVS_CUDA(cudaMalloc(&c->sort_scratch, radix_sort_scratch_bytes((int64_t)n)));
    c->cap_w = cap;
    return PVS_OK;
}

pvs_status cursor_alloc_rows(pvs_cursor* c) {
    pvs_status s = cursor_alloc_full(c);
    if (s != PVS_OK) return s;
    return cursor_alloc_ws(c, c->rows);
}

pvs_status cursor_out_reserve(pvs_cursor* c, int64_t n) {
    if (n <= c->out_cap) return PVS_OK;
    dev_free(c->d_ids), dev_free(c->d_scores);
    if (c->h_ids) cudaFreeHost(c->h_ids);
    if (c->h_scores) cudaFreeHost(c->h_scores);
    c->h_ids = nullptr, c->h_scores = nullptr, c->out_cap = 0;
    const int64_t cap = std::max<int64_t>(n, 256);
    PVS_CUDA(dev_alloc(&c->d_ids, (size_t)cap));
    PVS_CUDA(dev_alloc(&c->d_scores, (size_t)cap));
    PVS_CUDA(cudaMallocHost(&c->h_ids, cap * sizeof(int64_t)));
    PVS_CUDA(cudaMallocHost(&c->h_scores, cap * sizeof(float)));
    c->out_cap = cap;
    return PVS_OK;
}

int grid_for(const pvs_cursor* c, int64_t items, int per_block = 256) {
    const int64_t g = std::max<int64_t>(1, (items + per_block - 1) / per_block);
    return (int)std::min<int64_t>(g, 4 * (int64_t)c->index->num_sms);
}

pvs_status fail(pvs_cursor* c, pvs_status s) {
    if (s < 0 && c->state >= 0) c->state = s;
    return s;
}

// Add the timed interval pass once its end event has completed.
void harvest_interval_time(pvs_cursor* c) {
    if (!c->ev_pending) return;
    if (cudaEventQuery(c->ev_end) != cudaSuccess) {
        cudaGetLastError();
        return;
    }
    float ms = 0.0f;
    if (cudaEventElapsedTime(&ms, c->ev_begin, c->ev_end) == cudaSuccess) c->interval_ms += ms;
    c->ev_pending = false;
}

// A pinned status word that the last kernel of a pull writes after its
// outputs (never a status value while pending).
constexpr int kStatusPending = 0x7fffffff;

// Wait for the status word to be published: spin, yielding every 256 reads,
// for at most 2 s; false when it was not published in that time.
bool wait_published(const int* word) {
    const volatile int* w = word;
    const auto t0 = std::chrono::steady_clock::now();
    for (uint32_t i = 1;; ++i) {
        if (*w != kStatusPending) {
            std::atomic_thread_fence(std::memory_order_acquire);
            return true;
        }
        if ((i & 255u) == 0) {
            if (std::chrono::steady_clock::now() - t0 > std::chrono::seconds(2)) return false;
            std::this_thread::yield();
        }
    }
}

// Read the device status word; a failure makes the cursor Failed.
pvs_status check_device_status(pvs_cursor* c) {
    cudaStream_t st = c->stream;
    PVS_CUDA(cudaMemcpyAsync(c->h_small, c->d_status, sizeof(int), cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaStreamSynchronize(st));
    const int s = (int)c->h_small[0];
    if (s != 0) return fail(c, (pvs_status)s);
    return PVS_OK;
}

pvs_status interval_pass(pvs_cursor* c) {
    pvs_index* x = c->index;
    IntervalArgs a;
    a.codes = x->codes;
    a.scale = x->scale;
    a.vnorm = x->vnorm;
    a.enorm = x->enorm;
    a.tomb = c->snap->d_tomb;
    a.rows = c->rows;
    a.m_pad = x->m_pad;
    a.zq = c->zq;
    a.qs = c->qs;
    a.lo = c->lo;
    a.hi = c->hi;
    a.status = c->d_status;
    a.wait_ns = x->wait_ns;
    // per-slot largest lower bounds, for the first working set (see
    // build_working_set): only when no row is tombstoned and every slot
    // scans at least kSlotTop rows, so that every entry is a live row's bound
    int64_t min_rows = 0;
    const int64_t slots = interval_slots(c->rows, x->m_pad, x->num_sms, &min_rows);
    c->slot_fresh = false;
    c->slot_n = 0;
    if (slots > 0 && c->snap->d_tomb == nullptr && min_rows >= kSlotTop) {
        if (c->slot_cap < slots * kSlotTop) {
            dev_free(c->slot_top);
            c->slot_cap = 0;
            PVS_CUDA(dev_alloc(&c->slot_top, (size_t)(slots * kSlotTop)));
            c->slot_cap = slots * kSlotTop;
        }
        a.slot_top = c->slot_top;
        c->slot_n = slots * kSlotTop;
    }
    if (!c->ev_begin) {
        PVS_CUDA(cudaEventCreate(&c->ev_begin));
        PVS_CUDA(cudaEventCreate(&c->ev_end));
    }
    // Interval passes of one index run one after another: each saturates
    // HBM, so overlapping two gains nothing; pulls of other cursors still
    // overlap the pass.  The pass waits for the previous pass's end event.
    std::lock_guard<std::mutex> lock(x->pass_mutex);
    if (!x->pass_done) PVS_CUDA(cudaEventCreateWithFlags(&x->pass_done, cudaEventDisableTiming));
    else PVS_CUDA(cudaStreamWaitEvent(c->stream, x->pass_done, 0));
    PVS_CUDA(cudaEventRecord(c->ev_begin, c->stream));
    PVS_CUDA(launch_interval_pass(a, x->num_sms, c->stream));
    c->slot_fresh = a.slot_top != nullptr;
    PVS_CUDA(cudaEventRecord(c->ev_end, c->stream));
    PVS_CUDA(cudaEventRecord(x->pass_done, c->stream));
    c->ev_pending = true;
    c->interval_passes++;
    c->code_bytes += c->rows * (int64_t)(x->m_pad + 12);
    c->scanned = true;
    c->bmax_valid = false;   // this pass writes no block maxima
    if (x->wait_ns < kWaitLimitNs) {
        // a shortened wait limit (pvs_index_set_wait_limit) makes a timed-out
        // pass likely: its bounds are then incomplete, so its status is read
        // here, before any later kernel of the pull uses them
        return check_device_status(c);
    }
    return PVS_OK;
}

// (Re)build the working set so that it holds the next `want` ranks.
pvs_status build_working_set(pvs_cursor* c, int64_t want) {
    pvs_index* x = c->index;
    const int64_t remaining = c->visible - c->emitted;
    int64_t H = std::max<int64_t>({want, 2 * c->horizon, 2048});
    if (H > remaining) H = remaining;
    if (H < remaining && c->slot_fresh && H <= c->slot_n) {
        // Each of the slot_n per-slot entries is the lower bound of a
        // distinct live row, so at least H rows have lo >= the H-th largest
        // entry v: v is at most the H-th largest lo of all rows, and the
        // rows with hi >= v hold the working set (a few more rows than the
        // exact threshold keeps; a few thousand entries are selected from
        // instead of every row).
        PVS_CUDA(launch_select_small(c->slot_top, c->slot_n, (uint64_t)H, c->sel, c->stream));
    } else if (H < remaining) {
        PVS_CUDA(launch_select_f32_n(c->lo, c->rows, (uint64_t)H, c->sel, grid_for(c, c->rows),
                                     c->stream));
    } else {
        PVS_CUDA(cudaMemsetAsync(c->sel, 0, sizeof(SelectState), c->stream));  // tau = 0: all live
    }
    PVS_CUDA(launch_compact_ordered(c->lo, c->hi, c->rows, c->sel, c->w_id, c->w_lo, c->w_hi,
                                    &c->ctr->w_len, c->compact_scratch, c->stream));
    c->slot_fresh = false;   // later builds select from the current bounds
    c->horizon = H;
    c->horizon_base = c->emitted;
    c->horizon_builds++;
    c->fresh_ws = true;
    // new indices: no frontier, default hint (front_k and front_hint are adjacent)
    PVS_CUDA(cudaMemsetAsync(&c->ctr->front_k, 0, 2 * sizeof(unsigned int), c->stream));
    return PVS_OK;
}

// The first working sets of the cursors of one stream that are due for
// one from their pass's per-slot lower bounds (build_working_set's first
// case), built together: four launches for all of them instead of four per
// cursor.  Cursors of one grouped pass share rows and slot count.  Cursors
// that do not qualify are left to prepare_pull.
// pulls[i]: the ranks cursor i's next pull computes (0: no pull).
pvs_status build_first_working_sets(pvs_cursor* const* cs, int32_t nc, const int64_t* pulls) {
    WsGroupArgs a;
    a.n = 0;
    pvs_cursor* picked[kGroupMax];
    int64_t H_of[kGroupMax];
    for (int32_t i = 0; i < nc && a.n < kGroupMax; ++i) {
        pvs_cursor* c = cs[i];
        if (c->state != PVS_OK || c->batch_ws || !c->scanned || !c->slot_fresh) continue;
        const int64_t n_eff = pulls[i];
        if (n_eff <= 0 || c->emitted + n_eff - c->horizon_base <= c->horizon) continue;
        const int64_t remaining = c->visible - c->emitted;
        const int64_t H = std::min<int64_t>(std::max<int64_t>({n_eff, 2 * c->horizon, 2048}),
                                            remaining);
        if (H >= remaining || H > c->slot_n) continue;
        if (a.n > 0 && (c->rows != a.rows || c->slot_n != a.slot_n)) continue;
        a.rows = c->rows;
        a.slot_n = c->slot_n;
        a.slot[a.n] = c->slot_top;
        a.k[a.n] = (uint64_t)H;
        a.sel[a.n] = c->sel;
        a.lo[a.n] = c->lo;
        a.hi[a.n] = c->hi;
        a.w_id[a.n] = c->w_id;
        a.w_lo[a.n] = c->w_lo;
        a.w_hi[a.n] = c->w_hi;
        a.w_len[a.n] = &c->ctr->w_len;
        a.scratch[a.n] = c->compact_scratch;
        a.bmax[a.n] = c->bmax_valid ? c->bmax : nullptr;
        picked[a.n] = c;
        H_of[a.n] = H;
        ++a.n;
    }
    if (a.n < 2) return PVS_OK;   // prepare_pull builds a lone one
    cudaStream_t st = picked[0]->stream;
    PVS_CUDA(launch_ws_group(a, st));
    for (int i = 0; i < a.n; ++i) {
        pvs_cursor* c = picked[i];
        c->slot_fresh = false;
        c->horizon = H_of[i];
        c->horizon_base = c->emitted;
        c->horizon_builds++;
        c->fresh_ws = true;
        // new indices: no frontier, default hint (front_k and front_hint are adjacent)
        PVS_CUDA(cudaMemsetAsync(&c->ctr->front_k, 0, 2 * sizeof(unsigned int), st));
    }
    return PVS_OK;
}

// One pull of n_eff >= 1 ranks into device buffers d_ids / d_scores.
// Full bounds for a cursor whose working set came from a batched pass: a
// single-query interval pass, then the working set's resolved scores and
// delivered items are carried over before the working set is rebuilt.
pvs_status rescan_from_batch(pvs_cursor* c) {
    pvs_status s = cursor_alloc_full(c);
    if (s != PVS_OK) return s;
    s = interval_pass(c);
    if (s != PVS_OK) return s;
    c->slot_fresh = false;   // the scatter below changes bounds (delivered rows leave)
    PVS_CUDA(launch_scatter_ws(c->w_id, c->w_lo, c->w_hi, &c->ctr->w_len, c->lo, c->hi,
                               grid_for(c, c->cap_w), c->stream));
    // the working set is rebuilt from the full bounds; its arrays may grow
    PVS_CUDA(cudaStreamSynchronize(c->stream));
    s = cursor_alloc_ws(c, c->rows);
    if (s != PVS_OK) return s;
    c->batch_ws = false;
    c->horizon = 0;   // the next pull rebuilds the working set from the full bounds
    return PVS_OK;
}

// Make the cursor's working set hold the next n_eff ranks.
pvs_status prepare_pull(pvs_cursor* c, int64_t n_eff) {
    pvs_status s;
    if (!c->scanned && !c->batch_ws) {
        s = cursor_alloc_rows(c);
        if (s != PVS_OK) return s;
        s = interval_pass(c);
        if (s != PVS_OK) return s;
    }
    if (c->emitted + n_eff - c->horizon_base > c->horizon) {
        if (c->batch_ws) {
            s = rescan_from_batch(c);
            if (s != PVS_OK) return s;
        }
        s = build_working_set(c, n_eff);
        if (s != PVS_OK) return s;
    }
    return PVS_OK;
}

// status_mirror: a pinned host word the one-launch path sets to the status
// after the pull (host-buffer pulls); null for device-buffer pulls.
// Exhaustive float32 scanning (PVS_GEN_FULL_SCAN): the first pull scores
// every visible row exactly and sorts all keys once; every pull emits the
// next keys of that order.
pvs_status scan_pull(pvs_cursor* c, int64_t n_eff, int64_t* d_ids, float* d_scores,
                     int* status_mirror) {
    pvs_index* x = c->index;
    cudaStream_t st = c->stream;
    if (!c->scan_ready) {
        const int64_t rows = std::max<int64_t>(c->rows, 1);
        if (c->scan_cap < rows) {
            dev_free(c->scan_keys), dev_free(c->scan_tmp);
            if (c->scan_scratch) cudaFree(c->scan_scratch);
            c->scan_scratch = nullptr;
            c->scan_cap = 0;
            if (dev_alloc(&c->scan_keys, (size_t)rows) != cudaSuccess ||
                dev_alloc(&c->scan_tmp, (size_t)rows) != cudaSuccess ||
                cudaMalloc(&c->scan_scratch, radix_sort_scratch_bytes(rows)) != cudaSuccess)
                return fail(c, PVS_ERR_OOM);
            c->scan_cap = rows;
        }
        cudaError_t e = launch_scan_scores(c->qraw, x->raw, x->m_raw, c->rows, c->snap->d_tomb,
                                           c->scan_keys, c->d_status, c->ctr, st);
        if (e == cudaSuccess && c->rows > 1)
            e = launch_radix_sort_desc(c->scan_keys, c->scan_tmp, c->rows, c->scan_scratch, st);
        if (e != cudaSuccess) return fail(c, cuda_status(e));
        c->scan_ready = true;
    }
    cudaError_t e = launch_scan_emit(c->scan_keys + c->emitted, n_eff, d_ids, d_scores,
                                     c->d_status, status_mirror, st);
    if (e != cudaSuccess) return fail(c, cuda_status(e));
    c->emitted += n_eff;
    c->pulls++;
    return PVS_OK;
}

pvs_status pull(pvs_cursor* c, int64_t n_eff, int64_t* d_ids, float* d_scores,
                int* status_mirror = nullptr) {
    if (c->generator == PVS_GEN_FULL_SCAN) return scan_pull(c, n_eff, d_ids, d_scores, status_mirror);
    pvs_index* x = c->index;
    cudaStream_t st = c->stream;
    pvs_status s = prepare_pull(c, n_eff);
    if (s != PVS_OK) return fail(c, s);
    if (n_eff <= kPullFusedMax) {
        // one launch, no host round trip; failures surface at the next sync
        PullArgs a;
        a.w_id = c->w_id;
        a.w_lo = c->w_lo;
        a.w_hi = c->w_hi;
        a.w_len = &c->ctr->w_len;
        a.lo = c->lo;
        a.hi = c->hi;
        a.qraw = c->qraw;
        a.raw = x->raw;
        a.m_raw = x->m_raw;
        a.n = (int)n_eff;
        a.cand = c->cand;
        a.keys = reinterpret_cast<unsigned long long*>(c->keys);
        a.out_ids = d_ids;
        a.out_scores = d_scores;
        a.status = c->d_status;
        a.ctr = c->ctr;
        a.front = c->front;
        a.status_mirror = status_mirror;
        // the first pull of a working set refines most of it: spread that
        // over every SM; later pulls take one cluster launch
        cudaError_t e = c->fresh_ws ? launch_pull_fused(a, 2 * x->num_sms, st)
                                    : launch_pull_cluster(a, st);
        if (e != cudaSuccess) return fail(c, cuda_status(e));
        c->fresh_ws = false;
        c->emitted += n_eff;
        c->pulls++;
        return PVS_OK;
    }
    const int grid_w = grid_for(c, std::min<int64_t>(c->rows, (int64_t)1 << 22));
    // rows leave without the one-launch pull's frontier count: drop the frontier
    cudaError_t e = cudaMemsetAsync(&c->ctr->front_k, 0, sizeof(unsigned int), st);
    if (e == cudaSuccess)
        e = launch_select_f32(c->w_lo, &c->ctr->w_len, (uint64_t)n_eff, c->sel, grid_w, st);
    if (e == cudaSuccess)
        e = launch_candidates(c->w_lo, c->w_hi, &c->ctr->w_len, c->sel, c->cand, &c->ctr->cand,
                              grid_w, st);
    if (e == cudaSuccess)
        e = launch_refine(c->cand, &c->ctr->cand, c->w_id, c->w_lo, c->w_hi, c->lo, c->hi, c->qraw,
                          x->raw, x->m_raw, c->d_status, c->ctr, 2 * x->num_sms, st);
    if (e == cudaSuccess) e = launch_make_keys(c->cand, &c->ctr->cand, c->w_lo, c->keys, grid_w, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(c->h_small + 1, &c->ctr->cand, sizeof(unsigned int),
                            cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(c->h_small, c->d_status, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return fail(c, cuda_status(e));
    harvest_interval_time(c);
    if ((int)c->h_small[0] != 0) return fail(c, (pvs_status)(int)c->h_small[0]);
    const int64_t cand = c->h_small[1];
    if (cand < n_eff) return fail(c, PVS_ERR_INVALID);   // internal invariant
    c->candidates += cand;
    if (cand <= kBitonicMax)
        e = launch_bitonic_desc(c->keys, (int)cand, st);
    else
        e = launch_radix_sort_desc(c->keys, c->keys_tmp, cand, c->sort_scratch, st);
    if (e == cudaSuccess)
        e = launch_emit(c->keys, (int)n_eff, c->w_id, c->w_lo, c->w_hi, c->lo, c->hi, d_ids,
                        d_scores, st);
    if (e != cudaSuccess) return fail(c, cuda_status(e));
    c->emitted += n_eff;
    c->pulls++;
    return PVS_OK;
}

// ---------------------------------------------------------------------------
// batched open: one tensor-core interval pass for up to kBatchMax queries
// ---------------------------------------------------------------------------
constexpr int kBatchMax = 256;

// Stream-ordered scratch that is released (stream-ordered) at scope exit.
struct DevBuf {
    cudaStream_t st = nullptr;
    cudaMemPool_t pool = nullptr;
    std::vector<void*> ptrs;
    DevBuf(cudaStream_t s, cudaMemPool_t p) : st(s), pool(p) {}
    template <typename T>
    T* get(size_t count) {
        void* p = nullptr;
        const size_t bytes = std::max<size_t>(count, 1) * sizeof(T);
        const cudaError_t e = pool ? cudaMallocFromPoolAsync(&p, bytes, pool, st)
                                   : cudaMallocAsync(&p, bytes, st);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        ptrs.push_back(p);
        return static_cast<T*>(p);
    }
    ~DevBuf() {
        for (void* p : ptrs) cudaFreeAsync(p, st);
    }
};

// Status words (and, if ctr is given, counters) of n cursors that share
// stream st: one gather launch, one copy back, one synchronisation.
pvs_status gather_state(pvs_cursor* const* cs, int n, cudaStream_t st, int* status,
                        DevCounters* ctr) {
    if (n <= 0) return PVS_OK;
    DevBuf buf(st, cs[0]->index->scratch_pool);
    CursorRef* d_refs = buf.get<CursorRef>((size_t)n);
    int* d_status = buf.get<int>((size_t)n);
    DevCounters* d_ctr = ctr ? buf.get<DevCounters>((size_t)n) : nullptr;
    if (!d_refs || !d_status || (ctr && !d_ctr)) return PVS_ERR_OOM;
    std::vector<CursorRef> refs((size_t)n);
    for (int i = 0; i < n; ++i) refs[(size_t)i] = CursorRef{cs[i]->d_status, cs[i]->ctr};
    PVS_CUDA(cudaMemcpyAsync(d_refs, refs.data(), (size_t)n * sizeof(CursorRef),
                             cudaMemcpyHostToDevice, st));
    PVS_CUDA(launch_gather_state(d_refs, n, d_status, d_ctr, st));
    PVS_CUDA(cudaMemcpyAsync(status, d_status, (size_t)n * sizeof(int), cudaMemcpyDeviceToHost,
                             st));
    if (ctr)
        PVS_CUDA(cudaMemcpyAsync(ctr, d_ctr, (size_t)n * sizeof(DevCounters),
                                 cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaStreamSynchronize(st));
    return PVS_OK;
}

// gather_state over cursors on any mix of streams: one round per stream.
pvs_status gather_state_any(pvs_cursor* const* cs, int n, int* status, DevCounters* ctr) {
    std::vector<cudaStream_t> streams;
    for (int i = 0; i < n; ++i)
        if (std::find(streams.begin(), streams.end(), cs[i]->stream) == streams.end())
            streams.push_back(cs[i]->stream);
    std::vector<pvs_cursor*> group;
    std::vector<int> where, g_status;
    std::vector<DevCounters> g_ctr;
    for (cudaStream_t st : streams) {
        group.clear();
        where.clear();
        for (int i = 0; i < n; ++i)
            if (cs[i]->stream == st) {
                group.push_back(cs[i]);
                where.push_back(i);
            }
        g_status.assign(group.size(), 0);
        g_ctr.assign(ctr ? group.size() : 0, DevCounters{});
        pvs_status s = gather_state(group.data(), (int)group.size(), st, g_status.data(),
                                    ctr ? g_ctr.data() : nullptr);
        if (s != PVS_OK) return s;
        for (size_t j = 0; j < group.size(); ++j) {
            status[where[j]] = g_status[j];
            if (ctr) ctr[where[j]] = g_ctr[j];
        }
    }
    return PVS_OK;
}

struct BatchQueries {
    int nq = 0, nq_pad = 0;
    int8_t* zq = nullptr;          // [nq][m_pad]
    float* qraw = nullptr;         // [nq][m_raw]
    QueryScalars* qs = nullptr;    // [nq]
    uint16_t* qcodes = nullptr;    // [nq_pad][m_pad] bf16, zero rows past nq
};

// bf16 copy of every code row (the tensor-core pass reads it), extended on
// stream st; st then waits for the last conversion, whichever stream ran it.
// Caller holds x->pass_mutex.
pvs_status ensure_bf16(pvs_index* x, cudaStream_t st) {
    if (!x->codes_bf16) {
        PVS_CUDA(dev_alloc(&x->codes_bf16, (size_t)std::max<int64_t>(x->cap, 1) * x->m_pad));
        x->bf16_rows = 0;
    }
    if (!x->bf16_ready) PVS_CUDA(cudaEventCreateWithFlags(&x->bf16_ready, cudaEventDisableTiming));
    if (x->bf16_rows < x->size) {
        const int64_t r0 = x->bf16_rows;
        PVS_CUDA(launch_codes_to_bf16(x->codes + r0 * x->m_pad, x->codes_bf16 + r0 * x->m_pad,
                                      (x->size - r0) * x->m_pad, st));
        x->bf16_rows = x->size;
        PVS_CUDA(cudaEventRecord(x->bf16_ready, st));
    } else {
        PVS_CUDA(cudaStreamWaitEvent(st, x->bf16_ready, 0));
    }
    return PVS_OK;
}

// Encode nq queries on the index stream; checks their status (waits).
// Encode nq queries for the batched pass.  With check_now the call waits and
// reports a non-finite query; otherwise the caller reads bq->qs[i].status
// later, at its own synchronisation point.
pvs_status encode_batch(pvs_index* x, const float* queries, int nq, bool on_device, DevBuf& buf,
                        BatchQueries* bq, cudaStream_t st, bool check_now = true) {
    bq->nq = nq;
    bq->nq_pad = (int)round_up(nq, 32);
    bq->zq = buf.get<int8_t>((size_t)nq * x->m_pad);
    bq->qraw = buf.get<float>((size_t)nq * x->m_raw);
    bq->qs = buf.get<QueryScalars>((size_t)nq);
    bq->qcodes = buf.get<uint16_t>((size_t)bq->nq_pad * x->m_pad);
    const float* qd = queries;
    if (!on_device) {
        float* tmp = buf.get<float>((size_t)nq * x->m);
        if (!tmp) return PVS_ERR_OOM;
        PVS_CUDA(cudaMemcpyAsync(tmp, queries, (size_t)nq * x->m * sizeof(float),
                                 cudaMemcpyHostToDevice, st));
        qd = tmp;
    }
    if (!bq->zq || !bq->qraw || !bq->qs || !bq->qcodes) return PVS_ERR_OOM;
    PVS_CUDA(launch_encode_queries(qd, nq, x->m, x->m_pad, x->m_raw, bq->zq, bq->qraw, bq->qs, st));
    PVS_CUDA(cudaMemsetAsync(bq->qcodes, 0, (size_t)bq->nq_pad * x->m_pad * sizeof(uint16_t), st));
    PVS_CUDA(launch_codes_to_bf16(bq->zq, bq->qcodes, (int64_t)nq * x->m_pad, st));
    {
        std::lock_guard<std::mutex> lock(x->pass_mutex);
        pvs_status s = ensure_bf16(x, st);
        if (s != PVS_OK) return s;
    }
    if (!check_now) return PVS_OK;
    std::vector<QueryScalars> h(nq);
    PVS_CUDA(cudaMemcpyAsync(h.data(), bq->qs, nq * sizeof(QueryScalars), cudaMemcpyDeviceToHost,
                             st));
    PVS_CUDA(cudaStreamSynchronize(st));
    for (int i = 0; i < nq; ++i)
        if (h[i].status != 0) return (pvs_status)h[i].status;
    return PVS_OK;
}

// A cursor with its small buffers, fresh counters and the given snapshot.
// With zero_state false the caller zeroes the counters and status word on the
// device itself (the batched open does it in its query copy).
pvs_status acquire_cursor(pvs_index* x, const std::shared_ptr<SnapData>& sd, pvs_cursor** out,
                          bool zero_state = true) {
    pvs_cursor* c = nullptr;
    {
        std::lock_guard<std::mutex> lock(x->pool_mutex);
        if (!x->cursor_pool.empty()) {
            c = x->cursor_pool.back();
            x->cursor_pool.pop_back();
            x->pool_bytes -= cursor_device_bytes(c);
        }
    }
    if (!c) {
        c = new (std::nothrow) pvs_cursor();
        if (!c) return PVS_ERR_OOM;
    }
    cursor_reset(c);
    c->index = x;
    c->stream = x->stream;
    c->snap = sd;
    c->rows = sd->rows;
    c->visible = sd->visible;
    *out = c;
    if (!c->zq &&
        (dev_alloc(&c->zq, (size_t)x->m_pad) != cudaSuccess ||
         dev_alloc(&c->qraw, (size_t)x->m_raw) != cudaSuccess ||
         dev_alloc(&c->qs, 1) != cudaSuccess || dev_alloc(&c->sel, 1) != cudaSuccess ||
         dev_alloc(&c->ctr, 1) != cudaSuccess || dev_alloc(&c->d_status, 1) != cudaSuccess ||
         cudaMallocHost(&c->h_small, 16 * sizeof(unsigned int)) != cudaSuccess))
        return PVS_ERR_OOM;
    if (zero_state) {
        PVS_CUDA(cudaMemsetAsync(c->ctr, 0, sizeof(DevCounters), c->stream));
        PVS_CUDA(cudaMemsetAsync(c->d_status, 0, sizeof(int), c->stream));
    }
    c->state = c->visible == 0 ? PVS_EXHAUSTED : PVS_OK;
    return PVS_OK;
}

// Up to kBatchMax cursors from one batched pass:
//   1. encode the queries; bf16 query codes for the MMA;
//   2. thresholds: on every 16th 128-row tile (every tile for small corpora)
//      the pass dumps all intervals; tau_q = the k-th largest lower bound of
//      query q there, k sized so that about 3x the horizon rows of the whole
//      corpus reach it;
//   3. the filter pass appends every row with hi >= tau_q to query q's
//      working set and counts the rows with lo >= tau_q: those rows precede
//      every row outside the working set, so the cursor can deliver that many
//      ranks before it needs a single-query pass;
//   4. each working set is sorted by id into its cursor.
// A query whose working set overflows, or whose count is 0, falls back to a
// single-query interval pass at its first pull.
pvs_status open_batch_group(pvs_index* x, const std::shared_ptr<SnapData>& sd,
                            const float* queries, int nq, bool on_device, int horizon,
                            cudaStream_t st, pvs_cursor** out) {
    DevBuf buf(st, x->scratch_pool);
    BatchQueries bq;
    // one synchronisation at the end: query statuses are read with the pass's
    pvs_status s = encode_batch(x, queries, nq, on_device, buf, &bq, st, /*check_now=*/false);
    if (s != PVS_OK) return s;
    for (int i = 0; i < nq; ++i) {
        s = acquire_cursor(x, sd, &out[i], /*zero_state=*/false);
        if (s != PVS_OK) return s;
        out[i]->stream = st;
    }
    QueryDst* d_qd = buf.get<QueryDst>((size_t)nq);
    if (!d_qd) return PVS_ERR_OOM;
    {
        // a pageable source is staged before cudaMemcpyAsync returns
        std::vector<QueryDst> qd(nq);
        for (int i = 0; i < nq; ++i)
            qd[i] = QueryDst{out[i]->zq, out[i]->qraw, out[i]->qs, out[i]->ctr, out[i]->d_status};
        PVS_CUDA(cudaMemcpyAsync(d_qd, qd.data(), nq * sizeof(QueryDst), cudaMemcpyHostToDevice, st));
        PVS_CUDA(launch_copy_queries(bq.zq, bq.qraw, bq.qs, d_qd, nq, x->m_pad, x->m_raw, st));
    }
    std::vector<QueryScalars> h_qs(nq);
    const int64_t rows = sd->rows;
    if (rows == 0) {
        PVS_CUDA(cudaMemcpyAsync(h_qs.data(), bq.qs, nq * sizeof(QueryScalars),
                                 cudaMemcpyDeviceToHost, st));
        PVS_CUDA(cudaStreamSynchronize(st));
        for (int i = 0; i < nq; ++i)
            if (h_qs[i].status != 0) return (pvs_status)h_qs[i].status;
        return PVS_OK;
    }

    // Sample every stride-th tile and take tau_q = the k_s-th largest sampled
    // lower bound, k_s = 2 H / stride + 4: about 2 H rows of the corpus reach
    // it.  It misses the horizon (fewer than H rows reach it) only when at
    // least k_s of the top-H rows were sampled; that count is about
    // Poisson(H / stride), so this happens for about 1e-5 of the queries
    // (H = 200: stride 12, k_s = 38, mean 16.7), which then rescan.
    const int64_t ntiles = (rows + 127) / 128;
    int stride = (int)std::min<int64_t>(16, std::max<int64_t>(1, (3 * (int64_t)horizon) / 48));
    if (ntiles < 8 * (int64_t)stride) stride = 1;
    const int64_t ld = ((ntiles + stride - 1) / stride) * 128;
    const unsigned int k_s =
        stride == 1 ? (unsigned int)horizon
                    : (unsigned int)((2 * (int64_t)horizon + stride - 1) / stride + 4);
    const int w_cap = (int)std::min<int64_t>((int64_t)kWsSortMax, std::max<int64_t>(rows, 1));
    float* dlo = buf.get<float>((size_t)nq * ld);
    float* dhi = dlo;   // the sampling pass needs the lower bounds only
    float* tau = buf.get<float>((size_t)nq);
    float* rmax = buf.get<float>((size_t)nq);
    int* status = buf.get<int>(1);
    int32_t* wid = buf.get<int32_t>((size_t)nq * w_cap);
    float* wlo = buf.get<float>((size_t)nq * w_cap);
    float* whi = buf.get<float>((size_t)nq * w_cap);
    unsigned int* wlen = buf.get<unsigned int>((size_t)nq);
    unsigned int* heff = buf.get<unsigned int>((size_t)nq);
    WsDst* d_ws = buf.get<WsDst>((size_t)nq);
    if (!dlo || !dhi || !tau || !rmax || !status || !wid || !wlo || !whi || !wlen ||
        !heff || !d_ws)
        return PVS_ERR_OOM;
    PVS_CUDA(cudaMemsetAsync(status, 0, sizeof(int), st));
    PVS_CUDA(cudaMemsetAsync(wlen, 0, nq * sizeof(unsigned int), st));
    PVS_CUDA(cudaMemsetAsync(heff, 0, nq * sizeof(unsigned int), st));

    BatchArgs a{};
    a.rows = rows;
    a.m_pad = x->m_pad;
    a.nq = nq;
    a.nq_pad = bq.nq_pad;
    a.scale = x->scale;
    a.vnorm = x->vnorm;
    a.enorm = x->enorm;
    a.tomb = sd->d_tomb;
    a.qs = bq.qs;
    a.status = status;
    // 2. thresholds from the sampled tiles
    a.mode = 0;
    a.tile_stride = stride;
    a.dump_lo = dlo;
    a.dump_hi = nullptr;
    a.dump_ld = ld;
    PVS_CUDA(launch_batch_intervals(a, x->codes_bf16, bq.qcodes, x->num_sms, st));
    PVS_CUDA(launch_batch_tau(dlo, ld, (unsigned int)ld, nq, k_s, tau, st));
    PVS_CUDA(launch_rmax(bq.qs, nq, x->norm_maxes, rmax, st));   // maxima over all rows: a valid bound
    // 3. the filter pass over every row
    a.mode = 1;
    a.tile_stride = 1;
    a.dump_lo = a.dump_hi = nullptr;
    a.dump_ld = 0;
    a.tau = tau;
    a.rmax = rmax;
    a.w_id = wid;
    a.w_lo = wlo;
    a.w_hi = whi;
    a.w_cap = w_cap;
    a.w_len = wlen;
    a.h_eff = heff;
    cudaEvent_t ev0 = nullptr, ev1 = nullptr;
    PVS_CUDA(cudaEventCreate(&ev0));
    PVS_CUDA(cudaEventCreate(&ev1));
    {
        std::lock_guard<std::mutex> lock(x->pass_mutex);   // one HBM pass at a time
        if (x->pass_done) PVS_CUDA(cudaStreamWaitEvent(st, x->pass_done, 0));
        PVS_CUDA(cudaEventRecord(ev0, st));
        PVS_CUDA(launch_batch_intervals(a, x->codes_bf16, bq.qcodes, x->num_sms, st));
        PVS_CUDA(cudaEventRecord(ev1, st));
        if (!x->pass_done)
            PVS_CUDA(cudaEventCreateWithFlags(&x->pass_done, cudaEventDisableTiming));
        PVS_CUDA(cudaEventRecord(x->pass_done, st));
    }
    // 4. ordered working sets into the cursors
    std::vector<WsDst> ws(nq);
    for (int i = 0; i < nq; ++i) {
        s = cursor_alloc_ws(out[i], w_cap);
        if (s != PVS_OK) return s;
        ws[i] = WsDst{out[i]->w_id, out[i]->w_lo, out[i]->w_hi, &out[i]->ctr->w_len};
    }
    PVS_CUDA(cudaMemcpyAsync(d_ws, ws.data(), nq * sizeof(WsDst), cudaMemcpyHostToDevice, st));
    PVS_CUDA(launch_ws_sort(wid, wlo, whi, w_cap, wlen, d_ws, nq, st));
    std::vector<unsigned int> h_wlen(nq), h_heff(nq);
    int h_status = 0;
    PVS_CUDA(cudaMemcpyAsync(h_wlen.data(), wlen, nq * sizeof(unsigned int), cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaMemcpyAsync(h_heff.data(), heff, nq * sizeof(unsigned int), cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaMemcpyAsync(&h_status, status, sizeof(int), cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaMemcpyAsync(h_qs.data(), bq.qs, nq * sizeof(QueryScalars), cudaMemcpyDeviceToHost,
                             st));
    PVS_CUDA(cudaStreamSynchronize(st));
    float pass_ms = 0.0f;
    cudaEventElapsedTime(&pass_ms, ev0, ev1);
    cudaEventDestroy(ev0);
    cudaEventDestroy(ev1);
    for (int i = 0; i < nq; ++i)   // a non-finite query fails the batch
        if (h_qs[i].status != 0) return (pvs_status)h_qs[i].status;
    if (h_status != 0) return (pvs_status)h_status;
    for (int i = 0; i < nq; ++i) {
        pvs_cursor* c = out[i];
        if (h_wlen[i] <= (unsigned int)w_cap && h_heff[i] > 0) {
            c->batch_ws = true;
            c->fresh_ws = true;
            c->horizon = h_heff[i];
            c->horizon_base = 0;
        }
        c->batch_passes = 1;
        c->batch_ms = pass_ms;   // the filter pass, shared by the group's cursors
    }
    return PVS_OK;
}

}  // namespace

// ===========================================================================
// C ABI
// ===========================================================================
// The index's device is current for the duration of a call (the CUDA
// runtime's current device belongs to the calling host thread).
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

static int index_device(const pvs_index* x) { return x ? x->device : -1; }
static int cursor_device(const pvs_cursor* c) { return c && c->index ? c->index->device : -1; }
static int first_cursor_device(pvs_cursor* const* cs, int32_t nc) {
    return cs && nc > 0 ? cursor_device(cs[0]) : -1;
}

extern "C" {

int64_t pvs_launch_count(void) { return (int64_t)g_launches.load(); }

pvs_status pvs_cursor_set_generator(pvs_cursor* c, int32_t generator) {
    if (!c || !c->index) return PVS_ERR_INVALID;
    if (generator != PVS_GEN_INTERVALS && generator != PVS_GEN_FULL_SCAN) return PVS_ERR_INVALID;
    if (c->pulls != 0 || c->emitted != 0 || c->batch_ws) return PVS_ERR_INVALID;
    c->generator = generator;
    return PVS_OK;
}

pvs_status pvs_cursor_set_stream(pvs_cursor* c, void* cuda_stream) {
    DeviceGuard device_guard(cursor_device(c));
    if (!c || !c->index) return PVS_ERR_INVALID;
    PVS_CUDA(cudaStreamSynchronize(c->stream));
    c->stream = cuda_stream ? static_cast<cudaStream_t>(cuda_stream) : c->index->stream;
    return PVS_OK;
}

const char* pvs_status_string(int32_t s) {
    switch (s) {
        case PVS_OK: return "ok";
        case PVS_EXHAUSTED: return "exhausted";
        case PVS_ERR_INVALID: return "invalid argument";
        case PVS_ERR_NONFINITE: return "non-finite input";
        case PVS_ERR_OVERFLOW: return "overflow";
        case PVS_ERR_INTERVAL: return "authoritative score outside its interval";
        case PVS_ERR_CUDA: return "CUDA error";
        case PVS_ERR_OOM: return "out of memory";
        case PVS_ERR_TIMEOUT: return "device wait timed out";
        case PVS_ERR_FAILED: return "cursor failed earlier";
        default: return "unknown status";
    }
}

pvs_status pvs_build(const float* vecs, int64_t n, int32_t dim, int32_t vecs_on_device,
                     void* cuda_stream, pvs_index** out) {
    return pvs_build_ex(vecs, n, dim, vecs_on_device, cuda_stream, PVS_QUANT_PER_VECTOR, out);
}

}  // extern "C"

namespace {

// An empty index for vectors of dimension dim: device, stream, status word
// and scratch pool (no rows yet).
pvs_status index_create(int32_t dim, void* cuda_stream, pvs_index** out) {
    pvs_index* x = new (std::nothrow) pvs_index();
    if (!x) return PVS_ERR_OOM;
    auto bail = [&](pvs_status s) {
        pvs_index_free(x);
        return s;
    };
    if (cudaGetDevice(&x->device) != cudaSuccess) return bail(PVS_ERR_CUDA);
    if (cudaDeviceGetAttribute(&x->num_sms, cudaDevAttrMultiProcessorCount, x->device) !=
        cudaSuccess)
        return bail(PVS_ERR_CUDA);
    x->m = dim;
    x->m_pad = (int)round_up(dim, kCodeAlign);
    x->m_raw = (int)round_up(dim, 4);
    {
        size_t free_b = 0, total_b = 0;
        if (cudaMemGetInfo(&free_b, &total_b) != cudaSuccess) return bail(PVS_ERR_CUDA);
        x->pool_limit = std::max(kCursorPoolBytes, total_b / 4);
    }
    if (cuda_stream) {
        x->stream = static_cast<cudaStream_t>(cuda_stream);
    } else {
        if (cudaStreamCreateWithFlags(&x->stream, cudaStreamNonBlocking) != cudaSuccess)
            return bail(PVS_ERR_CUDA);
        x->own_stream = true;
    }
    if (cudaMalloc(&x->d_status, sizeof(int)) != cudaSuccess) return bail(PVS_ERR_OOM);
    {
        cudaMemPoolProps props{};
        props.allocType = cudaMemAllocationTypePinned;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = x->device;
        if (cudaMemPoolCreate(&x->scratch_pool, &props) != cudaSuccess) {
            x->scratch_pool = nullptr;
            return bail(PVS_ERR_CUDA);
        }
        uint64_t keep = UINT64_MAX;
        cudaMemPoolSetAttribute(x->scratch_pool, cudaMemPoolAttrReleaseThreshold, &keep);
    }
    *out = x;
    return PVS_OK;
}

}  // namespace

extern "C" {

pvs_status pvs_build_ex(const float* vecs, int64_t n, int32_t dim, int32_t vecs_on_device,
                        void* cuda_stream, int32_t quantization, pvs_index** out) {
    if (!out) return PVS_ERR_INVALID;
    *out = nullptr;
    if (dim < 1 || dim > kMaxDim || n < 0 || n >= ((int64_t)1 << 31) || (n > 0 && !vecs) ||
        (quantization != PVS_QUANT_PER_VECTOR && quantization != PVS_QUANT_GLOBAL))
        return PVS_ERR_INVALID;
    pvs_index* x = nullptr;
    pvs_status s0 = index_create(dim, cuda_stream, &x);
    if (s0 != PVS_OK) return s0;
    auto bail = [&](pvs_status s) {
        pvs_index_free(x);
        return s;
    };
    if (vecs_on_device && n > 0 && !is_device_ptr(vecs)) return bail(PVS_ERR_INVALID);
    if (quantization == PVS_QUANT_GLOBAL) {
        // one scale for the corpus: RN(max |v_j| / 127), from the largest entry
        x->quant = PVS_QUANT_GLOBAL;
        unsigned int* mx = nullptr;
        if (dev_alloc(&x->gscale, 1) != cudaSuccess || dev_alloc(&mx, 1) != cudaSuccess) {
            dev_free(mx);
            return bail(PVS_ERR_OOM);
        }
        cudaError_t e = cudaMemsetAsync(mx, 0, sizeof(unsigned int), x->stream);
        if (e == cudaSuccess && vecs_on_device) {
            e = launch_maxabs(vecs, n * (int64_t)dim, mx, x->stream);
        } else if (e == cudaSuccess) {
            float m = 0.0f;
            for (int64_t i = 0; i < n * (int64_t)dim; ++i) m = std::max(m, std::fabs(vecs[i]));
            unsigned int bits;
            std::memcpy(&bits, &m, sizeof bits);
            e = cudaMemcpyAsync(mx, &bits, sizeof bits, cudaMemcpyHostToDevice, x->stream);
        }
        if (e == cudaSuccess) e = launch_scale_from_maxabs(mx, x->gscale, x->stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(x->stream);
        dev_free(mx);
        if (e != cudaSuccess) return bail(cuda_status(e));
    }
    pvs_status s = index_reserve(x, n);
    if (s != PVS_OK) return bail(s);
    s = index_fill(x, vecs, n, vecs_on_device != 0);
    if (s != PVS_OK) return bail(s);
    x->size = n;
    x->live = n;
    s = refresh_norm_maxes(x);
    if (s != PVS_OK) return bail(s);
    *out = x;
    return PVS_OK;
}

pvs_status pvs_index_import(const float* vecs, const int8_t* codes, const float* scale,
                            const float* vnorm, const float* enorm, int64_t n, int32_t dim,
                            void* cuda_stream, pvs_index** out) {
    if (!out) return PVS_ERR_INVALID;
    *out = nullptr;
    if (dim < 1 || dim > kMaxDim || n < 0 || n >= ((int64_t)1 << 31) ||
        (n > 0 && (!vecs || !codes || !scale || !vnorm || !enorm)))
        return PVS_ERR_INVALID;
    // what the method relies on without recomputing it: codes in [-127, 127]
    // (the Int8 dot products cannot overflow), finite inputs, positive scales
    for (int64_t i = 0; i < n; ++i) {
        if (!(std::isfinite(scale[i]) && scale[i] > 0.0f) || !std::isfinite(vnorm[i]) ||
            !std::isfinite(enorm[i]) || vnorm[i] < 0.0f || enorm[i] < 0.0f)
            return PVS_ERR_INVALID;
        for (int32_t j = 0; j < dim; ++j) {
            const int8_t z = codes[i * (int64_t)dim + j];
            if (z < -127) return PVS_ERR_INVALID;
            if (!std::isfinite(vecs[i * (int64_t)dim + j])) return PVS_ERR_NONFINITE;
        }
    }
    pvs_index* x = nullptr;
    pvs_status s = index_create(dim, cuda_stream, &x);
    if (s != PVS_OK) return s;
    auto bail = [&](pvs_status st) {
        pvs_index_free(x);
        return st;
    };
    s = index_reserve(x, n);
    if (s != PVS_OK) return bail(s);
    cudaStream_t st = x->stream;
    if (n > 0) {
        // padded rows: zero bytes and floats beyond dim, as the builder writes them
        cudaError_t e = cudaMemsetAsync(x->codes, 0, (size_t)n * x->m_pad, st);
        if (e == cudaSuccess)
            e = cudaMemsetAsync(x->raw, 0, (size_t)n * x->m_raw * sizeof(float), st);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(x->codes, (size_t)x->m_pad, codes, (size_t)dim, (size_t)dim,
                                  (size_t)n, cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(x->raw, (size_t)x->m_raw * sizeof(float), vecs,
                                  (size_t)dim * sizeof(float), (size_t)dim * sizeof(float),
                                  (size_t)n, cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(x->scale, scale, n * sizeof(float), cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(x->vnorm, vnorm, n * sizeof(float), cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(x->enorm, enorm, n * sizeof(float), cudaMemcpyHostToDevice, st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(st);
        if (e != cudaSuccess) return bail(cuda_status(e));
    }
    x->size = n;
    x->live = n;
    s = refresh_norm_maxes(x);
    if (s != PVS_OK) return bail(s);
    *out = x;
    return PVS_OK;
}

pvs_status pvs_index_set_wait_limit(pvs_index* x, int64_t ns) {
    if (!x || ns < 0) return PVS_ERR_INVALID;
    x->wait_ns = (unsigned long long)std::min<int64_t>(ns, (int64_t)kWaitLimitNs);
    return PVS_OK;
}

pvs_status pvs_append(pvs_index* x, const float* vecs, int64_t n, int32_t vecs_on_device) {
    DeviceGuard device_guard(index_device(x));
    if (!x || n < 0 || (n > 0 && !vecs) || x->size + n >= ((int64_t)1 << 31))
        return PVS_ERR_INVALID;
    if (n == 0) return PVS_OK;
    if (vecs_on_device && !is_device_ptr(vecs)) return PVS_ERR_INVALID;
    pvs_status s = index_reserve(x, x->size + n);
    if (s != PVS_OK) return s;
    s = index_fill(x, vecs, n, vecs_on_device != 0);
    if (s != PVS_OK) return s;
    x->size += n;
    x->live += n;
    return refresh_norm_maxes(x);
}

pvs_status pvs_tombstone(pvs_index* x, const int64_t* ids, int64_t n) {
    DeviceGuard device_guard(index_device(x));
    if (!x || n < 0 || (n > 0 && !ids)) return PVS_ERR_INVALID;
    for (int64_t i = 0; i < n; ++i)
        if (ids[i] < 0 || ids[i] >= x->size) return PVS_ERR_INVALID;
    for (int64_t i = 0; i < n; ++i) {
        const int64_t id = ids[i];
        uint32_t& w = x->h_tomb[(size_t)(id >> 5)];
        const uint32_t b = 1u << (id & 31);
        if (!(w & b)) {
            w |= b;
            x->tombstoned++;
            x->live--;
        }
    }
    return PVS_OK;
}

int64_t pvs_index_size(const pvs_index* x) { return x ? x->size : -1; }
int64_t pvs_index_live(const pvs_index* x) { return x ? x->live : -1; }
int32_t pvs_index_dim(const pvs_index* x) { return x ? x->m : -1; }

pvs_status pvs_index_export(const pvs_index* x, int64_t first, int64_t count, int8_t* codes,
                            float* scale, float* vnorm, float* enorm) {
    DeviceGuard device_guard(index_device(x));
    if (!x || first < 0 || count < 0 || first + count > x->size) return PVS_ERR_INVALID;
    if (count == 0) return PVS_OK;
    if (codes)
        PVS_CUDA(cudaMemcpy2D(codes, (size_t)x->m, x->codes + first * x->m_pad, (size_t)x->m_pad,
                              (size_t)x->m, (size_t)count, cudaMemcpyDeviceToHost));
    if (scale)
        PVS_CUDA(cudaMemcpy(scale, x->scale + first, count * sizeof(float), cudaMemcpyDeviceToHost));
    if (vnorm)
        PVS_CUDA(cudaMemcpy(vnorm, x->vnorm + first, count * sizeof(float), cudaMemcpyDeviceToHost));
    if (enorm)
        PVS_CUDA(cudaMemcpy(enorm, x->enorm + first, count * sizeof(float), cudaMemcpyDeviceToHost));
    return PVS_OK;
}

void pvs_index_free(pvs_index* x) {
    DeviceGuard device_guard(index_device(x));
    if (!x) return;
    if (x->stream) cudaStreamSynchronize(x->stream);
    for (pvs_cursor* c : x->cursor_pool) {
        cursor_free_device(c);
        delete c;
    }
    x->cursor_pool.clear();
    x->pool_bytes = 0;
    dev_free(x->codes), dev_free(x->scale), dev_free(x->vnorm), dev_free(x->enorm);
    dev_free(x->raw), dev_free(x->d_status), dev_free(x->d_stage), dev_free(x->codes_bf16);
    if (x->pass_done) cudaEventDestroy(x->pass_done);
    if (x->scratch_pool) cudaMemPoolDestroy(x->scratch_pool);
    if (x->bf16_ready) cudaEventDestroy(x->bf16_ready);
    dev_free(x->resid), dev_free(x->rparam);
    if (x->resid_ready) cudaEventDestroy(x->resid_ready);
    dev_free(x->norm_maxes);
    dev_free(x->gscale);
    if (x->own_stream && x->stream) cudaStreamDestroy(x->stream);
    delete x;
}

pvs_status pvs_snapshot_create(pvs_index* x, pvs_snapshot** out) {
    DeviceGuard device_guard(index_device(x));
    if (!x || !out) return PVS_ERR_INVALID;
    *out = nullptr;
    auto d = make_snapdata(x);
    if (!d) return PVS_ERR_OOM;
    pvs_snapshot* s = new (std::nothrow) pvs_snapshot();
    if (!s) return PVS_ERR_OOM;
    s->index = x;
    s->data = std::move(d);
    *out = s;
    return PVS_OK;
}

int64_t pvs_snapshot_visible(const pvs_snapshot* s) { return s ? s->data->visible : -1; }

void pvs_snapshot_free(pvs_snapshot* s) {
    DeviceGuard device_guard(s ? index_device(s->index) : -1);
    delete s;
}

}  // extern "C"

// Open a cursor whose device work runs on `stream` from the start (null: the
// index's stream), ordered after the work queued so far on the index's stream.
pvs_status pvs::cursor_open_on(pvs_index* x, const pvs_snapshot* snap, const float* query,
                               int32_t query_on_device, cudaStream_t stream, pvs_cursor** out) {
    DeviceGuard device_guard(index_device(x));
    if (!out) return PVS_ERR_INVALID;
    *out = nullptr;
    if (!x || !query || (snap && snap->index != x)) return PVS_ERR_INVALID;
    if (query_on_device && !is_device_ptr(query)) return PVS_ERR_INVALID;
    pvs_cursor* c = nullptr;
    {
        std::lock_guard<std::mutex> lock(x->pool_mutex);
        if (!x->cursor_pool.empty()) {   // reuse a closed cursor's buffers
            c = x->cursor_pool.back();
            x->cursor_pool.pop_back();
            x->pool_bytes -= cursor_device_bytes(c);
        }
    }
    if (!c) {
        c = new (std::nothrow) pvs_cursor();
        if (!c) return PVS_ERR_OOM;
    }
    auto bail = [&](pvs_status s) {
        cursor_free_device(c);
        delete c;
        return s;
    };
    cursor_reset(c);
    c->index = x;
    c->stream = stream ? stream : x->stream;
    c->snap = snap ? snap->data : make_snapdata(x);
    if (!c->snap) return bail(PVS_ERR_OOM);
    c->rows = c->snap->rows;
    c->visible = c->snap->visible;
    cudaStream_t st = c->stream;
    if (!c->zq &&
        (dev_alloc(&c->zq, (size_t)x->m_pad) != cudaSuccess ||
         dev_alloc(&c->qraw, (size_t)x->m_raw) != cudaSuccess ||
         dev_alloc(&c->qs, 1) != cudaSuccess || dev_alloc(&c->sel, 1) != cudaSuccess ||
         dev_alloc(&c->ctr, 1) != cudaSuccess || dev_alloc(&c->d_status, 1) != cudaSuccess ||
         cudaMallocHost(&c->h_small, 16 * sizeof(unsigned int)) != cudaSuccess))
        return bail(PVS_ERR_OOM);
    cudaError_t e = cudaSuccess;
    if (st != x->stream) {   // after the index's queued builds and appends
        if (!c->ev_order) e = cudaEventCreateWithFlags(&c->ev_order, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventRecord(c->ev_order, x->stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(st, c->ev_order, 0);
        if (e != cudaSuccess) return bail(cuda_status(e));
    }
    // a host query is staged in the cursor's raw query buffer, which the
    // encoder then rewrites in place with the same values (plus zero padding)
    const float* qd = query;
    if (!query_on_device) {
        e = cudaMemcpyAsync(c->qraw, query, x->m * sizeof(float), cudaMemcpyHostToDevice, st);
        qd = c->qraw;
    }
    if (e == cudaSuccess) e = cudaMemsetAsync(c->ctr, 0, sizeof(DevCounters), st);
    if (e == cudaSuccess) e = cudaMemsetAsync(c->d_status, 0, sizeof(int), st);
    if (e == cudaSuccess) e = launch_encode_query(qd, x->m, x->m_pad, x->m_raw, c->zq, c->qraw, c->qs, st);
    int* enc_status = reinterpret_cast<int*>(c->h_small) + 3;   // pinned
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(enc_status, &c->qs->status, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return bail(cuda_status(e));
    if (*enc_status != 0) return bail((pvs_status)*enc_status);
    c->state = c->visible == 0 ? PVS_EXHAUSTED : PVS_OK;
    *out = c;
    return PVS_OK;
}

static_assert(pvs::kGroupMax == PVS_GROUP_MAX, "group size of the C ABI");

// SMs left free of the grouped pass.  Measured at 8.8M x 768 with eight
// queries per pass and eight groups in flight (ranks/s; pass ms): 0 SMs
// 4.78M (1.24 ms), 16 4.80M (1.19), 32 5.19M (1.22), 48 5.26M (1.29), 56
// 5.54M (1.40), 64 5.17M (1.51), 80 4.31M (1.82); 32 keeps the pass near
// the HBM roofline.
constexpr int kGroupReserveSms = 32;

namespace {

// One grouped interval pass for the nq (>= 2) freshly opened cursors cs[],
// which share one snapshot: their bounds and per-slot lower bounds, on
// stream `ps`; every cursor's own stream then waits for the pass.
pvs_status group_pass(pvs_index* x, pvs_cursor* const* cs, int nq, cudaStream_t ps) {
    IntervalGroupArgs a;
    a.codes = x->codes;
    a.scale = x->scale;
    a.vnorm = x->vnorm;
    a.enorm = x->enorm;
    a.tomb = cs[0]->snap->d_tomb;
    a.rows = cs[0]->rows;
    a.m_pad = x->m_pad;
    a.nq = nq;
    a.wait_ns = x->wait_ns;
    // the pass runs on all but kGroupReserveSms SMs: pulls and working-set
    // builds of other groups run beside it (the pass's shared memory and
    // registers leave no room for them on its own SMs)
    const int pass_sms = std::max(x->num_sms / 2, x->num_sms - kGroupReserveSms);
    int64_t min_rows = 0;
    const int64_t slots = interval_group_slots(a.rows, x->m_pad, nq, pass_sms, &min_rows);
    const bool use_slots = slots > 0 && a.tomb == nullptr && min_rows >= kSlotTop;
    for (int i = 0; i < nq; ++i) {
        pvs_cursor* c = cs[i];
        pvs_status s = cursor_alloc_rows(c);
        if (s != PVS_OK) return s;
        c->slot_fresh = false;
        c->slot_n = 0;
        a.slot_top[i] = nullptr;
        if (use_slots) {
            if (c->slot_cap < slots * kSlotTop) {
                dev_free(c->slot_top);
                c->slot_cap = 0;
                PVS_CUDA(dev_alloc(&c->slot_top, (size_t)(slots * kSlotTop)));
                c->slot_cap = slots * kSlotTop;
            }
            a.slot_top[i] = c->slot_top;
            c->slot_n = slots * kSlotTop;
        }
        a.zq[i] = c->zq;
        a.qs[i] = c->qs;
        a.lo[i] = c->lo;
        a.hi[i] = c->hi;
        a.bmax[i] = c->bmax;
        a.status[i] = c->d_status;
        if (!c->ev_begin) {
            PVS_CUDA(cudaEventCreate(&c->ev_begin));
            PVS_CUDA(cudaEventCreate(&c->ev_end));
        }
    }
    {
        // passes of one index run one after another (each saturates HBM)
        std::lock_guard<std::mutex> lock(x->pass_mutex);
        if (!x->pass_done)
            PVS_CUDA(cudaEventCreateWithFlags(&x->pass_done, cudaEventDisableTiming));
        else
            PVS_CUDA(cudaStreamWaitEvent(ps, x->pass_done, 0));
        for (int i = 0; i < nq; ++i) PVS_CUDA(cudaEventRecord(cs[i]->ev_begin, ps));
        PVS_CUDA(launch_interval_group(a, pass_sms, ps));
        for (int i = 0; i < nq; ++i) PVS_CUDA(cudaEventRecord(cs[i]->ev_end, ps));
        PVS_CUDA(cudaEventRecord(x->pass_done, ps));
    }
    for (int i = 0; i < nq; ++i) {
        pvs_cursor* c = cs[i];
        if (c->stream != ps) PVS_CUDA(cudaStreamWaitEvent(c->stream, c->ev_end, 0));
        c->slot_fresh = a.slot_top[i] != nullptr;
        c->ev_pending = true;
        c->interval_passes++;
        c->code_bytes += c->rows * (int64_t)(x->m_pad + 12) / nq;
        c->group_size = nq;
        c->scanned = true;
        c->bmax_valid = true;
    }
    if (x->wait_ns < kWaitLimitNs) {   // as in interval_pass: check before any pull
        PVS_CUDA(cudaStreamSynchronize(ps));
        for (int i = 0; i < nq; ++i) {
            pvs_status s = check_device_status(cs[i]);
            if (s != PVS_OK) return s;
        }
    }
    return PVS_OK;
}

}  // namespace

pvs_status pvs::cursor_open_group(pvs_index* x, const pvs_snapshot* snap, const float* queries,
                                  int32_t nq, int32_t queries_on_device, cudaStream_t pass_stream,
                                  const cudaStream_t* cursor_streams, pvs_cursor** out) {
    DeviceGuard device_guard(index_device(x));
    if (!out || nq < 1 || nq > kGroupMax) return PVS_ERR_INVALID;
    for (int i = 0; i < nq; ++i) out[i] = nullptr;
    if (!x || !queries || (snap && snap->index != x)) return PVS_ERR_INVALID;
    if (queries_on_device && !is_device_ptr(queries)) return PVS_ERR_INVALID;
    cudaStream_t ps = pass_stream ? pass_stream : x->stream;
    // one visible set for the whole group
    pvs_snapshot own;
    if (!snap) {
        own.index = x;
        own.data = make_snapdata(x);
        if (!own.data) return PVS_ERR_OOM;
        snap = &own;
    }
    pvs_cursor* cs[kGroupMax] = {nullptr};
    auto bail = [&](pvs_status s) {
        for (int i = 0; i < nq; ++i)
            if (cs[i]) pvs_cursor_close(cs[i]);
        return s;
    };
    for (int i = 0; i < nq; ++i) {
        cudaStream_t st = cursor_streams && cursor_streams[i] ? cursor_streams[i] : ps;
        pvs_status s = cursor_open_on(x, snap, queries + (int64_t)i * x->m, queries_on_device,
                                      st, &cs[i]);
        if (s != PVS_OK) return bail(s);
    }
    // one query, nothing visible, or rows the grouped pass does not serve:
    // each cursor runs its own pass at its first pull
    if (nq >= 2 && cs[0]->visible > 0 && interval_group_supported(x->m_pad, nq)) {
        // the pass runs on ps after every cursor's queued work (their queries)
        for (int i = 0; i < nq; ++i) {
            if (cs[i]->stream == ps) continue;
            cudaError_t e = cudaSuccess;
            if (!cs[i]->ev_order) e = cudaEventCreateWithFlags(&cs[i]->ev_order, cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventRecord(cs[i]->ev_order, cs[i]->stream);
            if (e == cudaSuccess) e = cudaStreamWaitEvent(ps, cs[i]->ev_order, 0);
            if (e != cudaSuccess) return bail(cuda_status(e));
        }
        pvs_status s = group_pass(x, cs, nq, ps);
        if (s != PVS_OK) {
            for (int i = 0; i < nq; ++i) fail(cs[i], s);
            return bail(s);
        }
    }
    for (int i = 0; i < nq; ++i) out[i] = cs[i];
    return PVS_OK;
}

extern "C" {

pvs_status pvs_cursor_open(pvs_index* x, const pvs_snapshot* snap, const float* query,
                           int32_t query_on_device, pvs_cursor** out) {
    return pvs::cursor_open_on(x, snap, query, query_on_device, nullptr, out);
}

pvs_status pvs_cursor_open_group(pvs_index* x, const pvs_snapshot* snap, const float* queries,
                                 int32_t nq, int32_t queries_on_device, void* pass_stream,
                                 void* const* cursor_streams, pvs_cursor** out) {
    return pvs::cursor_open_group(x, snap, queries, nq, queries_on_device,
                                  static_cast<cudaStream_t>(pass_stream),
                                  reinterpret_cast<const cudaStream_t*>(cursor_streams), out);
}

pvs_status pvs_cursor_open_batch(pvs_index* x, const pvs_snapshot* snap, const float* queries,
                                 int32_t nq, int32_t queries_on_device, int32_t horizon,
                                 void* cuda_stream, pvs_cursor** out) {
    DeviceGuard device_guard(index_device(x));
    if (!x || !queries || !out || nq < 0 || horizon < 1) return PVS_ERR_INVALID;
    if (queries_on_device && !is_device_ptr(queries)) return PVS_ERR_INVALID;
    for (int32_t i = 0; i < nq; ++i) out[i] = nullptr;
    std::shared_ptr<SnapData> sd = snap ? snap->data : make_snapdata(x);
    if (!sd) return PVS_ERR_OOM;
    for (int32_t g0 = 0; g0 < nq; g0 += kBatchMax) {
        const int32_t g = std::min<int32_t>(kBatchMax, nq - g0);
        pvs_status s = open_batch_group(x, sd, queries + (size_t)g0 * x->m, g,
                                        queries_on_device != 0, horizon,
                                        cuda_stream ? static_cast<cudaStream_t>(cuda_stream)
                                                    : x->stream,
                                        out + g0);
        if (s != PVS_OK) {
            for (int32_t j = 0; j < nq; ++j) {
                if (out[j]) pvs_cursor_close(out[j]);
                out[j] = nullptr;
            }
            return s;
        }
    }
    return PVS_OK;
}

pvs_status pvs_batch_bounds(pvs_index* x, const pvs_snapshot* snap, const float* queries,
                            int32_t nq, int32_t queries_on_device, float* lo, float* hi) {
    DeviceGuard device_guard(index_device(x));
    if (!x || !queries || !lo || !hi || nq < 1 || nq > kBatchMax) return PVS_ERR_INVALID;
    if (queries_on_device && !is_device_ptr(queries)) return PVS_ERR_INVALID;
    std::shared_ptr<SnapData> sd = snap ? snap->data : make_snapdata(x);
    if (!sd) return PVS_ERR_OOM;
    const int64_t rows = sd->rows;
    if (rows == 0) return PVS_OK;
    cudaStream_t st = x->stream;
    DevBuf buf(st, x->scratch_pool);
    BatchQueries bq;
    pvs_status s = encode_batch(x, queries, nq, queries_on_device, buf, &bq, st);
    if (s != PVS_OK) return s;
    const int64_t ntiles = (rows + 127) / 128;
    const int64_t ld = ntiles * 128;
    float* dlo = buf.get<float>((size_t)nq * ld);
    float* dhi = buf.get<float>((size_t)nq * ld);
    int* status = buf.get<int>(1);
    if (!dlo || !dhi || !status) return PVS_ERR_OOM;
    PVS_CUDA(cudaMemsetAsync(status, 0, sizeof(int), st));
    BatchArgs a{};
    a.rows = rows;
    a.m_pad = x->m_pad;
    a.nq = nq;
    a.nq_pad = bq.nq_pad;
    a.scale = x->scale;
    a.vnorm = x->vnorm;
    a.enorm = x->enorm;
    a.tomb = sd->d_tomb;
    a.qs = bq.qs;
    a.mode = 0;
    a.tile_stride = 1;
    a.dump_lo = dlo;
    a.dump_hi = dhi;
    a.dump_ld = ld;
    a.status = status;
    PVS_CUDA(launch_batch_intervals(a, x->codes_bf16, bq.qcodes, x->num_sms, st));
    int h_status = 0;
    PVS_CUDA(cudaMemcpyAsync(&h_status, status, sizeof(int), cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaMemcpy2DAsync(lo, rows * sizeof(float), dlo, ld * sizeof(float),
                               rows * sizeof(float), nq, cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaMemcpy2DAsync(hi, rows * sizeof(float), dhi, ld * sizeof(float),
                               rows * sizeof(float), nq, cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaStreamSynchronize(st));
    return (pvs_status)h_status;
}

}  // extern "C"

// The next n ranks of each of nc cursors (one index, one stream) in one set
// of launches; cursor i's ranks go to ids[i][0 .. n) and scores[i][0 .. n)
// (device or host per outputs_on_device).
// The cursor's state after a delivery: Exhausted once the caller has every rank.
static pvs_status delivery_state(pvs_cursor* c) {
    if (c->state >= 0 && c->emitted - c->ahead == c->visible) c->state = PVS_EXHAUSTED;
    return c->state == PVS_EXHAUSTED ? PVS_EXHAUSTED : PVS_OK;
}

// Ranks a pull computes for a request of `need` while nothing is ahead: up
// to `readahead` times the request (at most one fused launch's worth, and
// never past the list's end); large requests exactly.
static int64_t pull_size(const pvs_cursor* c, int64_t need, int32_t readahead) {
    if (need > kPullFusedMax) return need;
    const int64_t want = std::min<int64_t>(kPullFusedMax, need * std::max<int32_t>(1, readahead));
    return std::min<int64_t>(std::max(want, need), c->visible - c->emitted);
}

pvs_status pvs::next_batch_rows(pvs_cursor* const* cursors, int32_t nc, int32_t n,
                                int32_t outputs_on_device, int64_t* const* ids,
                                float* const* scores, int32_t* n_out) {
    DeviceGuard device_guard(first_cursor_device(const_cast<pvs_cursor**>(cursors), nc));
    if (!cursors || nc < 0 || n < 0 || !n_out || (nc > 0 && n > 0 && (!ids || !scores)))
        return PVS_ERR_INVALID;
    if (nc == 0) return PVS_OK;
    pvs_index* x = cursors[0] ? cursors[0]->index : nullptr;
    if (!x) return PVS_ERR_INVALID;
    cudaStream_t st = cursors[0]->stream;
    for (int32_t i = 0; i < nc; ++i) {
        n_out[i] = 0;
        if (!cursors[i] || cursors[i]->index != x || cursors[i]->stream != st ||
            cursors[i]->generator != PVS_GEN_INTERVALS || (n > 0 && (!ids[i] || !scores[i])))
            return PVS_ERR_INVALID;
    }
    for (int32_t i = 0; i < nc; ++i)
        if (cursors[i]->state < 0) return PVS_ERR_FAILED;
    if (n > kPullFusedMax) {   // large pulls: one cursor at a time
        for (int32_t i = 0; i < nc; ++i) {
            pvs_status s = outputs_on_device
                               ? pvs_next_device(cursors[i], n, ids[i], scores[i], &n_out[i])
                               : pvs_next(cursors[i], n, ids[i], scores[i], &n_out[i]);
            if (s < 0) return s;
        }
        return PVS_OK;
    }
    // per cursor: the ranks delivered now, first from those computed ahead
    // (take), then from this call's pull (rest), which computes pulls[i]
    std::vector<int64_t> take((size_t)nc), rest((size_t)nc), pulls((size_t)nc);
    std::vector<RankCopy> copies;
    bool host_async = false;   // device ranks copied to host rows, not yet waited for
    for (int32_t i = 0; i < nc; ++i) {
        pvs_cursor* c = cursors[i];
        const int64_t need = std::min<int64_t>(n, c->visible - (c->emitted - c->ahead));
        n_out[i] = (int32_t)need;
        take[i] = std::min(need, c->ahead);
        rest[i] = need - take[i];
        pulls[i] = rest[i] > 0 ? pull_size(c, rest[i], c->readahead) : 0;
        if (take[i] > 0) {
            const int64_t* si = (c->ahead_host ? c->h_ids : c->d_ids) + c->ahead_pos;
            const float* ss = (c->ahead_host ? c->h_scores : c->d_scores) + c->ahead_pos;
            if (outputs_on_device) {
                copies.push_back(RankCopy{si, ss, ids[i], scores[i], (int)take[i]});
            } else if (c->ahead_host) {
                std::memcpy(ids[i], si, take[i] * sizeof(int64_t));
                std::memcpy(scores[i], ss, take[i] * sizeof(float));
            } else {
                PVS_CUDA(cudaMemcpyAsync(ids[i], si, take[i] * sizeof(int64_t),
                                         cudaMemcpyDeviceToHost, st));
                PVS_CUDA(cudaMemcpyAsync(scores[i], ss, take[i] * sizeof(float),
                                         cudaMemcpyDeviceToHost, st));
                host_async = true;
            }
            c->ahead_pos += take[i];
            c->ahead -= take[i];
        }
    }
    // ranks taken from the buffers leave them before a pull refills them
    if (!copies.empty()) PVS_CUDA(launch_copy_ranks(copies.data(), (int)copies.size(), st));
    copies.clear();
    {
        pvs_status s = build_first_working_sets(cursors, nc, pulls.data());
        if (s != PVS_OK) return s;
    }
    std::vector<PullArgs> args;
    std::vector<int32_t> who;
    args.reserve(nc);
    for (int32_t i = 0; i < nc; ++i) {
        if (pulls[i] <= 0) continue;
        pvs_cursor* c = cursors[i];
        pvs_status s = cursor_out_reserve(c, pulls[i]);   // nothing is ahead now
        if (s != PVS_OK) return fail(c, s);
        s = prepare_pull(c, pulls[i]);
        if (s != PVS_OK) return fail(c, s);
        PullArgs a;
        a.w_id = c->w_id;
        a.w_lo = c->w_lo;
        a.w_hi = c->w_hi;
        a.w_len = &c->ctr->w_len;
        a.lo = c->scanned ? c->lo : nullptr;
        a.hi = c->scanned ? c->hi : nullptr;
        a.qraw = c->qraw;
        a.raw = x->raw;
        a.m_raw = x->m_raw;
        a.n = (int)pulls[i];
        a.cand = c->cand;
        a.keys = reinterpret_cast<unsigned long long*>(c->keys);
        // device outputs: the cursor's device buffers; host outputs: its
        // pinned buffers, which the kernels write directly
        a.out_ids = outputs_on_device ? c->d_ids : c->h_ids;
        a.out_scores = outputs_on_device ? c->d_scores : c->h_scores;
        a.status = c->d_status;
        a.ctr = c->ctr;
        a.front = nullptr;   // a few pulls per batch: a frontier would not pay for itself
        a.status_mirror = nullptr;
        args.push_back(a);
        who.push_back(i);
    }
    if (!args.empty()) {
        bool fresh = false;
        for (int32_t i : who) fresh = fresh || cursors[i]->fresh_ws;
        if (fresh) {   // first pull of new working sets: refinement on every SM
            const int per = std::min(64, std::max(4, 2 * x->num_sms / (int)args.size()));
            PVS_CUDA(launch_pull_batch(args.data(), (int)args.size(), per, x->m_raw, st));
        } else {
            PVS_CUDA(launch_pull_cluster_batch(args.data(), (int)args.size(), st));
        }
    }
    for (int32_t i : who) {
        pvs_cursor* c = cursors[i];
        c->emitted += pulls[i];
        c->pulls++;
        c->fresh_ws = false;
        c->ahead = pulls[i];
        c->ahead_pos = 0;
        c->ahead_host = !outputs_on_device;
    }
    if (outputs_on_device) {
        for (int32_t i : who) {
            pvs_cursor* c = cursors[i];
            copies.push_back(RankCopy{c->d_ids, c->d_scores, ids[i] + take[i],
                                      scores[i] + take[i], (int)rest[i]});
        }
        if (!copies.empty()) PVS_CUDA(launch_copy_ranks(copies.data(), (int)copies.size(), st));
    } else {
        if (!who.empty()) {
            std::vector<pvs_cursor*> pulled;
            for (int32_t i : who) pulled.push_back(cursors[i]);
            std::vector<int> dev_status(pulled.size(), 0);
            pvs_status s = gather_state(pulled.data(), (int)pulled.size(), st, dev_status.data(),
                                        nullptr);   // also waits for the pulls' outputs
            if (s != PVS_OK) return s;
            pvs_status result = PVS_OK;
            for (size_t j = 0; j < pulled.size(); ++j)
                if (dev_status[j] != 0) result = fail(pulled[j], (pvs_status)dev_status[j]);
            if (result != PVS_OK) return result;
            for (int32_t i : who) {
                pvs_cursor* c = cursors[i];
                std::memcpy(ids[i] + take[i], c->h_ids, rest[i] * sizeof(int64_t));
                std::memcpy(scores[i] + take[i], c->h_scores, rest[i] * sizeof(float));
            }
        } else if (host_async) {
            PVS_CUDA(cudaStreamSynchronize(st));
        }
    }
    for (int32_t i : who) {
        cursors[i]->ahead_pos = rest[i];
        cursors[i]->ahead -= rest[i];
    }
    for (int32_t i = 0; i < nc; ++i) delivery_state(cursors[i]);
    return PVS_OK;
}

extern "C" {

pvs_status pvs_next_batch(pvs_cursor** cursors, int32_t nc, int32_t n, int32_t outputs_on_device,
                          int64_t* ids, float* scores, int32_t* n_out) {
    if (!cursors || nc < 0 || n < 0 || !n_out || (nc > 0 && n > 0 && (!ids || !scores)))
        return PVS_ERR_INVALID;
    std::vector<int64_t*> id_rows((size_t)std::max(nc, 1));
    std::vector<float*> score_rows((size_t)std::max(nc, 1));
    for (int32_t i = 0; i < nc; ++i) {
        id_rows[(size_t)i] = ids ? ids + (int64_t)i * n : nullptr;
        score_rows[(size_t)i] = scores ? scores + (int64_t)i * n : nullptr;
    }
    return pvs::next_batch_rows(cursors, nc, n, outputs_on_device, id_rows.data(),
                                score_rows.data(), n_out);
}

static pvs_status next_common(pvs_cursor* c, int32_t n, int32_t* n_out, int64_t* n_eff) {
    *n_eff = 0;
    if (n_out) *n_out = 0;
    if (!c || n < 0 || !n_out) return PVS_ERR_INVALID;
    if (c->state < 0) return PVS_ERR_FAILED;
    const int64_t remaining = c->visible - (c->emitted - c->ahead);
    *n_eff = std::min<int64_t>(n, remaining);
    return PVS_OK;
}

// A pull of r >= 1 ranks into the cursor's pinned buffers at [at, at + r);
// they become the ranks ahead (ahead_pos = at).  The buffers must already
// hold at + r entries when at > 0 (they are only reallocated while empty).
static pvs_status pull_to_pinned(pvs_cursor* c, int64_t r, int64_t at = 0) {
    pvs_status s;
    if (at == 0) {
        s = cursor_out_reserve(c, r);
        if (s != PVS_OK) return fail(c, s);
    } else if (at + r > c->out_cap) {
        return fail(c, PVS_ERR_INVALID);   // internal invariant
    }
    if (r <= kPullFusedMax) {
        // the kernels write ids, scores and the status word straight into the
        // cursor's pinned host buffers: one launch, one wait
        int* mirror = reinterpret_cast<int*>(c->h_small) + 2;
        *reinterpret_cast<volatile int*>(mirror) = kStatusPending;
        s = pull(c, r, c->h_ids + at, c->h_scores + at, mirror);
        if (s != PVS_OK) return s;
        if (!wait_published(mirror)) {
            // nothing published within the limit: an asynchronous error, or a
            // very slow pull; the stream decides
            cudaError_t e = cudaStreamSynchronize(c->stream);
            if (e != cudaSuccess) return fail(c, cuda_status(e));
        }
        harvest_interval_time(c);
        const int dev_status = *reinterpret_cast<volatile int*>(mirror);
        if (dev_status != 0) return fail(c, (pvs_status)dev_status);
    } else {
        s = pull(c, r, c->d_ids + at, c->d_scores + at);
        if (s != PVS_OK) return s;
        cudaStream_t st = c->stream;
        cudaError_t e = cudaMemcpyAsync(c->h_ids + at, c->d_ids + at, r * sizeof(int64_t),
                                        cudaMemcpyDeviceToHost, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(c->h_scores + at, c->d_scores + at, r * sizeof(float),
                                cudaMemcpyDeviceToHost, st);
        if (e != cudaSuccess) return fail(c, cuda_status(e));
        s = check_device_status(c);
        if (s != PVS_OK) return s;
    }
    c->ahead = r;
    c->ahead_pos = at;
    c->ahead_host = true;
    return PVS_OK;
}

// Ranks ahead in the device buffers moved to the front of the pinned ones.
static pvs_status ahead_to_host(pvs_cursor* c) {
    if (c->ahead == 0) {
        c->ahead_pos = 0;
        c->ahead_host = true;
        return PVS_OK;
    }
    if (c->ahead_host) {
        if (c->ahead_pos > 0) {
            std::memmove(c->h_ids, c->h_ids + c->ahead_pos, c->ahead * sizeof(int64_t));
            std::memmove(c->h_scores, c->h_scores + c->ahead_pos, c->ahead * sizeof(float));
        }
    } else {
        cudaStream_t st = c->stream;
        cudaError_t e = cudaMemcpyAsync(c->h_ids, c->d_ids + c->ahead_pos,
                                        c->ahead * sizeof(int64_t), cudaMemcpyDeviceToHost, st);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(c->h_scores, c->d_scores + c->ahead_pos, c->ahead * sizeof(float),
                                cudaMemcpyDeviceToHost, st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(st);
        if (e != cudaSuccess) return fail(c, cuda_status(e));
    }
    c->ahead_pos = 0;
    c->ahead_host = true;
    return PVS_OK;
}

pvs_status pvs_next(pvs_cursor* c, int32_t n, int64_t* ids, float* scores, int32_t* n_out) {
    DeviceGuard device_guard(cursor_device(c));
    int64_t n_eff;
    pvs_status s = next_common(c, n, n_out, &n_eff);
    if (s != PVS_OK) return s;
    if (n_eff > 0 && (!ids || !scores)) return PVS_ERR_INVALID;
    int64_t off = 0;
    while (off < n_eff) {
        if (c->ahead == 0) {
            s = pull_to_pinned(c, pull_size(c, n_eff - off, c->readahead));
            if (s < 0) return s;
        } else if (!c->ahead_host) {
            s = ahead_to_host(c);
            if (s < 0) return s;
        }
        const int64_t take = std::min(n_eff - off, c->ahead);
        std::memcpy(ids + off, c->h_ids + c->ahead_pos, take * sizeof(int64_t));
        std::memcpy(scores + off, c->h_scores + c->ahead_pos, take * sizeof(float));
        c->ahead_pos += take;
        c->ahead -= take;
        off += take;
    }
    *n_out = (int32_t)n_eff;
    return delivery_state(c);
}

}  // extern "C"

// The next n ranks in the cursor's pinned buffers, for host code of this
// library that reads them once (the EAHR driver): *ids and *scores point
// there and stay valid until the cursor's next pull.  As pvs_next, without
// read-ahead (the driver sizes its pulls itself).
pvs_status pvs::next_pinned(pvs_cursor* c, int32_t n, const int64_t** ids, const float** scores,
                            int32_t* n_out) {
    DeviceGuard device_guard(cursor_device(c));
    int64_t n_eff;
    pvs_status s = next_common(c, n, n_out, &n_eff);
    if (s != PVS_OK) return s;
    if (!ids || !scores) return PVS_ERR_INVALID;
    if (n_eff > c->ahead) {
        if (c->ahead == 0) {
            s = pull_to_pinned(c, n_eff);
        } else {
            // ranks a pvs_next left ahead come first, the rest right after them
            s = ahead_to_host(c);
            if (s == PVS_OK && c->ahead + (n_eff - c->ahead) > c->out_cap) {
                std::vector<int64_t> keep_ids(c->h_ids, c->h_ids + c->ahead);
                std::vector<float> keep_sc(c->h_scores, c->h_scores + c->ahead);
                const int64_t k = c->ahead;
                c->ahead = 0;
                s = cursor_out_reserve(c, n_eff);
                if (s == PVS_OK) {
                    std::memcpy(c->h_ids, keep_ids.data(), k * sizeof(int64_t));
                    std::memcpy(c->h_scores, keep_sc.data(), k * sizeof(float));
                    c->ahead = k;
                } else {
                    fail(c, s);
                }
            }
            if (s == PVS_OK) {
                const int64_t k = c->ahead;
                s = pull_to_pinned(c, n_eff - k, k);
                c->ahead += k;
                c->ahead_pos = 0;
            }
        }
        if (s < 0) return s;
    } else if (!c->ahead_host) {
        s = ahead_to_host(c);
        if (s < 0) return s;
    }
    *ids = c->h_ids + c->ahead_pos;
    *scores = c->h_scores + c->ahead_pos;
    c->ahead_pos += n_eff;
    c->ahead -= n_eff;
    *n_out = (int32_t)n_eff;
    return delivery_state(c);
}

extern "C" {

pvs_status pvs_next_device(pvs_cursor* c, int32_t n, int64_t* ids, float* scores,
                           int32_t* n_out) {
    DeviceGuard device_guard(cursor_device(c));
    int64_t n_eff;
    pvs_status s = next_common(c, n, n_out, &n_eff);
    if (s != PVS_OK) return s;
    if (n_eff > 0 && (!ids || !scores)) return PVS_ERR_INVALID;
    int64_t off = 0;
    RankCopy copies[2];
    int ncopy = 0;
    while (off < n_eff) {
        if (c->ahead == 0) {
            const int64_t r = pull_size(c, n_eff - off, c->readahead);
            if (r > kPullFusedMax) {   // a large pull goes straight to the caller
                if (ncopy) {
                    PVS_CUDA(launch_copy_ranks(copies, ncopy, c->stream));
                    ncopy = 0;
                }
                s = pull(c, r, ids + off, scores + off);
                if (s != PVS_OK) return s;
                off += r;
                break;
            }
            if (ncopy) {   // the buffer is reused: earlier copies first
                PVS_CUDA(launch_copy_ranks(copies, ncopy, c->stream));
                ncopy = 0;
            }
            s = cursor_out_reserve(c, r);
            if (s != PVS_OK) return fail(c, s);
            s = pull(c, r, c->d_ids, c->d_scores);
            if (s != PVS_OK) return s;
            c->ahead = r;
            c->ahead_pos = 0;
            c->ahead_host = false;
        }
        const int64_t take = std::min(n_eff - off, c->ahead);
        const int64_t* src_i = (c->ahead_host ? c->h_ids : c->d_ids) + c->ahead_pos;
        const float* src_s = (c->ahead_host ? c->h_scores : c->d_scores) + c->ahead_pos;
        copies[ncopy++] = RankCopy{src_i, src_s, ids + off, scores + off, (int)take};
        c->ahead_pos += take;
        c->ahead -= take;
        off += take;
    }
    if (ncopy) PVS_CUDA(launch_copy_ranks(copies, ncopy, c->stream));
    *n_out = (int32_t)n_eff;
    return delivery_state(c);
}

pvs_status pvs_cursor_set_readahead(pvs_cursor* c, int32_t pages) {
    if (!c || pages < 1) return PVS_ERR_INVALID;
    c->readahead = pages;
    return PVS_OK;
}

pvs_status pvs_cursor_sync(pvs_cursor* c) {
    DeviceGuard device_guard(cursor_device(c));
    if (!c) return PVS_ERR_INVALID;
    if (c->state < 0) return (pvs_status)c->state;
    pvs_status s = check_device_status(c);
    if (s != PVS_OK) return s;
    return (pvs_status)c->state;
}

static void fill_stats(pvs_cursor* c, const DevCounters& d, pvs_stats* out) {
    std::memset(out, 0, sizeof(*out));
    out->visible = c->visible;
    out->emitted = c->emitted - c->ahead;   // delivered to the caller
    out->refined = (int64_t)d.refined;
    out->exact_fallbacks = (int64_t)d.exact_fallbacks;
    out->interval_passes = c->interval_passes;
    out->horizon_builds = c->horizon_builds;
    out->pulls = c->pulls;
    out->candidates = c->candidates + (int64_t)d.cand_total;
    out->code_bytes = c->code_bytes;
    out->state = c->state;
    harvest_interval_time(c);
    out->interval_ms = c->interval_ms;
    out->batch_passes = c->batch_passes;
    out->batch_ms = c->batch_ms;
}

pvs_status pvs_cursor_stats(pvs_cursor* c, pvs_stats* out) {
    DeviceGuard device_guard(cursor_device(c));
    if (!c || !out) return PVS_ERR_INVALID;
    std::memset(out, 0, sizeof(*out));
    DevCounters d{};
    cudaError_t e = cudaMemcpyAsync(&d, c->ctr, sizeof(d), cudaMemcpyDeviceToHost, c->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) return cuda_status(e);
    if (c->state >= 0) check_device_status(c);
    fill_stats(c, d, out);
    return PVS_OK;
}

static bool valid_cursor_list(pvs_cursor* const* cs, int32_t nc) {
    if (!cs || nc < 0) return false;
    for (int32_t i = 0; i < nc; ++i)
        if (!cs[i] || !cs[i]->index) return false;
    return true;
}

pvs_status pvs_cursor_sync_batch(pvs_cursor** cursors, int32_t nc, int32_t* states) {
    DeviceGuard device_guard(first_cursor_device(cursors, nc));
    if (!valid_cursor_list(cursors, nc) || (nc > 0 && !states)) return PVS_ERR_INVALID;
    std::vector<int> dev_status((size_t)nc, 0);
    pvs_status s = gather_state_any(cursors, nc, dev_status.data(), nullptr);
    if (s != PVS_OK) return s;
    for (int32_t i = 0; i < nc; ++i) {
        pvs_cursor* c = cursors[i];
        if (c->state >= 0 && dev_status[(size_t)i] != 0) fail(c, (pvs_status)dev_status[(size_t)i]);
        states[i] = c->state;
    }
    return PVS_OK;
}

pvs_status pvs_cursor_stats_batch(pvs_cursor** cursors, int32_t nc, pvs_stats* out) {
    DeviceGuard device_guard(first_cursor_device(cursors, nc));
    if (!valid_cursor_list(cursors, nc) || (nc > 0 && !out)) return PVS_ERR_INVALID;
    std::vector<int> dev_status((size_t)nc, 0);
    std::vector<DevCounters> d((size_t)nc, DevCounters{});
    pvs_status s = gather_state_any(cursors, nc, dev_status.data(), d.data());
    if (s != PVS_OK) return s;
    for (int32_t i = 0; i < nc; ++i) {
        pvs_cursor* c = cursors[i];
        if (c->state >= 0 && dev_status[(size_t)i] != 0) fail(c, (pvs_status)dev_status[(size_t)i]);
        fill_stats(c, d[(size_t)i], &out[i]);
    }
    return PVS_OK;
}

pvs_status pvs_cursor_bounds(pvs_cursor* c, int64_t first, int64_t count, float* lo,
                             float* hi) {
    DeviceGuard device_guard(cursor_device(c));
    if (!c || first < 0 || count < 0 || first + count > c->rows || (count > 0 && (!lo || !hi)) ||
        c->generator != PVS_GEN_INTERVALS)
        return PVS_ERR_INVALID;
    if (c->state < 0) return PVS_ERR_FAILED;
    pvs_status s = PVS_OK;
    if (c->batch_ws) {
        s = rescan_from_batch(c);
        if (s != PVS_OK) return fail(c, s);
    } else if (!c->scanned) {
        s = cursor_alloc_rows(c);
        if (s != PVS_OK) return fail(c, s);
        s = interval_pass(c);
        if (s != PVS_OK) return fail(c, s);
    }
    s = check_device_status(c);
    if (s != PVS_OK) return s;
    if (count == 0) return PVS_OK;
    cudaStream_t st = c->stream;
    PVS_CUDA(cudaMemcpyAsync(lo, c->lo + first, count * sizeof(float), cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaMemcpyAsync(hi, c->hi + first, count * sizeof(float), cudaMemcpyDeviceToHost, st));
    PVS_CUDA(cudaStreamSynchronize(st));
    return PVS_OK;
}

pvs_status pvs_cursor_score_ids(pvs_cursor* c, const int64_t* ids, int32_t n, float* scores) {
    DeviceGuard device_guard(cursor_device(c));
    if (!c || n < 0 || (n > 0 && (!ids || !scores))) return PVS_ERR_INVALID;
    for (int32_t i = 0; i < n; ++i)
        if (ids[i] < 0 || ids[i] >= c->rows) return PVS_ERR_INVALID;
    if (n == 0) return PVS_OK;
    cudaStream_t st = c->stream;
    int64_t* d_ids = nullptr;
    float* d_out = nullptr;
    cudaError_t e = dev_alloc(&d_ids, (size_t)n);
    if (e == cudaSuccess) e = dev_alloc(&d_out, (size_t)n);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(d_ids, ids, n * sizeof(int64_t), cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess)
        e = launch_score_ids(d_ids, n, c->qraw, c->index->raw, c->index->m_raw, d_out, c->ctr, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(scores, d_out, n * sizeof(float), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    dev_free(d_ids);
    dev_free(d_out);
    return cuda_status(e);
}

// Return a cursor's buffers to its index's pool (or free them); the caller
// has waited for the cursor's stream.
static void release_cursor(pvs_cursor* c) {
    pvs_index* x = c->index;
    harvest_interval_time(c);
    if (x) {
        std::lock_guard<std::mutex> lock(x->pool_mutex);
        const size_t bytes = cursor_device_bytes(c);
        if (x->cursor_pool.size() < kCursorPool &&
            x->pool_bytes + bytes <= x->pool_limit) {   // keep the buffers for the next cursor
            x->pool_bytes += bytes;
            cursor_reset(c);
            x->cursor_pool.push_back(c);
            return;
        }
    }
    cursor_free_device(c);
    delete c;
}

void pvs_cursor_close(pvs_cursor* c) {
    DeviceGuard device_guard(cursor_device(c));
    if (!c) return;
    if (c->index) cudaStreamSynchronize(c->stream);
    release_cursor(c);
}

void pvs_cursor_close_batch(pvs_cursor** cursors, int32_t nc) {
    DeviceGuard device_guard(first_cursor_device(cursors, nc));
    if (!cursors || nc <= 0) return;
    std::vector<cudaStream_t> synced;
    for (int32_t i = 0; i < nc; ++i) {
        pvs_cursor* c = cursors[i];
        if (!c || !c->index) continue;
        if (std::find(synced.begin(), synced.end(), c->stream) == synced.end()) {
            cudaStreamSynchronize(c->stream);
            synced.push_back(c->stream);
        }
    }
    for (int32_t i = 0; i < nc; ++i)
        if (cursors[i]) release_cursor(cursors[i]);
}

}  // extern "C"
