// Internal host-side structures of libpvs.so (index, snapshot, cursor).
#pragma once

#include <cstdint>
#include <memory>
#include <mutex>
#include <vector>

#include <cuda_runtime.h>

#include "../../include/pvs.h"
#include "kernels.h"

namespace pvs {

struct SnapData {
    int64_t rows = 0;                 // rows [0, rows) exist in the snapshot
    int64_t visible = 0;              // rows minus tombstones
    std::vector<uint32_t> h_tomb;     // tombstone bits of rows [0, rows)
    uint32_t* d_tomb = nullptr;       // device copy, null if nothing is deleted
    ~SnapData();
    bool is_visible(int64_t id) const {
        if (id < 0 || id >= rows) return false;
        if (h_tomb.empty()) return true;
        return ((h_tomb[(size_t)(id >> 5)] >> (id & 31)) & 1u) == 0;
    }
};

}  // namespace pvs

struct pvs_index {
    int device = 0;
    int num_sms = 0;
    int m = 0, m_pad = 0, m_raw = 0;
    int64_t size = 0, cap = 0, live = 0;
    int8_t* codes = nullptr;          // [cap][m_pad]
    float* scale = nullptr;           // [cap]
    float* vnorm = nullptr;           // [cap]
    float* enorm = nullptr;           // [cap]
    float* raw = nullptr;             // [cap][m_raw]
    std::vector<uint32_t> h_tomb;     // [cap/32]
    int64_t tombstoned = 0;
    cudaStream_t stream = nullptr;
    bool own_stream = false;
    int* d_status = nullptr;
    float* d_stage = nullptr;         // host-input staging
    size_t stage_floats = 0;
    std::vector<pvs_cursor*> cursor_pool;   // closed cursors whose buffers are reused
    size_t pool_bytes = 0;                  // device bytes held by pooled cursors
    size_t pool_limit = 0;                  // at most this many (a quarter of the device)
    std::mutex pool_mutex;                  // cursors may open / close on several threads
    std::mutex pass_mutex;                  // orders interval passes of this index
    cudaEvent_t pass_done = nullptr;        // end of the last interval pass queued
    // bf16 copy of the codes for the tensor-core batched pass (built on demand)
    uint16_t* codes_bf16 = nullptr;         // [cap][m_pad]
    int64_t bf16_rows = 0;                  // rows converted so far
    cudaEvent_t bf16_ready = nullptr;       // end of the last conversion (any stream)
    // 4-bit codes of each row's quantization residual, for the exact rank
    // counts of the EAHR finish (built on demand, extended over appended
    // rows): v = scale z + rscale z2 + r2 with ||r2|| <= rnorm, z2 in [-7, 7]
    // stored as z2 + 8, two per byte (dims 8t + k: byte k / 2 of word t, the
    // low nibble for even k); rparam[row] = (scale, rscale, rnorm, wnorm) with
    // wnorm >= ||scale z + rscale z2||
    uint8_t* resid = nullptr;               // [cap][m_pad / 2]
    float4* rparam = nullptr;               // [cap]
    int64_t resid_rows = 0;                 // rows coded so far
    cudaEvent_t resid_ready = nullptr;      // end of the last residual build (any stream)
    std::mutex resid_mutex;
    // max vnorm and max enorm (float bits) over every row; refreshed by build and
    // append (upper bounds for any snapshot), read by the batched pass
    unsigned int* norm_maxes = nullptr;
    // stream-ordered scratch of batched calls; keeps its memory between calls
    // (the device's default pool hands memory back at every synchronisation)
    cudaMemPool_t scratch_pool = nullptr;
    // scalar-quantization intervals: one scale for every row (else null)
    int quant = PVS_QUANT_PER_VECTOR;
    float* gscale = nullptr;                // device, one float
    // device-side wait limit of this index's interval passes (ns; 0: no wait)
    unsigned long long wait_ns = pvs::kWaitLimitNs;
};

struct pvs_snapshot {
    pvs_index* index = nullptr;
    std::shared_ptr<pvs::SnapData> data;
};

struct pbm_cursor;

struct pvs_cursor {
    pvs_index* index = nullptr;
    cudaStream_t stream = nullptr;    // where this cursor's device work runs
    std::shared_ptr<pvs::SnapData> snap;
    int64_t rows = 0, visible = 0, emitted = 0;
    int state = PVS_OK;
    bool scanned = false;
    // query
    int8_t* zq = nullptr;
    float* qraw = nullptr;
    pvs::QueryScalars* qs = nullptr;
    // bounds of every row of the snapshot (buffers hold cap_rows rows)
    int64_t cap_rows = 0;
    float* lo = nullptr;
    float* hi = nullptr;
    // the largest hi of each 16-row block, written by a grouped pass (upper
    // bounds of hi from then on: refinement and delivery only lower hi)
    float* bmax = nullptr;
    bool bmax_valid = false;
    // working set (ordered by id): rows that can hold the next `horizon` ranks
    int64_t cap_w = 0;                // capacity of the working-set arrays
    bool batch_ws = false;            // working set came from a batched pass (no full bounds)
    bool fresh_ws = false;            // no pull since the working set was built (many candidates)
    int32_t* w_id = nullptr;
    float* w_lo = nullptr;
    float* w_hi = nullptr;
    int64_t horizon = 0, horizon_base = 0;
    unsigned int* compact_scratch = nullptr;
    // the interval pass's largest lower bounds per row slot (kSlotTop each):
    // while fresh (the pass's bounds unchanged, every slot holding at least
    // kSlotTop live rows), the H-th largest of them bounds the H-th largest
    // lower bound of all rows from below
    float* slot_top = nullptr;
    int64_t slot_cap = 0, slot_n = 0;
    bool slot_fresh = false;
    // pull scratch
    int32_t* cand = nullptr;
    int32_t* front = nullptr;         // frontier of the one-launch pull (kFrontCap entries)
    uint64_t* keys = nullptr;
    uint64_t* keys_tmp = nullptr;
    void* sort_scratch = nullptr;
    pvs::SelectState* sel = nullptr;
    pvs::DevCounters* ctr = nullptr;
    int* d_status = nullptr;
    // output staging
    int64_t* d_ids = nullptr;
    float* d_scores = nullptr;
    int64_t out_cap = 0;
    int64_t* h_ids = nullptr;         // pinned
    float* h_scores = nullptr;        // pinned
    // ranks computed ahead of the caller (Sec. 2.1: the list is a stable
    // prefix, so a rank computed early is the rank delivered later): they sit
    // at [ahead_pos, ahead_pos + ahead) of h_ids / h_scores when ahead_host,
    // else of d_ids / d_scores.  `emitted` counts them; the caller has
    // received emitted - ahead ranks.
    int64_t ahead = 0, ahead_pos = 0;
    bool ahead_host = false;
    int32_t readahead = 4;            // a pull computes up to this many pages
    unsigned int* h_small = nullptr;  // pinned scratch (counts, status)
    // rank queries (fusion.cu): pinned staging, a second stream and an
    // event, kept between calls
    void* rq_pinned = nullptr;
    cudaStream_t rq_stream = nullptr;
    cudaEvent_t rq_event = nullptr;
    // stats
    int64_t pulls = 0, interval_passes = 0, horizon_builds = 0, candidates = 0;
    int64_t code_bytes = 0;           // code + parameter bytes read for this cursor (a
                                      // grouped pass's bytes are split among its queries)
    int32_t group_size = 1;           // queries that shared the cursor's interval pass
    int64_t batch_passes = 0;         // batched (tensor-core) passes this cursor took part in
    double batch_ms = 0.0;            // device time of that pass (shared by its cursors)
    cudaEvent_t ev_begin = nullptr, ev_end = nullptr;   // around the last interval pass
    cudaEvent_t ev_order = nullptr;   // orders a cursor's own stream after the index's
    bool ev_pending = false;
    double interval_ms = 0.0;
    // rank generator (PVS_GEN_*); exhaustive scanning keeps every row's key, sorted
    int generator = PVS_GEN_INTERVALS;
    bool scan_ready = false;
    uint64_t* scan_keys = nullptr;
    uint64_t* scan_tmp = nullptr;
    void* scan_scratch = nullptr;
    int64_t scan_cap = 0;
};

namespace pvs {
// Accessors used by the EAHR driver.
int64_t cursor_visible(const pvs_cursor* c);
int64_t cursor_emitted(const pvs_cursor* c);
const SnapData* cursor_snapshot(const pvs_cursor* c);
// pvs_next with the ranks left in the cursor's pinned buffers (valid until
// its next pull) instead of copied out.
pvs_status next_pinned(pvs_cursor* c, int32_t n, const int64_t** ids, const float** scores,
                       int32_t* n_out);
// Complete-list weighted RRF on the device (fusion.cu).  Per list i the
// contribution of rank r is a[i] / (b[i] r + c[i]) (0 when a[i] == 0).
struct FuseWeights {
    double a[2], b[2], c[2];
};
// One item near the top of the fused order: the binary32 value of its fused
// score (bits), its id and its ranks in the two lists (0: not in the list).
struct FusedCand {
    uint32_t fbits;
    int32_t id, rd, rs;
};
// The candidates for T*_K of the complete dense ranking of `dense`'s query
// over its snapshot and the host sparse list: every item of T*_K is among
// them, in descending binary32 fused-score order (the caller orders them
// exactly).  Does not use or change the cursor's ranked state.  Errors:
// PVS_ERR_INVALID (a sparse id outside the snapshot, deleted or repeated),
// PVS_ERR_OVERFLOW, PVS_ERR_OOM, PVS_ERR_CUDA.
pvs_status fuse_complete(pvs_cursor* dense, const int64_t* sparse, int64_t ns,
                         const FuseWeights& w, int32_t K, std::vector<FusedCand>* out);
// Ranks of a few items (fusion.cu).  Dense: row dense_ids[i]'s rank in the
// complete dense ranking of `dense`'s query over its snapshot (1-based) lies
// in [dense_lo[i], dense_hi[i]]; with `exact` the two are equal, else they
// come from the rows' intervals alone (no row is scored exactly; the item's
// own row may be counted in the width).  Sparse: sparse_rank[i] = the
// position + 1 of sparse_ids[i] in the host list `sparse` (0: not in it).
// The dense items must be visible and not yet delivered by the cursor, and
// the cursor must hold no ranks computed ahead of delivery.  *supported is
// false, and nothing runs, when the cursor keeps no bounds of every row (a
// batched working set, the full-scan generator).  At most kRankQueryMax
// items per list.  Errors: PVS_ERR_INVALID (a bad argument, or a sparse id
// outside the snapshot, deleted or repeated), PVS_ERR_INTERVAL (an exact
// score outside its interval), PVS_ERR_OVERFLOW, PVS_ERR_OOM, PVS_ERR_CUDA.
constexpr int32_t kRankQueryMax = 1024;
// A sparse list on the device ahead of need.  From a host list
// (stage_sparse_list): the ids copied, and checked as in fuse_complete (the
// verdict is read when the ranks are used); rank_queries finds its ids in the
// list.  From a PBM query (pbm_stage_ranks): rank_of[x] = position + 1 of id
// x (0: not in the list).  Built on its own stream (stage_sparse_list may hold
// the calling thread while the pageable list is copied); rank_queries orders
// its reads after it.
struct StagedList {
    pvs_index* index = nullptr;       // device and scratch pool
    cudaStream_t stream = nullptr;
    cudaEvent_t ready = nullptr;      // recorded after the scatter
    int32_t* rank_of = nullptr;       // [rows], or null: look the ids up in `list`
    int64_t* list = nullptr;          // the list's ids on the device (or null)
    uint32_t* seen = nullptr;         // a bit per id, set by the check of `list`
    const uint32_t* tomb = nullptr;   // the snapshot's deletions, for the check
    int64_t n = 0;                    // ids in `list`
    bool checked = true;              // the check of `list` is queued
    int* status = nullptr;            // the scatter's verdict on the ids
    int64_t rows = 0;
};
pvs_status stage_sparse_list(pvs_cursor* dense, const int64_t* sparse, int64_t ns,
                             StagedList** out);
// Queue the check of a list staged by stage_sparse_list (once; `ready` then
// marks its end).  Kept apart so that its kernel need not run beside the
// dense list's interval pass.
pvs_status check_staged_list(StagedList* s);
// The complete ranking of a PBM cursor's query (U_s = the visible items with
// S > 0, by (S desc, id asc), S evaluated as the PBM kernels do, App. A.2)
// staged the same way (pbm_capi.cu); scratch from pool_owner's pool.
pvs_status pbm_stage_ranks(pbm_cursor* sparse, pvs_index* pool_owner, StagedList** out);
void free_staged_list(StagedList* s);
// `staged` (or null): the same list, already scattered.
pvs_status rank_queries(pvs_cursor* dense, const int32_t* dense_ids, int32_t nd, bool exact,
                        const int64_t* sparse, int64_t ns, const int32_t* sparse_ids, int32_t nsq,
                        int64_t* dense_lo, int64_t* dense_hi, int64_t* sparse_rank,
                        bool* supported, const StagedList* staged = nullptr);
// pvs_next_batch with each cursor's outputs at its own address: cursor i's
// next n ranks to ids[i], scores[i] (device or host per outputs_on_device).
pvs_status next_batch_rows(pvs_cursor* const* cursors, int32_t nc, int32_t n,
                           int32_t outputs_on_device, int64_t* const* ids, float* const* scores,
                           int32_t* n_out);
// Open nq <= kGroupMax cursors whose bounds come from one grouped interval
// pass on pass_stream (null: the index's stream); cursor i's later work runs
// on cursor_streams[i] (null array or entry: pass_stream).
pvs_status cursor_open_group(pvs_index* x, const pvs_snapshot* snap, const float* queries,
                             int32_t nq, int32_t queries_on_device, cudaStream_t pass_stream,
                             const cudaStream_t* cursor_streams, pvs_cursor** out);
// Open a cursor whose device work runs on `stream` (null: the index's stream).
pvs_status cursor_open_on(pvs_index* x, const pvs_snapshot* snap, const float* query,
                          int32_t query_on_device, cudaStream_t stream, pvs_cursor** out);
}  // namespace pvs
