// Host-side launchers of the PVS device kernels (internal to libpvs.so).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace pvs {

// Process-wide count of kernels launched by the library (pvs_launch_count).
void count_launches(int k);

constexpr int kTileRows = 64;         // rows per interval-pass tile
constexpr int kCodeAlign = 64;        // code rows padded to a multiple of 64 bytes
constexpr int kMaxDim = 32767;
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // 2 s device-side wait limit

// Encoded query scalars (Sec. 2.3.1, App. A.1).
struct QueryScalars {
    float s;       // s_q
    float qnorm;   // ||q||_2 rounded up
    float qhat;    // ||s_q z_q||_2 rounded up
    float enorm;   // ||q - s_q z_q||_2 rounded up
    float gamma;   // gamma_m
    int status;    // PVS status of the encoding
};

// Radix-select state for the k-th largest ordered key.
struct SelectState {
    uint64_t prefix;     // decided high bits of the key
    uint64_t k;          // remaining rank among keys that match the prefix
    uint32_t hist[256];
};

// Per-cursor device counters.
struct DevCounters {
    unsigned long long refined;
    unsigned long long exact_fallbacks;
    unsigned int w_len;      // working-set length
    unsigned int cand;       // candidates of the current pull
    unsigned long long cand_total;   // candidates over fused pulls
    // frontier carried between one-launch pulls: every live working-set row
    // with hi >= front_bound (a float key) is among the front_n entries of
    // PullArgs::front, and at least front_k live rows have lo >= front_bound;
    // front_k == 0: no frontier.  front_hint: the multiple of n the next
    // whole-set gather starts with (0: the widest).
    unsigned int front_n;
    unsigned int front_bound;
    unsigned int front_k;
    unsigned int front_hint;
};

// Where one cursor keeps its device status word and counters.
struct CursorRef {
    const int* status;
    const DevCounters* ctr;
};

// ---- fused single-CTA pull (pull_kernel.cu) ----------------------------------
constexpr int kPullFusedMax = 256;   // largest pull served by one fused launch
struct PullArgs {
    int32_t* w_id;
    float* w_lo;
    float* w_hi;
    const unsigned int* w_len;
    float* lo;                // bounds of every row (kept in step with the working set)
    float* hi;
    const float* qraw;
    const float* raw;
    int m_raw;
    int n;                    // ranks to emit, 1 .. kPullFusedMax
    int32_t* cand;            // scratch, >= working-set capacity
    unsigned long long* keys; // scratch, >= working-set capacity
    int64_t* out_ids;         // device
    float* out_scores;        // device
    int* status;
    DevCounters* ctr;
    int32_t* front;           // frontier of working-set indices, kFrontCap entries
    int* status_mirror;       // pinned host word: the status after the pull (null: none)
};
cudaError_t launch_pull_fused(const PullArgs& a, int refine_grid, cudaStream_t st);
// Many cursors at once: the per-cursor arguments travel as kernel
// parameters, up to kPullPack cursors per launch (the parameter space holds
// 32,764 bytes), so no copy of them is staged; every CTA reads only its own
// cursor's entry, one address for all its threads.  The host array is read
// at launch.
constexpr int kPullPack = 224;
struct PullArgsPack {
    PullArgs a[kPullPack];
};
static_assert(sizeof(PullArgsPack) <= 31 * 1024, "kernel parameter space");
// One launch per pull (n <= kPullFusedMax): a cluster of CTAs selects,
// refines and emits (one cluster per cursor in the batch form).
cudaError_t launch_pull_cluster(const PullArgs& a, cudaStream_t st);
cudaError_t launch_pull_cluster_batch(const PullArgs* host_args, int ncursors, cudaStream_t st);
// Ranks computed ahead, handed to the callers' buffers: for every entry,
// count ids and scores from src to dst (device or pinned host memory), in
// stream order, one launch per 64 entries (the entries are read at launch).
struct RankCopy {
    const int64_t* src_ids;
    const float* src_scores;
    int64_t* dst_ids;
    float* dst_scores;
    int count;
};
cudaError_t launch_copy_ranks(const RankCopy* host, int n, cudaStream_t st);
cudaError_t launch_pull_batch(const PullArgs* host_args, int ncursors, int refine_blocks_per_cursor,
                              int m_raw, cudaStream_t st);
// ncursors <= kPullPack entries of p.
cudaError_t launch_refine_batch(const PullArgsPack& p, int ncursors, int blocks_per_cursor,
                                int m_raw, cudaStream_t st);

// ---- batched open support (pull_kernel.cu, batch_support.cu) ----------------
constexpr int kWsSortMax = 8192;     // largest per-query working set of a batched open
constexpr int kFrontCap = 4096;      // frontier entries (the one-launch pull's gather capacity)
struct WsDst {                       // a cursor's working-set arrays
    int32_t* w_id;
    float* w_lo;
    float* w_hi;
    unsigned int* w_len;
};
struct QueryDst {                    // a cursor's query buffers and fresh device state
    int8_t* zq;
    float* qraw;
    QueryScalars* qs;
    DevCounters* ctr;                // zeroed by the copy
    int* status;                     // zeroed by the copy
};
cudaError_t launch_batch_tau(const float* dump_lo, int64_t ld, unsigned int nsample, int nq,
                             unsigned int k, float* tau, cudaStream_t st);
cudaError_t launch_ws_sort(const int32_t* w_id_b, const float* w_lo_b, const float* w_hi_b,
                           int cap, const unsigned int* w_len_b, const WsDst* dst, int nq,
                           cudaStream_t st);
cudaError_t launch_norm_max(const float* vnorm, const float* enorm, int64_t rows,
                            unsigned int* out, cudaStream_t st);
cudaError_t launch_rmax(const QueryScalars* qs, int nq, const unsigned int* maxes, float* rmax,
                        cudaStream_t st);
cudaError_t launch_copy_queries(const int8_t* zq_b, const float* qraw_b, const QueryScalars* qs_b,
                                const QueryDst* dst, int nq, int m_pad, int m_raw,
                                cudaStream_t st);
cudaError_t launch_scatter_ws(const int32_t* w_id, const float* w_lo, const float* w_hi,
                              const unsigned int* w_len, float* lo, float* hi, int grid,
                              cudaStream_t st);

// ---- build / encode (build_kernels.cu) -------------------------------------
// Quantize rows [0, n) of `vecs` (row stride m floats) into codes (stride
// m_pad), params, and a raw copy (stride m_raw, zero padded).
// fixed_scale (device, may be null): one scale for every row (scalar-
// quantization intervals) instead of each row's own.
cudaError_t launch_build(const float* vecs, int64_t n, int m, int m_pad, int m_raw,
                         int8_t* codes, float* scale, float* vnorm, float* enorm, float* raw,
                         int* status, cudaStream_t st, const float* fixed_scale = nullptr);
// *out = max(*out, bits of max |v_i|) over count floats (*out zeroed by the caller).
cudaError_t launch_maxabs(const float* v, int64_t count, unsigned int* out, cudaStream_t st);
// *s = RN(maxabs / 127) (1 for 0; 2^-149 if the quotient underflows).
cudaError_t launch_scale_from_maxabs(const unsigned int* maxabs_bits, float* s, cudaStream_t st);

// ---- exhaustive float32 scanning (scan_kernels.cu) ---------------------------
// keys[row] = rank_key(authoritative score, row) for every visible row < rows
// (0 for a deleted row); ctr->refined counts the scored rows.
cudaError_t launch_scan_scores(const float* qraw, const float* raw, int m_raw, int64_t rows,
                               const uint32_t* tomb, uint64_t* keys, int* status,
                               DevCounters* ctr, cudaStream_t st);
// ids / scores of keys[0 .. n); *mirror = *status afterwards when mirror is set.
cudaError_t launch_scan_emit(const uint64_t* keys, int64_t n, int64_t* ids, float* scores,
                             const int* status, int* mirror, cudaStream_t st);
// Encode one query: codes zq[m_pad], raw copy qraw[m_raw], scalars.
cudaError_t launch_encode_query(const float* q, int m, int m_pad, int m_raw, int8_t* zq,
                                float* qraw, QueryScalars* qs, cudaStream_t st);
// Encode nq queries (row stride m), one warp each.
cudaError_t launch_encode_queries(const float* q, int nq, int m, int m_pad, int m_raw,
                                  int8_t* zq, float* qraw, QueryScalars* qs, cudaStream_t st);

// ---- interval pass (interval_kernels.cu) ------------------------------------
struct IntervalArgs {
    const int8_t* codes;
    const float* scale;
    const float* vnorm;
    const float* enorm;
    const uint32_t* tomb;   // tombstone bitmap of the snapshot, or null
    int64_t rows;           // rows [0, rows) are scanned
    int m_pad;
    const int8_t* zq;
    const QueryScalars* qs;
    float* lo;
    float* hi;
    int* status;
    // optional: the kSlotTop largest live lower bounds of every row slot of
    // the staged pass (slot = CTA x row position in a tile; each row belongs
    // to one slot), kSlotTop per slot, -inf where a slot had fewer live rows
    float* slot_top = nullptr;
    // limit of each wait for a tile or a free stage (device ns; 0: never
    // wait).  Waits for the pass's own copies in flight before it exits keep
    // the full 2 s limit whatever this is, so no copy outlives the kernel.
    unsigned long long wait_ns = kWaitLimitNs;
};
constexpr int kSlotTop = 4;
cudaError_t launch_interval_pass(const IntervalArgs& a, int num_sms, cudaStream_t st);
// Slots whose kSlotTop lower bounds a pass over `rows` rows of m_pad bytes
// writes to slot_top (0: that pass writes none), and the fewest rows any
// of them scans.
int64_t interval_slots(int64_t rows, int m_pad, int num_sms, int64_t* min_rows_per_slot);
// Plain reference-style variant without staging (used for tiny inputs).
cudaError_t launch_interval_simple(const IntervalArgs& a, cudaStream_t st);

// Grouped pass: the intervals of up to kGroupMax queries from one read of the
// codes (each code tile is staged once and scored against every query of
// the group).  Per query g < nq: its codes zq[g] and scalars qs[g], and its
// own outputs lo[g], hi[g], status[g] and slot_top[g] (may be null).  A
// slot of the grouped pass is (CTA, consumer warp, MMA row pair):
// interval_group_slots gives their count and the fewest rows any scans.
constexpr int kGroupMax = 16;
struct IntervalGroupArgs {
    const int8_t* codes;
    const float* scale;
    const float* vnorm;
    const float* enorm;
    const uint32_t* tomb;
    int64_t rows;
    int m_pad;
    int nq;
    const int8_t* zq[kGroupMax];
    const QueryScalars* qs[kGroupMax];
    float* lo[kGroupMax];
    float* hi[kGroupMax];
    int* status[kGroupMax];
    float* slot_top[kGroupMax];
    // largest upper bound of each 16-row block ((rows + 15) / 16 floats per
    // query; -inf where no row is live), or null
    float* bmax[kGroupMax];
    unsigned long long wait_ns = kWaitLimitNs;
};
constexpr int kBmaxRows = 16;
// True when a grouped pass serves nq queries over rows of m_pad bytes.
bool interval_group_supported(int m_pad, int nq);
cudaError_t launch_interval_group(const IntervalGroupArgs& a, int num_sms, cudaStream_t st);

// First working sets of the n <= kGroupMax cursors of a grouped pass, in four
// launches for all of them (grid dimension y = the cursor): per cursor g the
// k[g]-th largest of its slot_n per-slot lower bounds (select_small), then the
// ordered compaction of its rows with key(hi) >= that threshold
// (launch_compact_ordered's count, scan and scatter).
struct WsGroupArgs {
    int n;
    int64_t rows;
    int64_t slot_n;
    const float* slot[kGroupMax];
    uint64_t k[kGroupMax];
    SelectState* sel[kGroupMax];
    const float* lo[kGroupMax];
    const float* hi[kGroupMax];
    int32_t* w_id[kGroupMax];
    float* w_lo[kGroupMax];
    float* w_hi[kGroupMax];
    unsigned int* w_len[kGroupMax];
    unsigned int* scratch[kGroupMax];   // compact_scratch_elems(rows) each
    // the pass's 16-row block maxima of hi (upper bounds of the current hi:
    // refinement and delivery only lower a row's upper bound), or null; with
    // all of them set, only the blocks that reach the threshold are read
    const float* bmax[kGroupMax];
};
cudaError_t launch_ws_group(const WsGroupArgs& a, cudaStream_t st);
int64_t interval_group_slots(int64_t rows, int m_pad, int nq, int num_sms,
                             int64_t* min_rows_per_slot);

// ---- selection / compaction / sort (select_kernels.cu) ----------------------
// k-th largest key (1-based) among live entries of a float array: key of
// vals[i] with vals[i] != -inf, i < *len (len in device memory).  Result in
// sel->prefix (as a 32-bit ordered key).  k must be <= live count.
cudaError_t launch_select_f32(const float* vals, const unsigned int* len, uint64_t k,
                              SelectState* sel, int grid, cudaStream_t st);
// Same over `rows` entries with a host-known length.
// As launch_select_f32_n in one single-CTA launch, for short arrays (tens of
// thousands of values).
cudaError_t launch_select_small(const float* vals, int64_t len, uint64_t k, SelectState* sel,
                                cudaStream_t st);
cudaError_t launch_select_f32_n(const float* vals, int64_t rows, uint64_t k, SelectState* sel,
                                int grid, cudaStream_t st);
// Ordered compaction: for i < rows with lo[i] != -inf and key(hi[i]) >=
// sel->prefix, append (i, lo, hi) to (w_id, w_lo, w_hi) in index order;
// writes the count to *w_len.  `scratch` holds >= compact_scratch(rows) uints.
size_t compact_scratch_elems(int64_t rows);
cudaError_t launch_compact_ordered(const float* lo, const float* hi, int64_t rows,
                                   const SelectState* sel, int32_t* w_id, float* w_lo,
                                   float* w_hi, unsigned int* w_len, unsigned int* scratch,
                                   cudaStream_t st);
// Candidates of a pull: i < *w_len, live, key(w_hi[i]) >= sel->prefix ->
// cand[] (unordered), count in *cand_len (zeroed by the launcher).
cudaError_t launch_candidates(const float* w_lo, const float* w_hi, const unsigned int* w_len,
                              const SelectState* sel, int32_t* cand, unsigned int* cand_len,
                              int grid, cudaStream_t st);
// keys[i] = rank_key(w_lo[cand[i]], cand[i]) for i < *cand_len.
cudaError_t launch_make_keys(const int32_t* cand, const unsigned int* cand_len,
                             const float* w_lo, uint64_t* keys, int grid, cudaStream_t st);
// Sort `count` 64-bit keys descending, in place (count <= kBitonicMax).
constexpr int kBitonicMax = 8192;
cudaError_t launch_bitonic_desc(uint64_t* keys, int count, cudaStream_t st);
// LSD radix sort of `count` 64-bit keys descending; result in keys.
size_t radix_sort_scratch_bytes(int64_t count);
cudaError_t launch_radix_sort_desc(uint64_t* keys, uint64_t* tmp, int64_t count, void* scratch,
                                   cudaStream_t st);
// Emit the first n sorted keys: ids/scores out (device), mark emitted.
cudaError_t launch_emit(const uint64_t* keys, int n, const int32_t* w_id, float* w_lo,
                        float* w_hi, float* lo, float* hi, int64_t* out_ids, float* out_scores,
                        cudaStream_t st);

// ---- batched interval pass on the tensor cores (batch_gemm.cu) --------------
struct BatchArgs {
    int64_t rows;                 // corpus rows [0, rows) are scanned
    int m_pad;                    // K (multiple of 64)
    int nq, nq_pad;               // queries; nq_pad multiple of 32, <= 256
    const float* scale;
    const float* vnorm;
    const float* enorm;
    const uint32_t* tomb;         // tombstones of the snapshot, or null
    const QueryScalars* qs;       // [nq]
    int mode;                     // 0: dump, 1: filter
    int tile_stride;              // process 128-row tiles 0, s, 2s, ...
    float* dump_lo;               // dump: [nq][dump_ld], row (i*128 + r) of tile i*s
    float* dump_hi;
    int64_t dump_ld;
    const float* tau;             // filter: [nq] thresholds
    const float* rmax;            // filter: [nq] upper bound of the interval half-width
    int32_t* w_id;                // filter: [nq][w_cap] working sets (unordered)
    float* w_lo;
    float* w_hi;
    int w_cap;
    unsigned int* w_len;          // [nq] (may exceed w_cap: overflow)
    unsigned int* h_eff;          // [nq] rows with lo >= tau
    int* status;
};
cudaError_t launch_batch_intervals(const BatchArgs& a, const uint16_t* codes_bf16,
                                   const uint16_t* qcodes_bf16, int num_sms, cudaStream_t st);
// status_out[i] = *refs[i].status; ctr_out[i] = *refs[i].ctr (ctr_out may be null).
cudaError_t launch_gather_state(const CursorRef* refs, int n, int* status_out,
                                DevCounters* ctr_out, cudaStream_t st);
cudaError_t launch_codes_to_bf16(const int8_t* src, uint16_t* dst, int64_t count,
                                 cudaStream_t st);

// ---- refinement (refine_kernels.cu) -----------------------------------------
// Authoritative score of every unresolved candidate (w_lo < w_hi): exact
// RN_f32(sum_j q_j v_j), containment check, then w_lo = w_hi = lo = hi = s.
cudaError_t launch_refine(const int32_t* cand, const unsigned int* cand_len,
                          const int32_t* w_id, float* w_lo, float* w_hi, float* lo, float* hi,
                          const float* qraw, const float* raw, int m_raw, int* status,
                          DevCounters* ctr, int grid, cudaStream_t st);
// Authoritative scores of explicit ids (tests / diagnostics).
cudaError_t launch_score_ids(const int64_t* ids, int n, const float* qraw, const float* raw,
                             int m_raw, float* out, DevCounters* ctr, cudaStream_t st);

}  // namespace pvs
