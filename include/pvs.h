/*
 * pvs.h -- C ABI of the GB300 PVS / EAHR library (libpvs.so).
 *
 * Method: "Exact Adaptive Hybrid Retrieval Without Fixed Top-L Cutoffs",
 * arXiv 2608.07152.
 *   - PVS (Per-Vector Scalar Quantization) resumable exact dense ranking,
 *     Sec. 2.3.1 and Appendix A.1;
 *   - the ranked-list contract (stable exact prefix, Open / Exhausted /
 *     Failed), Sec. 2.1;
 *   - EAHR adaptive weighted-RRF fusion with ordered certification,
 *     Sec. 2.1 and 2.2.
 *
 * Conventions for every entry point:
 *   - Every call returns a pvs_status.  Negative values are errors; on an
 *     error no output is produced and, for a cursor, the cursor becomes
 *     Failed for good (Sec. 2.1: a Failed list invalidates the request).
 *   - Item ids are row numbers in insertion order (0, 1, 2, ...); the tie
 *     order between equal scores is ascending id.
 *   - Vectors are row-major float32, `dim` floats per row, no padding.
 *   - "on_device" flags say whether a pointer is CUDA device memory (or
 *     managed memory) of the current device (1) or host memory (0).
 *   - The library owns index, snapshot and cursor objects; the caller owns
 *     every buffer it passes in.  Threads: distinct cursors of one index may
 *     be opened, pulled and closed from different host threads at once; a
 *     single cursor must not be used by two threads at once, and index
 *     mutations (pvs_append, pvs_tombstone, pvs_index_free) must not overlap
 *     any other call on that index.
 *   - Index work runs on the CUDA stream given to pvs_build (or a
 *     library-created stream when NULL); a cursor's work runs on that stream
 *     too unless pvs_cursor_set_stream moves it.
 */
#ifndef PVS_H_
#define PVS_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum pvs_status {
    PVS_OK = 0,
    PVS_EXHAUSTED = 1,        /* the ranked list is complete (Sec. 2.1)        */
    PVS_ERR_INVALID = -1,     /* bad argument or call sequence                 */
    PVS_ERR_NONFINITE = -2,   /* non-finite vector entry (App. A.1)            */
    PVS_ERR_OVERFLOW = -3,    /* a bound or score overflows float32, or the
                                 Int8 accumulator could overflow (App. A.1)    */
    PVS_ERR_INTERVAL = -4,    /* an authoritative score fell outside its
                                 interval (App. A.1): the request fails        */
    PVS_ERR_CUDA = -5,        /* a CUDA runtime call failed                    */
    PVS_ERR_OOM = -6,         /* device or host allocation failed              */
    PVS_ERR_TIMEOUT = -7,     /* a device-side wait ran out of time            */
    PVS_ERR_FAILED = -8       /* the cursor failed earlier                     */
} pvs_status;

/* Corpus quantization of an index (pvs_build_ex). */
typedef enum pvs_quantization {
    PVS_QUANT_PER_VECTOR = 0,   /* PVS: each vector its own scale (Sec. 2.3.1)             */
    PVS_QUANT_GLOBAL = 1        /* scalar-quantization intervals: one scale for the corpus,
                                   the rank-generator ablation of Sec. 3.5 / 4.4           */
} pvs_quantization;

/* Rank generator of a cursor (pvs_cursor_set_generator). */
typedef enum pvs_generator {
    PVS_GEN_INTERVALS = 0,      /* score intervals, selective exact evaluation (default)   */
    PVS_GEN_FULL_SCAN = 1       /* exhaustive float32 scanning: every visible row scored
                                   exactly, one full sort (ablation, Sec. 3.5 / 4.4)       */
} pvs_generator;

typedef struct pvs_index pvs_index;
typedef struct pvs_snapshot pvs_snapshot;
typedef struct pvs_cursor pvs_cursor;

/* Counters of one cursor (the logical counters of Sec. 3.5 plus device
 * traffic). */
typedef struct pvs_stats {
    int64_t visible;          /* n_i: items in the cursor's ranked list        */
    int64_t emitted;          /* d_i: ranks delivered so far                   */
    int64_t refined;          /* authoritative float32 score evaluations       */
    int64_t exact_fallbacks;  /* evaluations that needed the exact accumulator */
    int64_t interval_passes;  /* full passes over the Int8 codes               */
    int64_t horizon_builds;   /* candidate-set (re)builds from the bounds      */
    int64_t pulls;            /* device pulls (a call served from ranks computed
                                 ahead of it needs none)                       */
    int64_t candidates;       /* candidate entries certified over all pulls    */
    int64_t code_bytes;       /* bytes of codes + per-vector params scanned    */
    int32_t state;            /* PVS_OK (Open), PVS_EXHAUSTED, or the failure  */
    int32_t reserved;
    double interval_ms;       /* device time of the interval passes, measured
                                 with CUDA events on the cursor's stream       */
    int64_t batch_passes;     /* batched tensor-core passes that served it     */
    double batch_ms;          /* device time of that batched pass (shared by
                                 the cursors of its group), CUDA events       */
} pvs_stats;

/* ---------------------------------------------------------------------------
 * Index (Sec. 2.3.1: PVS stores per vector an Int8 code z_v in [-127,127]^m,
 * a scale s_v > 0, and here the upward-rounded norms ||v||_2 and
 * ||v - s_v z_v||_2 that the residual bound E and guard G need (App. A.1);
 * the raw float32 vectors are kept for authoritative scoring).
 * ------------------------------------------------------------------------ */

/* Build an index over n vectors of dimension dim (1 <= dim <= 32767,
 * 0 <= n < 2^31).  `vecs` is n*dim floats, host or device per
 * vecs_on_device.  `cuda_stream` is a cudaStream_t (NULL: the library
 * creates one).  Errors: PVS_ERR_INVALID (null out, bad sizes),
 * PVS_ERR_NONFINITE (an entry is NaN or +-inf; App. A.1), PVS_ERR_OVERFLOW
 * (a norm bound overflows float32), PVS_ERR_OOM, PVS_ERR_CUDA.  On success
 * *out owns device copies of everything; free it with pvs_index_free. */
pvs_status pvs_build(const float* vecs, int64_t n, int32_t dim, int32_t vecs_on_device,
                     void* cuda_stream, pvs_index** out);

/* pvs_build with a choice of corpus quantization.  PVS_QUANT_GLOBAL gives
 * the scalar-quantization-interval index of the rank-generator ablation
 * (Sec. 3.5, 4.4; the paper gives no construction, reading of this
 * library): one scale s = RN(max_{v,j} |v_j| / 127) over the n vectors, the
 * codes, norm bounds and intervals of Sec. 2.3.1 / App. A.1 with s in place
 * of every s_v; queries keep their own scale.  pvs_append on such an index
 * uses the same s and fails with PVS_ERR_INVALID for a vector whose codes
 * would leave [-127, 127].  Errors as pvs_build, and PVS_ERR_INVALID for an
 * unknown quantization. */
pvs_status pvs_build_ex(const float* vecs, int64_t n, int32_t dim, int32_t vecs_on_device,
                        void* cuda_stream, int32_t quantization, pvs_index** out);

/* Append n vectors; they get ids size .. size+n-1.  Existing snapshots and
 * open cursors keep their visible set (Sec. 2.4: fixed snapshots).  Errors
 * as pvs_build; on error the index is unchanged. */
pvs_status pvs_append(pvs_index* index, const float* vecs, int64_t n, int32_t vecs_on_device);

/* Tombstone (delete) n ids given in host memory.  Deleting a deleted id is a
 * no-op.  Affects snapshots created afterwards only (Sec. 2.4: deletion
 * state defines the visible items of a snapshot).  Errors: PVS_ERR_INVALID
 * if an id is out of range (nothing is deleted then). */
pvs_status pvs_tombstone(pvs_index* index, const int64_t* ids, int64_t n);

int64_t pvs_index_size(const pvs_index* index);   /* rows ever inserted       */
int64_t pvs_index_live(const pvs_index* index);   /* rows not tombstoned      */
int32_t pvs_index_dim(const pvs_index* index);
/* Copy rows [first, first+count) of the index into caller buffers, any of
 * which may be NULL: codes as int8 [count x dim], scales, norm bounds of v and
 * of the residual v - s_v z_v (float32 [count]).  Host pointers. */
pvs_status pvs_index_export(const pvs_index* index, int64_t first, int64_t count,
                            int8_t* codes, float* scale, float* vnorm, float* enorm);
void pvs_index_free(pvs_index* index);

/* Load an index from data saved earlier (pvs_index_export gives codes,
 * scales and norm bounds; the caller keeps the raw vectors): n rows of
 * dimension dim, all HOST buffers -- vecs float32 [n x dim], codes int8
 * [n x dim], scale / vnorm / enorm float32 [n].  Nothing is re-quantized:
 * the library checks only what it relies on to stay in bounds (codes in
 * [-127, 127], finite vectors, finite positive scales, finite nonnegative
 * norm bounds) and otherwise trusts the parameters.  Parameters that do not
 * bound a row's score are caught by the failure rule of App. A.1 when that
 * row is scored exactly: the pull fails with PVS_ERR_INTERVAL and the cursor
 * is Failed.  `cuda_stream` as in pvs_build.  Errors: PVS_ERR_INVALID,
 * PVS_ERR_NONFINITE (a non-finite vector entry), PVS_ERR_OOM, PVS_ERR_CUDA. */
pvs_status pvs_index_import(const float* vecs, const int8_t* codes, const float* scale,
                            const float* vnorm, const float* enorm, int64_t n, int32_t dim,
                            void* cuda_stream, pvs_index** out);

/* Device-side time limit, in nanoseconds, of each wait of this index's
 * interval passes for a tile of codes or a free pipeline stage (default and
 * maximum 2e9, i.e. 2 s).  A wait that runs out sets PVS_ERR_TIMEOUT: the
 * pull fails and the cursor is Failed (Sec. 2.1); the GPU context stays
 * usable and other cursors are unaffected.  0 makes every such wait give up
 * at once unless its tile has already arrived, which lets tests reach the
 * timeout rule without a fault.  While the limit is below 2 s, each pass's
 * status is read on the host before the pull goes on.  The pass's waits for
 * its own copies in flight always keep the 2 s limit.  Must not overlap
 * other calls on the index.  Errors: PVS_ERR_INVALID (null index, ns < 0). */
pvs_status pvs_index_set_wait_limit(pvs_index* index, int64_t ns);

/* Freeze the currently visible set (rows inserted so far minus tombstones).
 * A snapshot may be freed while cursors opened on it are still open. */
pvs_status pvs_snapshot_create(pvs_index* index, pvs_snapshot** out);
int64_t pvs_snapshot_visible(const pvs_snapshot* snap);
void pvs_snapshot_free(pvs_snapshot* snap);

/* ---------------------------------------------------------------------------
 * Cursor: one query's resumable exact dense ranked list (Sec. 2.1, 2.3.1).
 * ------------------------------------------------------------------------ */

/* Open a cursor for one query (dim floats, host or device).  `snap` may be
 * NULL for the index's current visible set.  The query is encoded like a
 * corpus vector (Sec. 2.3.1).  The index must outlive the cursor.  Errors:
 * PVS_ERR_INVALID, PVS_ERR_NONFINITE, PVS_ERR_OVERFLOW, PVS_ERR_OOM,
 * PVS_ERR_CUDA. */
pvs_status pvs_cursor_open(pvs_index* index, const pvs_snapshot* snap, const float* query,
                           int32_t query_on_device, pvs_cursor** out);

/* Open nq cursors (queries: nq*dim floats) whose intervals come from one
 * tensor-core pass per group of up to 256 queries (the Int8 dot products of
 * all queries as one exact bf16 GEMM, Sec. 2.3.1 intervals in its
 * epilogue).  Each cursor keeps only the rows that can hold its first
 * ranks: `horizon` (>= 1) is the number of ranks it is prepared for; it can
 * usually deliver about three times that many before it needs a
 * single-query interval pass, and later ranks still come out exactly, at the
 * cost of that pass.  The work runs on `cuda_stream` (a cudaStream_t; NULL:
 * the index's stream), and so do the cursors afterwards: batched opens on
 * different streams from different threads overlap on the device (their
 * full passes over the codes still run one at a time).  The call returns
 * once the cursors are ready.  out[0..nq-1] receive the cursors.  Errors as
 * pvs_cursor_open; on error no cursor is returned. */
pvs_status pvs_cursor_open_batch(pvs_index* index, const pvs_snapshot* snap,
                                 const float* queries, int32_t nq, int32_t queries_on_device,
                                 int32_t horizon, void* cuda_stream, pvs_cursor** out);

/* Largest group of pvs_cursor_open_group. */
#define PVS_GROUP_MAX 16

/* Open nq (1 <= nq <= PVS_GROUP_MAX) cursors over one snapshot (`snap`, NULL:
 * the index's current visible set) whose score intervals come from ONE
 * streaming pass over the Int8 codes (Sec. 2.3.1, App. A.1): each tile of
 * codes is read once and scored against all nq queries, instead of once per
 * query.  Each cursor gets the same bounds, bit for bit, as a cursor of
 * pvs_cursor_open, and afterwards behaves like one.  queries: nq x dim
 * floats, host or device per queries_on_device.  The pass runs on
 * `pass_stream` (a cudaStream_t; NULL: the index's stream) after the
 * queries' encoding; cursor i's later work runs on cursor_streams[i] (an
 * array of nq cudaStream_t, or NULL; a NULL array or entry means
 * pass_stream), ordered after the pass, so the pulls of the group's queries
 * can run on their own streams while the next group's pass streams the
 * codes.  The call returns once the queries are encoded and the pass is
 * queued.  Row widths the grouped pass does not serve (dim rounded up to 64
 * not in {128, 256, 384, 512, 768, 1024}, or above 768 with nq > 8) and
 * nq == 1 give plain cursors
 * with a pass of their own at the first pull.  out[0..nq-1] receive the
 * cursors; close each with pvs_cursor_close.  Errors as pvs_cursor_open; on
 * error no cursor is returned. */
pvs_status pvs_cursor_open_group(pvs_index* index, const pvs_snapshot* snap,
                                 const float* queries, int32_t nq, int32_t queries_on_device,
                                 void* pass_stream, void* const* cursor_streams,
                                 pvs_cursor** out);

/* The next n ranks of each of nc cursors in one set of launches (all
 * cursors of one index and one stream).  Row i of ids / scores (nc x n,
 * int64 / float32, device or host per outputs_on_device) receives cursor i's
 * ranks and n_out[i] (host) their count.  Semantics per cursor as pvs_next
 * (host outputs: blocking, statuses checked) or pvs_next_device (device
 * outputs: queued).  Returns PVS_OK or the first error. */
pvs_status pvs_next_batch(pvs_cursor** cursors, int32_t nc, int32_t n, int32_t outputs_on_device,
                          int64_t* ids, float* scores, int32_t* n_out);

/* Read-ahead: a pull of n <= 256 ranks computes up to `pages` x n of them
 * (at most 256; default 4) and keeps the ones not asked for in the cursor,
 * so the next calls are served without device work (host outputs) or by a
 * copy (device outputs).  Exact either way (Sec. 2.1: the list is a stable
 * prefix, so a rank computed early is the rank delivered later).  pages = 1
 * computes exactly what is asked.  Errors: PVS_ERR_INVALID (pages < 1). */
pvs_status pvs_cursor_set_readahead(pvs_cursor* cursor, int32_t pages);

/* Deliver the next n exact ranks (Sec. 2.1: a stable exact prefix that is
 * only ever extended).  ids (int64) and scores (the authoritative float32
 * scores: the correctly rounded value of the exact inner product) are HOST
 * buffers of n entries; *n_out receives the count written.  Returns PVS_OK,
 * or PVS_EXHAUSTED once the last rank has been delivered (then
 * *n_out <= n; later calls deliver 0).  Blocks until the ranks are on the
 * host.  Errors: PVS_ERR_INVALID (n < 0 or null pointers), PVS_ERR_INTERVAL
 * (App. A.1 failure rule), PVS_ERR_OVERFLOW, PVS_ERR_TIMEOUT, PVS_ERR_CUDA,
 * PVS_ERR_FAILED (the cursor failed before). */
pvs_status pvs_next(pvs_cursor* cursor, int32_t n, int64_t* ids, float* scores, int32_t* n_out);

/* As pvs_next, but ids and scores are DEVICE buffers and the call only
 * enqueues the work on the cursor's stream; *n_out is exact on return.
 * Device-side failures surface at the next blocking call (pvs_cursor_sync,
 * pvs_next, pvs_cursor_stats); every rank delivered since the last
 * successful blocking call is then void. */
pvs_status pvs_next_device(pvs_cursor* cursor, int32_t n, int64_t* ids, float* scores,
                           int32_t* n_out);

/* Run the cursor's later device work on `cuda_stream` (a cudaStream_t; NULL:
 * back to the index's stream), after waiting for its queued work.  Cursors on
 * different streams overlap on the device: one query's pulls can run while
 * another query's interval pass streams the codes.  Ordering against work
 * the caller queues elsewhere is the caller's. */
pvs_status pvs_cursor_set_stream(pvs_cursor* cursor, void* cuda_stream);

/* Choose the cursor's rank generator (pvs_generator) before its first pull:
 * PVS_GEN_INTERVALS (default) or PVS_GEN_FULL_SCAN (every visible row scored
 * exactly at the first pull, then one full sort; pulls read it in order).
 * Both produce the same ranking.  Cursors of pvs_cursor_open_batch keep
 * PVS_GEN_INTERVALS.  Errors: PVS_ERR_INVALID (unknown generator, a cursor
 * already pulled, a batched cursor). */
pvs_status pvs_cursor_set_generator(pvs_cursor* cursor, int32_t generator);

/* Wait for the cursor's queued work; return its state (PVS_OK while Open,
 * PVS_EXHAUSTED, or the failure). */
pvs_status pvs_cursor_sync(pvs_cursor* cursor);
pvs_status pvs_cursor_stats(pvs_cursor* cursor, pvs_stats* out);
void pvs_cursor_close(pvs_cursor* cursor);

/* Batch forms of pvs_cursor_sync, pvs_cursor_stats and pvs_cursor_close for
 * the nc cursors of a batched open (a host array of nc non-null cursors; no
 * cursor twice).  They gather the device status words (and counters) of all
 * cursors that share a stream with one launch, one copy and one wait, instead
 * of one round trip per cursor.  pvs_cursor_sync_batch writes each cursor's
 * state to states[i] (host, nc entries: PVS_OK, PVS_EXHAUSTED or the
 * failure; a device failure makes that cursor Failed as pvs_cursor_sync
 * does) and returns PVS_OK unless the call itself failed (PVS_ERR_INVALID
 * for a null array or cursor, PVS_ERR_CUDA, PVS_ERR_OOM).
 * pvs_cursor_stats_batch writes out[i] (host, nc entries) as
 * pvs_cursor_stats would.  pvs_cursor_close_batch waits for each distinct
 * stream once, then closes every cursor; null entries are skipped. */
pvs_status pvs_cursor_sync_batch(pvs_cursor** cursors, int32_t nc, int32_t* states);
pvs_status pvs_cursor_stats_batch(pvs_cursor** cursors, int32_t nc, pvs_stats* out);
void pvs_cursor_close_batch(pvs_cursor** cursors, int32_t nc);

/* Diagnostics.  Copy to host the score interval [lo, hi] that the cursor
 * holds for ids first .. first+count-1 of its snapshot: the App. A.1 interval
 * before an item is scored, lo == hi == its authoritative score after, and
 * -inf once the item is delivered or computed ahead of the caller (read-ahead,
 * pvs_cursor_set_readahead) or if it is deleted.  Runs the interval
 * pass first if no pull has run it yet. */
pvs_status pvs_cursor_bounds(pvs_cursor* cursor, int64_t first, int64_t count, float* lo,
                             float* hi);

/* Authoritative float32 scores (correctly rounded exact inner products) of
 * n ids (host array, each < the cursor's snapshot size) against the cursor's
 * query, written to the host array `scores`.  Does not change the cursor. */
pvs_status pvs_cursor_score_ids(pvs_cursor* cursor, const int64_t* ids, int32_t n,
                                float* scores);

const char* pvs_status_string(int32_t status);

/* Diagnostics.  Score intervals of every row of `snap` (NULL: the current
 * visible set) for 1 <= nq <= 256 queries, computed by the tensor-core
 * batched pass; host outputs lo / hi of nq x rows floats (row-major by
 * query; -inf for deleted rows). */
pvs_status pvs_batch_bounds(pvs_index* index, const pvs_snapshot* snap, const float* queries,
                            int32_t nq, int32_t queries_on_device, float* lo, float* hi);

/* Number of CUDA kernels this library has launched in this process. */
int64_t pvs_launch_count(void);

/* ---------------------------------------------------------------------------
 * Allocation-free exact ranking.  The paper has no counterpart to this entry
 * point.  It exists for callers that cannot allocate device memory where
 * they need a ranking:
 *   - services whose device memory is owned by their own pool or budget
 *     (for instance a server that reserves almost all HBM for its indexes at
 *     start-up): an allocation outside that pool either fails or breaks the
 *     pool's accounting;
 *   - latency-critical callers: cudaMalloc can take milliseconds, and
 *     cudaFree waits for the whole device to go idle.
 * ------------------------------------------------------------------------ */

/* Largest vector count pvs_rank_exact_noalloc accepts. */
#define PVS_NOALLOC_MAX_VECTORS 8192

/* Rank n <= PVS_NOALLOC_MAX_VECTORS row-major float32 vectors `vecs`
 * (n x dim, DEVICE memory) against one query (dim floats, DEVICE memory) by
 * authoritative score -- the correctly rounded exact inner product, the same
 * score and order (score descending, ties by ascending row number) as
 * pvs_next -- and write the first `top` <= n row numbers and scores to the
 * DEVICE buffers out_ids (int64) and out_scores (float32).  Work is queued
 * on `cuda_stream` (a cudaStream_t; NULL for the legacy default stream); the
 * call then copies the device status word into host memory and waits for
 * the stream (cudaStreamSynchronize) before it returns, so the outputs are
 * complete on return.  The library sees raw pointers only: the caller
 * guarantees that query holds dim floats and that out_ids / out_scores hold
 * at least `top` entries.
 *
 * Allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 * Its scratch is one static device array of 8192 64-bit keys plus a status
 * word (64 KiB + 256 B) that every GPU loading the library holds until the
 * process exits.  All calls share that array; it keeps the last call's keys,
 * the status word is cleared by every call, and calls whose device work
 * overlaps (e.g. on two streams at once) race on it.  The first call on a
 * device looks up the array's device address (cudaGetSymbolAddress) with that
 * device current; make that first call before any stream capture begins.
 *
 * Errors: PVS_ERR_INVALID when n > PVS_NOALLOC_MAX_VECTORS, n < 0, top > n,
 * dim outside [1, 32767], or a pointer is not device memory;
 * PVS_ERR_NONFINITE for a NaN or infinite entry of the query or of a vector
 * (with n > 0); PVS_ERR_OVERFLOW when a score overflows float32;
 * PVS_ERR_CUDA when a CUDA call fails. */
pvs_status pvs_rank_exact_noalloc(const float* query, const float* vecs, int32_t n, int32_t dim,
                                  int32_t top, int64_t* out_ids, float* out_scores,
                                  void* cuda_stream);

/* ---------------------------------------------------------------------------
 * EAHR (Sec. 2.1, 2.2): ordered Top-K of complete-list weighted RRF over the
 * dense ranked list of a cursor and a sparse ranked list from the caller.
 * ------------------------------------------------------------------------ */

enum {
    EAHR_RANK_SCALED = 0,   /* g(r) = 1 / (r / w + k - 1)  (Sec. 2.1)         */
    EAHR_NUMERATOR = 1      /* g(r) = w / (k + r)                              */
};
enum {
    EAHR_POLICY_GEOMETRIC = 0,   /* pull the channel with the larger next
                                    contribution; pull sizes grow x2 (result
                                    unchanged: Sec. 2.4)                        */
    EAHR_POLICY_EQUAL_DEPTH = 1, /* both lists advance by `step` ranks, and
                                    certification runs after every step
                                    (the controlled-stream protocol, Sec. 3.4) */
    EAHR_POLICY_FROZEN = 2,      /* the paper's frozen scheduler (Sec. 3.5):
                                    each step reads `step` ranks from the list
                                    whose next unread rank contributes more; a
                                    list skipped 16 steps in a row is advanced;
                                    certification after every step through the
                                    first 4K ranks read, then whenever access
                                    has grown by clamp(access / 8, 64, 1024)
                                    since the last check, and at once when a
                                    list is exhausted                          */
    EAHR_POLICY_ADAPTIVE = 3     /* eahr_topk and eahr_topk_pbm (where the
                                    sparse ranks of the finish come from the
                                    query's complete PBM ranking, computed
                                    on the device): GEOMETRIC reading, and
                                    once the ranks read reach 2^12 (again
                                    each time they double) an exact finish:
                                    with LB the K-th largest L(x) of the
                                    items read, and B < LB, only the items
                                    with U(x) >= LB can be in T*_K; their
                                    missing ranks come from the device: a
                                    sparse rank from the host list, a dense
                                    rank as an interval from counting the
                                    rows whose bounds lie above or around
                                    the item's authoritative score.  When
                                    those intervals do not certify the order
                                    (Sec. 2.2 over the candidates), the rows
                                    around the scores of the candidates
                                    whose intervals overlap are scored and
                                    their ranks made exact (a few rounds,
                                    then every candidate's); the first such
                                    count gives the index 4-bit codes of
                                    each row's quantization residual
                                    (m_pad / 2 + 16 bytes per row, kept and
                                    extended over appended rows), whose
                                    tighter intervals place most of those
                                    rows without their fp32 rows.  An F known only as an
                                    interval is reported as NaN (its
                                    position is certified).  Failing that
                                    (too many candidates,
                                    a cursor without bounds of every row),
                                    once the ranks read reach (n_dense +
                                    n_sparse) / 16 clamped to [2^16, 2^18]
                                    (eahr_topk only):
                                    complete-list fusion on the device (every
                                    visible row's authoritative score, both
                                    lists' ranks, the fused order).  Both
                                    finishes rest on Sec. 2.2 (when early
                                    determination is impossible, fusing the
                                    complete lists gives the same result).
                                    Complete-list fusion, and an exact finish
                                    that needs a sparse rank, read the whole
                                    sparse list: an invalid id anywhere in it
                                    then fails the call.
                                    Other entry points treat it as GEOMETRIC  */
};

typedef struct eahr_params {
    int32_t K;          /* result size, >= 1                                   */
    int32_t k;          /* RRF rank constant, >= 1                             */
    int32_t form;       /* EAHR_RANK_SCALED or EAHR_NUMERATOR                  */
    int32_t policy;     /* EAHR_POLICY_*                                       */
    int32_t step;       /* first pull size (GEOMETRIC, ADAPTIVE) or step
                           (EQUAL_DEPTH, FROZEN); 0 selects 16, or 2^11 for
                           ADAPTIVE (its exact finish is first tried once
                           2^12 ranks are read)                              */
    int32_t w_num[2];   /* channel weights w_i = w_num[i] / w_den[i];          */
    int32_t w_den[2];   /* [0] dense, [1] sparse; 0 <= w_num < 2^16,
                           1 <= w_den < 2^16                                   */
} eahr_params;

typedef struct eahr_stats {
    int64_t depth[2];       /* d_i: ranks read from each list                  */
    int64_t length[2];      /* n_i: complete-list length of each list          */
    int32_t exhausted[2];   /* list i reached Exhausted                        */
    int32_t pulls[2];       /* producer calls per list                         */
    int32_t checks;         /* certification rounds                            */
    int32_t complete;       /* how EAHR_POLICY_ADAPTIVE finished: 0 certified
                               from the ranks read (Sec. 2.2), 1 complete-list
                               fusion on the device, 2 the remaining
                               candidates ordered by the rank intervals their
                               rows' bounds give, 3 by exact ranks (rows
                               scored)                                        */
} eahr_stats;

/* EAHR over a freshly opened dense cursor (no ranks delivered yet) and a
 * sparse ranked list given as host ids in rank order (the support U_s may be
 * a subset of the visible items).  Sparse ids are checked as the driver reads
 * them: an id outside the cursor's snapshot, or repeated within the list,
 * fails the call with PVS_ERR_INVALID when it is reached (entries the driver
 * never reads are not inspected).  Writes the q_K <= K ids of T*_K in order
 * to out_ids and their count to *n_out (Sec. 2.1: zero-score items are never
 * appended).  out_F (may be NULL) receives each item's fused score F as the
 * correctly rounded binary64 value of the exact rational where the prefixes
 * read determine it, and NaN where the item is still unread in an Open list
 * (its position is certified all the same, Sec. 2.2).  `st` may be NULL.
 * Errors: PVS_ERR_INVALID (bad parameters, cursor not fresh, bad sparse
 * list), any error of pvs_next (the request is then void). */
pvs_status eahr_topk(pvs_cursor* dense, const int64_t* sparse_ids, int64_t n_sparse,
                     const eahr_params* params, int64_t* out_ids, double* out_F,
                     int32_t* n_out, eahr_stats* st);

/* The same fusion over two ranked lists held in host memory (ids in rank
 * order, 0 <= id < 2^31; an id repeated within a list fails the call when it
 * is read).  For callers with their own producers and for the
 * controlled-stream protocol of Sec. 3.4. */
pvs_status eahr_topk_lists(const int64_t* list0, int64_t n0, const int64_t* list1, int64_t n1,
                           const eahr_params* params, int64_t* out_ids, double* out_F,
                           int32_t* n_out, eahr_stats* st);

#ifdef __cplusplus
}
#endif

#endif /* PVS_H_ */
