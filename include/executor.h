/*
 * executor.h -- native request executor in libpvs.so.
 *
 * Method: arXiv 2608.07152 Sec. 2.1 (a ranked list is read as a stable
 * prefix that is only extended, page after page, until the consumer stops)
 * and Sec. 2.3 (PVS: resumable exact dense ranking by intervals and exact
 * refinement).  The executor serves many such requests from host memory,
 * the way a search service does: for each request it opens a PVS cursor on
 * the request's query, reads `ranks` ranks in pages of `page` ranks through
 * pvs_next (every page is on the host before the next is requested, as when
 * a client pages through results) and closes the cursor.
 *
 * A fixed pool of native worker threads, each with its own CUDA stream on
 * the index's device, keeps up to `workers` requests in flight, so the
 * interval pass of one request overlaps the pages of the others on the
 * device.  No host interpreter is involved between pages.  With a group
 * size G >= 2 (pvs_executor_set_group) a worker serves G requests at a time:
 * their cursors come from one pvs_cursor_open_group (one pass over the Int8
 * codes for all G queries) and each page of the G cursors is one batched
 * pull; every request still receives its own pages.
 *
 * Conventions as pvs.h: the caller owns every buffer; the index must
 * outlive the executor and must not be changed (append, delete) while a run
 * is in progress.
 */
#ifndef PVS_EXECUTOR_H_
#define PVS_EXECUTOR_H_

#include <stdint.h>

#include "pvs.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pvs_executor pvs_executor;

typedef struct pvs_executor_stats {
    int64_t requests;    /* requests served (all runs)                       */
    int64_t failed;      /* of those, requests that ended in an error         */
    int64_t pages;       /* pvs_next calls                                    */
    int64_t ranks;       /* ranks delivered                                   */
    int32_t workers;     /* worker threads (and streams)                      */
    int32_t group;       /* requests per grouped open (1: none)               */
    int64_t interval_passes; /* passes over the Int8 codes (a grouped pass
                                counts once)                                 */
    double interval_ms;  /* their device time, CUDA events, summed           */
    int64_t refined;     /* authoritative float32 evaluations                 */
} pvs_executor_stats;

/*
 * Start `workers` (1 .. 64) worker threads for `index`, each with a
 * non-blocking CUDA stream on the index's device.  Errors: PVS_ERR_INVALID,
 * PVS_ERR_OOM, PVS_ERR_CUDA.
 */
pvs_status pvs_executor_create(pvs_index* index, int32_t workers, pvs_executor** out);

/*
 * Serve nq requests and return when all are done.  queries: nq x dim
 * float32, HOST memory (pinned memory makes the query copies asynchronous),
 * dim the index's dimension.  snap: the visible set the requests rank (NULL:
 * the index's current one).  Request i's ranks go to row i of ids (int64)
 * and scores (float32), nq x ranks HOST arrays; n_out[i] (host, nq entries)
 * receives how many ranks it delivered, and the rest of its row is -1 / NaN.
 * status (host, nq entries, may be NULL) receives each request's status:
 * PVS_OK (ranks delivered), PVS_EXHAUSTED (its list ended first: every
 * visible vector delivered) or its error (the ranks delivered before the
 * error stand; other requests are not affected).  ranks >= 1, 1 <= page <=
 * ranks.  Returns PVS_OK when no request failed, else the error of the
 * first failed request in request order.  Runs on one executor are
 * serialised.  Errors: PVS_ERR_INVALID for bad arguments (nothing runs).
 */
pvs_status pvs_executor_run(pvs_executor* ex, const pvs_snapshot* snap, const float* queries,
                            int32_t nq, int32_t ranks, int32_t page, int64_t* ids, float* scores,
                            int32_t* n_out, int32_t* status);

/*
 * pvs_executor_run with buffers_on_device selecting where queries, ids and
 * scores live: 0 as pvs_executor_run (host memory); 1 for device memory of
 * the index's device (nothing crosses the bus: each page is queued on the
 * worker's stream and a request is complete when the call returns).  n_out
 * and status are host arrays in both cases.
 */
pvs_status pvs_executor_run_ex(pvs_executor* ex, const pvs_snapshot* snap, const float* queries,
                               int32_t nq, int32_t ranks, int32_t page, int32_t buffers_on_device,
                               int64_t* ids, float* scores, int32_t* n_out, int32_t* status);

/*
 * Serve requests in groups of `group` (1 .. PVS_GROUP_MAX; default 1): the
 * queries of a group share one pass over the codes.  Must not be called
 * during a run.  Errors: PVS_ERR_INVALID.
 */
pvs_status pvs_executor_set_group(pvs_executor* ex, int32_t group);

pvs_status pvs_executor_stats_get(pvs_executor* ex, pvs_executor_stats* out);

/* Stop the workers (after a run in progress ends) and free the executor. */
void pvs_executor_destroy(pvs_executor* ex);

#ifdef __cplusplus
}
#endif

#endif /* PVS_EXECUTOR_H_ */
