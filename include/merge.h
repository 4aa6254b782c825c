/*
 * merge.h -- hierarchical Segment / Shard merging in libpvs.so.
 *
 * Method: arXiv 2608.07152 Sec. 2.4: every Segment produces a tie-complete
 * exact ranking; the rankings are merged within a Shard and then across
 * Shards under the same (score descending, identifier ascending) order into
 * one resumable request-level ranking; copies of one item in several
 * Segments with consistent scores are merged, conflicting copies invalidate
 * the request.  Ranked-list contract: Sec. 2.1.
 *
 * A merge cursor reads its children (PVS cursors, PBM cursors or other merge
 * cursors, so a Shard of Segments and a request of Shards are both merge
 * cursors) in chunks, keeps what it has read but not yet delivered, and
 * delivers the merged order.  Children due for more ranks at the same time
 * are read concurrently, one host thread each: children on streams of their
 * own (e.g. Segment indexes built without a shared stream) then also overlap
 * on the device.  A child's ids are mapped to the request's id
 * space by adding the child's id_offset.  Copies: an item delivered by two
 * children with the same score is delivered once (they are adjacent in the
 * merged order); the same id with another score fails the merge cursor with
 * PVS_ERR_INVALID.
 *
 * Conventions as pvs.h: negative statuses are errors and fail the merge
 * cursor for good; the caller owns every buffer; the merge cursor does not
 * own its children (close them after the merge cursor); children must be
 * fresh (nothing pulled yet) and used by nothing else while merged.
 */
#ifndef PVS_MERGE_H_
#define PVS_MERGE_H_

#include <stdint.h>

#include "pbm.h"
#include "pvs.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pvs_merge pvs_merge;

typedef enum pvs_child_kind {
    PVS_CHILD_DENSE = 0,    /* pvs_cursor*  */
    PVS_CHILD_SPARSE = 1,   /* pbm_cursor*  */
    PVS_CHILD_MERGE = 2     /* pvs_merge*   */
} pvs_child_kind;

typedef struct pvs_merge_child {
    int32_t kind;           /* pvs_child_kind                                  */
    int32_t reserved;
    void* cursor;           /* the child, not owned                            */
    int64_t id_offset;      /* request id = child id + id_offset (>= 0)        */
} pvs_merge_child;

typedef struct pvs_merge_stats {
    int64_t emitted;        /* ranks delivered                                 */
    int64_t read;           /* ranks read from the children                    */
    int64_t duplicates;     /* copies merged away                              */
    int64_t child_pulls;    /* next calls on the children                      */
    int64_t id_space;       /* request ids lie in [0, id_space)                */
    int64_t length;         /* sum of the children's list lengths (an upper
                               bound of the merged length)                     */
    int32_t state;          /* PVS_OK, PVS_EXHAUSTED or an error               */
    int32_t reserved;
} pvs_merge_stats;

/*
 * Open a merge cursor over count (1 .. 1024) children.  Errors:
 * PVS_ERR_INVALID (null or repeated child, unknown kind, negative offset, a
 * child that was already pulled or has failed, ids beyond 2^31), PVS_ERR_OOM.
 */
pvs_status pvs_merge_open(const pvs_merge_child* children, int32_t count, pvs_merge** out);

/*
 * The next up to n merged ranks (request ids, scores) into host buffers.
 * PVS_OK, or PVS_EXHAUSTED once every child is exhausted and everything
 * read has been delivered (then *n_out <= n).  Errors: a child's error,
 * PVS_ERR_INVALID (n < 1, conflicting copies), PVS_ERR_FAILED.
 */
pvs_status pvs_merge_next(pvs_merge* merge, int32_t n, int64_t* ids, float* scores,
                          int32_t* n_out);
pvs_status pvs_merge_stats_get(pvs_merge* merge, pvs_merge_stats* out);
void pvs_merge_close(pvs_merge* merge);

/*
 * EAHR (Sec. 2.2) with both channels read from merge cursors (a channel of
 * one Segment is a merge cursor of one child).  Both must be fresh.  The
 * request's id space is the larger of the two channels'.  Errors as
 * eahr_topk, and PVS_ERR_INVALID for conflicting copies in a channel.
 */
pvs_status eahr_topk_merge(pvs_merge* dense, pvs_merge* sparse, const eahr_params* p,
                           int64_t* out_ids, double* out_F, int32_t* n_out, eahr_stats* st);

#ifdef __cplusplus
}
#endif

#endif /* PVS_MERGE_H_ */
