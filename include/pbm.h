/*
 * pbm.h -- C ABI of the PBM sparse rank generator in libpvs.so.
 *
 * Method: arXiv 2608.07152, Sec. 2.3.2 (Posting Block-Max) and Appendix A.2
 * (its float32 range bound); the ranked-list contract is Sec. 2.1.
 *
 * PBM produces the complete exact sparse ranked list of a query: its
 * support U_s is the set of items with a positive sparse score
 * S(x) = sum_t q_t p_t(x) (Sec. 2.1: items outside U_s have no rank and
 * contribute nothing to fusion), ordered by S descending, ties by ascending
 * id.  Items with no matching posting, with only zero impacts or zero-weight
 * terms, or whose float32 score rounds to 0, are not in the list; neither
 * are items a snapshot deletes (pbm_cursor_open_snapshot).  PBM partitions
 * the id space into ranges of `block` consecutive ids, bounds every range by
 * H(R) = sum_t q_t m_t(R) with the block maxima m_t(R), expands the ranges
 * with H > 0 in decreasing order of H and publishes a rank once no
 * unexpanded range can hold an item ranked before it.  Ranks come in chunks
 * on demand; the cursor keeps the unexpanded ranges and the scored items
 * between calls.
 *
 * Float32 evaluation (App. A.2; readings of this library): both S and H
 * are accumulated term by term in the order the query lists its terms, each
 * step a float32 product rounded to nearest-even followed by a float32 sum
 * rounded to nearest-even (no fused multiply-add), starting from +0.  With
 * nonnegative finite inputs this keeps S_hat(x) <= H_hat(R) for x in R.
 *
 * Conventions: pbm_* calls return the pvs_status codes of pvs.h with the
 * same meaning; on an error nothing is produced and a cursor becomes Failed
 * for good.  The library owns pbm_index and pbm_cursor objects; the caller
 * owns every buffer it passes.  Distinct cursors may be used from different
 * host threads; one cursor by one thread at a time; pbm_index_free must not
 * overlap any other call on the index.
 */
#ifndef PBM_H_
#define PBM_H_

#include <stdint.h>

#include "pvs.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pbm_index pbm_index;
typedef struct pbm_cursor pbm_cursor;

/* Counters of one PBM cursor (the sparse counters of Sec. 3.5). */
typedef struct pbm_stats {
    int64_t items;             /* N, the id space (|U_s| <= N)               */
    int64_t emitted;           /* ranks delivered so far (= |U_s| once the
                                  list is Exhausted)                         */
    int64_t ranges;            /* ranges of the id space                     */
    int64_t ranges_expanded;   /* ranges whose items were scored             */
    int64_t postings_visited;  /* postings read while scoring               */
    int64_t items_scored;      /* items of expanded ranges (scored exactly)  */
    int64_t pulls;             /* pbm_next calls                             */
    int64_t rounds;            /* expand-and-certify rounds over all pulls   */
    int64_t pulls_from_window; /* pulls served on the host from an earlier
                                  pull's certified window (no device work)  */
    int32_t state;             /* PVS_OK, PVS_EXHAUSTED or an error          */
    int32_t reserved;
} pbm_stats;

/*
 * Build the PBM index of N = n_items items from term-major postings
 * (Sec. 2.3.2): the postings of term t are entries term_off[t] ..
 * term_off[t+1]-1 of docs / imps.  term_off: n_terms + 1 int64, term_off[0]
 * = 0, nondecreasing, term_off[n_terms] = n_postings.  docs: int32 item ids
 * in [0, n_items), strictly ascending within a term.  imps: float32 impacts,
 * finite and >= 0 (App. A.2).  block: range length in ids, 1 .. 4096 (0: the
 * default 128).  on_device: 1 when the three arrays are device memory of
 * the current device, 0 for host memory.  The arrays are copied; the caller
 * keeps them.  cuda_stream: stream for the build and for the cursors' work
 * (NULL: a library-created stream).
 * Errors: PVS_ERR_INVALID for a malformed array or size (checked on the
 * device, the whole index is rejected), PVS_ERR_NONFINITE for a non-finite
 * impact, PVS_ERR_OOM, PVS_ERR_CUDA.
 */
pvs_status pbm_build(const int64_t* term_off, int32_t n_terms, const int32_t* docs,
                     const float* imps, int64_t n_postings, int64_t n_items, int32_t block,
                     int32_t on_device, void* cuda_stream, pbm_index** out);
int64_t pbm_index_items(const pbm_index* index);
int64_t pbm_index_ranges(const pbm_index* index);
void pbm_index_free(pbm_index* index);   /* cursors must be closed first */

/*
 * Open a cursor for the query {(terms[i], weights[i])}, i < nq, whose
 * listed order is the summation order sigma (App. A.2).  terms: distinct
 * ids in [0, n_terms); weights: finite, >= 0 (a zero weight contributes
 * nothing).  nq may be 0 (every score is 0: the ranked list is empty);
 * nq <= 1024.  Host arrays; copied.  The range bounds H(R) are computed
 * here.  Errors: PVS_ERR_INVALID (bad term, repeated term, nq out of
 * range), PVS_ERR_NONFINITE (non-finite weight), PVS_ERR_OOM, PVS_ERR_CUDA.
 */
pvs_status pbm_cursor_open(pbm_index* index, const int32_t* terms, const float* weights,
                           int32_t nq, pbm_cursor** out);

/*
 * pbm_cursor_open over the visible set of a PVS snapshot (Sec. 2.4: every
 * channel of a request ranks the items of one fixed snapshot): items the
 * snapshot deletes are outside the ranked list.  The snapshot's rows must
 * be the PBM index's items (same id space, snapshot rows == n_items) and its
 * index on the same device; the snapshot may be freed while the cursor is
 * open.  snap NULL is pbm_cursor_open.  Errors as pbm_cursor_open, and
 * PVS_ERR_INVALID for a snapshot of another size or device.
 */
pvs_status pbm_cursor_open_snapshot(pbm_index* index, const pvs_snapshot* snap,
                                    const int32_t* terms, const float* weights, int32_t nq,
                                    pbm_cursor** out);

/*
 * pbm_cursor_open_snapshot with the cursor's device work (the bounds at open
 * and every pull) on cuda_stream (a cudaStream_t of the index's device, not
 * owned; NULL: the index's stream).  Cursors on streams of their own serve
 * requests from several host threads concurrently.  Closed cursors keep
 * their buffers for later opens of the same index (up to 32 of them).
 * Errors as pbm_cursor_open_snapshot.
 */
pvs_status pbm_cursor_open_stream(pbm_index* index, const pvs_snapshot* snap,
                                  const int32_t* terms, const float* weights, int32_t nq,
                                  void* cuda_stream, pbm_cursor** out);

/*
 * The next up to n ranks (n >= 1): ids (int64) and their scores S_hat
 * (float32, all > 0) in host memory, *n_out of them.  Returns PVS_OK, or
 * PVS_EXHAUSTED once the last item of the support has been delivered (then
 * *n_out < n, or *n_out == n for the call that delivers the last item;
 * later calls deliver 0).  Output is an
 * append-only exact prefix (Sec. 2.1).  A pull whose certified window (every
 * scored item above the bound of every range not yet expanded, at most 8,192
 * of them) holds more ranks than requested keeps the rest in the cursor's
 * pinned memory: later pulls that fit in them are served there, with no
 * device work (pbm_stats.pulls_from_window).  Errors: PVS_ERR_INVALID (n < 1,
 * null pointer), PVS_ERR_OVERFLOW (a score or bound overflowed float32),
 * PVS_ERR_OOM, PVS_ERR_CUDA, PVS_ERR_FAILED (the cursor failed earlier).
 */
pvs_status pbm_next(pbm_cursor* cursor, int32_t n, int64_t* ids, float* scores, int32_t* n_out);

/*
 * The range bounds H_hat(R) the cursor computed at open, for ranges first ..
 * first+count-1 (host float32 output; ranges already expanded still report
 * their bound).  For tests and diagnostics.
 */
pvs_status pbm_cursor_range_bounds(pbm_cursor* cursor, int64_t first, int64_t count, float* H);

pvs_status pbm_cursor_stats(pbm_cursor* cursor, pbm_stats* out);
void pbm_cursor_close(pbm_cursor* cursor);

/*
 * EAHR (Sec. 2.2) over a dense PVS cursor and a sparse PBM cursor, both
 * unused so far: the same contract as eahr_topk with the sparse ranks pulled
 * from PBM instead of a host array.  Both channels must see one visible set
 * (Sec. 2.4): the PBM index's items are the dense snapshot's rows, and the
 * PBM cursor deletes what the dense cursor's snapshot deletes (open it with
 * pbm_cursor_open_snapshot on that snapshot, or with pbm_cursor_open when
 * nothing is deleted); else PVS_ERR_INVALID.  The sparse support U_s is
 * usually much smaller than the visible set; items outside it contribute
 * nothing (Sec. 2.1).  Under EAHR_POLICY_ADAPTIVE a helper thread computes
 * the query's complete PBM ranking on the device (every item's S in the
 * query's term order, the visible items with S > 0 sorted by (S desc, id
 * asc)) while the lists are read, and the exact finish takes the
 * candidates' missing sparse ranks from it.
 */
pvs_status eahr_topk_pbm(pvs_cursor* dense, pbm_cursor* sparse, const eahr_params* p,
                         int64_t* out_ids, double* out_F, int32_t* n_out, eahr_stats* st);

#ifdef __cplusplus
}
#endif

#endif /* PBM_H_ */
