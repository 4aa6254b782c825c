// Host-side launchers of the PBM device kernels (internal to libpvs.so).
// Method: arXiv 2608.07152 Sec. 2.3.2 (Posting Block-Max), App. A.2.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "kernels.h"

namespace pvs {

constexpr int kPbmMaxTerms = 1024;     // query terms
constexpr int kPbmChunk = 1024;        // ranges per chunk of the bound pass
constexpr int kPbmMaxBlock = 4096;     // ids per range

// Device counters of a PBM cursor (one struct, mirrored to pinned memory).
struct PbmCounters {
    unsigned long long pool_len;         // scored items appended to the pool
    unsigned long long kmax;             // max rank key over unexpanded ranges (0: none)
    unsigned long long window;           // pool keys in (kmax, last)
    unsigned long long ranges_expanded;
    unsigned long long postings;
    unsigned long long items;
    unsigned long long collected;        // pool keys gathered for an emission
    unsigned long long pos_ranges;       // ranges with H > 0 (set at open)
    int status;
    int pad;
};

// ---- index build -------------------------------------------------------------
// Marks posting i as the first of its block (new term or new range of
// `block` ids), checks ids and impacts; flags[i] = 1 for a block start.
cudaError_t launch_pbm_mark(const int64_t* term_off, int n_terms, const int32_t* docs,
                            const float* imps, int64_t n_postings, int64_t n_items, int block,
                            uint8_t* flags, int* status, cudaStream_t st);
// Blocks from the start flags, in two steps: count (tile counts scanned in
// `scratch`, the block total in *nb_out) and, once the block arrays are
// allocated, write blk_range[b] and blk_pbeg[b] for every block start.
size_t pbm_scan_scratch_elems(int64_t n_postings);
cudaError_t launch_pbm_count_blocks(const uint8_t* flags, int64_t n_postings,
                                    unsigned int* scratch, unsigned long long* nb_out,
                                    cudaStream_t st);
cudaError_t launch_pbm_write_blocks(const uint8_t* flags, const int32_t* docs, int64_t n_postings,
                                    int block, const unsigned int* scratch, int32_t* blk_range,
                                    int64_t* blk_pbeg, cudaStream_t st);
// blk_max from blk_pbeg (run after the block count is known).
cudaError_t launch_pbm_block_max(const int64_t* blk_pbeg, const float* imps, int64_t nb,
                                 float* blk_max, cudaStream_t st);
// blk_off[t] = first block whose postings start at or after term_off[t].
cudaError_t launch_pbm_term_blocks(const int64_t* term_off, int n_terms, const int64_t* blk_pbeg,
                                   int64_t nb, int64_t* blk_off, cudaStream_t st);

// ---- query open ----------------------------------------------------------------
struct PbmQuery {
    const int32_t* terms;     // [nq]
    const float* weights;     // [nq]
    int nq;
};
// starts[i * (nchunk + 1) + k] = first block of query term i with range >= k * kPbmChunk.
cudaError_t launch_pbm_starts(const PbmQuery& q, const int64_t* blk_off, const int32_t* blk_range,
                              int64_t nchunk, int64_t* starts, cudaStream_t st);
// H[r] for every range, term by term in query order; *pos_ranges counts the
// ranges with H > 0 (only they can hold an item of the support U_s).
cudaError_t launch_pbm_bounds(const PbmQuery& q, const int64_t* starts, const int32_t* blk_range,
                              const float* blk_max, int64_t n_ranges, int64_t nchunk, float* H,
                              int* status, unsigned long long* pos_ranges, cudaStream_t st);

// ---- pulls ---------------------------------------------------------------------
// rkeys[r] = key(H[r], r * block): the ranges' competition keys (sorted once,
// descending, at open; the ranges are then expanded in that order).
cudaError_t launch_pbm_range_keys(const float* H, int64_t n_ranges, int block, uint64_t* rkeys,
                                  cudaStream_t st);
// ctr->kmax = sorted[next] (0 once every range is expanded) and the pool
// keys k with ctr->kmax < k < hi (the certified window): counted in
// ctr->collected, the first `cap` of them (any order) written to out.
cudaError_t launch_pbm_window(const uint64_t* sorted, int64_t next, int64_t n_ranges,
                              const uint64_t* pool, uint64_t hi, uint64_t* out, uint64_t cap,
                              PbmCounters* ctr, cudaStream_t st);
// One CTA: when 1 <= ctr->collected <= kPbmFastWindow and either need <=
// ctr->collected or `complete` (the window holds every remaining rank),
// sorts the collected keys and writes all of them as ids / scores to h_ids /
// h_scores; always copies *ctr to *h_mirror last.  h_* may be pinned host
// memory.
constexpr int kPbmFastWindow = 8192;
cudaError_t launch_pbm_finish(const uint64_t* keys, const PbmCounters* ctr, uint64_t need,
                              bool complete, int64_t* h_ids, float* h_scores,
                              PbmCounters* h_mirror, cudaStream_t st);
struct PbmExpandArgs {
    const uint64_t* ranges;       // sorted range keys of the ranges to expand
    int64_t count;                // how many
    PbmQuery q;
    const int64_t* starts;
    int64_t nchunk;
    const int32_t* blk_range;
    const int64_t* blk_pbeg;
    const int32_t* docs;
    const float* imps;
    int64_t n_items;
    int block;
    const uint32_t* tomb;         // deleted items (bit per id), null: none
    uint64_t* pool;
    PbmCounters* ctr;
};
cudaError_t launch_pbm_expand(const PbmExpandArgs& a, int grid, cudaStream_t st);
// Pool keys k with ctr->kmax < k < hi and k >= *from (from may be null)
// appended to out in any order (ctr->collected counts them; at most cap written).
cudaError_t launch_pbm_collect(const uint64_t* pool, const unsigned long long* from, uint64_t hi,
                               uint64_t* out, uint64_t cap, PbmCounters* ctr, cudaStream_t st);
// 64-bit radix selection: sel64[0] = the k-th largest (1-based) pool key k'
// with ctr->kmax < k' < hi; sel64 holds 2 + 256 words of state.
cudaError_t launch_pbm_select64(const uint64_t* pool, const PbmCounters* ctr, uint64_t hi,
                                uint64_t k, unsigned long long* sel64, cudaStream_t st);
// ids[i], scores[i] of the first m keys of a descending key array.
cudaError_t launch_pbm_emit(const uint64_t* keys, int m, int64_t* ids, float* scores,
                            cudaStream_t st);
// Complete sparse scores: for each query term j in order,
// acc[x] = RN(acc[x] + RN(q_j p_j(x))) over the term's postings (acc zeroed
// by the caller), the evaluation of the expand kernel for every item.
cudaError_t launch_pbm_score_all(const PbmQuery& q, const int64_t* term_off, const int32_t* docs,
                                 const float* imps, float* acc, int grid, cudaStream_t st);
// keys[0 .. *count) = rank keys of the visible items with acc > 0, in any
// order (*count zeroed by the caller).
cudaError_t launch_pbm_member_keys(const float* acc, int64_t n, const uint32_t* tomb,
                                   uint64_t* keys, unsigned long long* count, int grid,
                                   cudaStream_t st);
// rank_of[id of keys[i]] = i + 1 for i < m (keys sorted descending).
cudaError_t launch_pbm_rank_of(const uint64_t* keys, int64_t m, int32_t* rank_of, int grid,
                               cudaStream_t st);

}  // namespace pvs
