// PBM (Posting Block-Max) device kernels: arXiv 2608.07152 Sec. 2.3.2 and
// App. A.2.
//
// Index: term-major postings (docs ascending within a term) cut into blocks,
// one block per (term, range of `block` consecutive ids) that holds postings;
// a block records its range, its first posting and its maximum impact m_t(R).
//
// Query: H(R) = sum_t q_t m_t(R) for every range, and S(x) for the items of
// an expanded range, both accumulated term by term in the query's order with
// a float32 product and a float32 sum, each rounded to nearest-even
// (App. A.2: the same operations in the same order keep S_hat <= H_hat).
// Sequential term order per range or item comes from processing one query
// term at a time inside a CTA that owns the range (or the range chunk), with
// a barrier between terms; each range or item receives at most one
// contribution per term, so no two threads touch one accumulator at once.
//
// Ranking keys are the 64-bit rank keys (score descending, id ascending) of
// pvs_common.cuh; a range R competes with the key of (H(R), first id of R):
// an item y of R precedes x only if key(S(y), y) > key(S(x), x), and
// key(S(y), y) <= key(H(R), R.first) because S(y) <= H(R) and y >= R.first.
#include <cstdint>

#include "pbm_kernels.h"
#include "pvs_common.cuh"

namespace pvs {

namespace {

constexpr int kTile = 4096;          // postings per CTA of the block scan
constexpr int kScanThreads = 256;    // 16 postings per thread

__device__ __forceinline__ int64_t lower_bound_i32(const int32_t* a, int64_t lo, int64_t hi,
                                                   int64_t v) {
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if ((int64_t)a[mid] < v)
            lo = mid + 1;
        else
            hi = mid;
    }
    return lo;
}

__device__ __forceinline__ int64_t lower_bound_i64(const int64_t* a, int64_t lo, int64_t hi,
                                                   int64_t v) {
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if (a[mid] < v)
            lo = mid + 1;
        else
            hi = mid;
    }
    return lo;
}

int grid_for(int64_t n, int threads, int cap = 152 * 16) {
    int64_t g = (n + threads - 1) / threads;
    if (g < 1) g = 1;
    if (g > cap) g = cap;
    return (int)g;
}

}  // namespace

// ---------------------------------------------------------------------------
// index build
// ---------------------------------------------------------------------------

__global__ void pbm_term_starts_kernel(const int64_t* __restrict__ term_off, int n_terms,
                                       uint8_t* flags) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t < n_terms && term_off[t] < term_off[t + 1]) flags[term_off[t]] = 2;   // term start
}

// flags[i]: 2 = first posting of a term (set above), 1 = first posting of a
// new range within a term, 0 otherwise; ids checked in range and strictly
// ascending within a term, impacts finite and nonnegative.
__global__ void pbm_mark_kernel(const int32_t* __restrict__ docs, const float* __restrict__ imps,
                                int64_t n, int64_t n_items, int block, uint8_t* flags,
                                int* status) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const int32_t d = docs[i];
        const float p = imps[i];
        if (d < 0 || (int64_t)d >= n_items) set_status(status, PVS_ERR_INVALID);
        if (!isfinite(p))
            set_status(status, PVS_ERR_NONFINITE);
        else if (p < 0.0f)
            set_status(status, PVS_ERR_INVALID);
        if (flags[i] == 2 || i == 0) continue;
        const int32_t prev = docs[i - 1];
        if (d <= prev) set_status(status, PVS_ERR_INVALID);
        if (d / block != prev / block) flags[i] = 1;
    }
}

cudaError_t launch_pbm_mark(const int64_t* term_off, int n_terms, const int32_t* docs,
                            const float* imps, int64_t n_postings, int64_t n_items, int block,
                            uint8_t* flags, int* status, cudaStream_t st) {
    if (n_postings <= 0) return cudaSuccess;
    cudaError_t e = cudaMemsetAsync(flags, 0, (size_t)n_postings, st);
    if (e != cudaSuccess) return e;
    count_launches(2);
    pbm_term_starts_kernel<<<(n_terms + 255) / 256, 256, 0, st>>>(term_off, n_terms, flags);
    pbm_mark_kernel<<<grid_for(n_postings, 256), 256, 0, st>>>(docs, imps, n_postings, n_items,
                                                               block, flags, status);
    return cudaGetLastError();
}

size_t pbm_scan_scratch_elems(int64_t n_postings) {
    return (size_t)((n_postings + kTile - 1) / kTile) + 1;
}

__global__ void __launch_bounds__(kScanThreads) pbm_tile_count_kernel(const uint8_t* flags,
                                                                      int64_t n,
                                                                      unsigned int* tile_cnt) {
    const int64_t base = (int64_t)blockIdx.x * kTile;
    unsigned int c = 0;
    for (int j = threadIdx.x; j < kTile; j += kScanThreads) {
        const int64_t i = base + j;
        if (i < n && flags[i] != 0) ++c;
    }
    c = warp_sum(c);
    __shared__ unsigned int ws[kScanThreads / 32];
    if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = c;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned int t = 0;
        for (int w = 0; w < kScanThreads / 32; ++w) t += ws[w];
        tile_cnt[blockIdx.x] = t;
    }
}

// In-place exclusive scan of n counts by one CTA; total to *total.
__global__ void __launch_bounds__(1024) pbm_scan_kernel(unsigned int* cnt, int64_t n,
                                                        unsigned long long* total) {
    __shared__ unsigned long long part[1024];
    const int64_t per = (n + 1023) / 1024;
    const int64_t b = threadIdx.x * per, e = b + per < n ? b + per : n;
    unsigned long long s = 0;
    for (int64_t i = b; i < e; ++i) s += cnt[i];
    part[threadIdx.x] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned long long run = 0;
        for (int t = 0; t < 1024; ++t) {
            const unsigned long long x = part[t];
            part[t] = run;
            run += x;
        }
        *total = run;
    }
    __syncthreads();
    unsigned long long run = part[threadIdx.x];
    for (int64_t i = b; i < e; ++i) {
        const unsigned int x = cnt[i];
        cnt[i] = (unsigned int)run;
        run += x;
    }
}

cudaError_t launch_pbm_count_blocks(const uint8_t* flags, int64_t n_postings,
                                    unsigned int* scratch, unsigned long long* nb_out,
                                    cudaStream_t st) {
    const int64_t tiles = (n_postings + kTile - 1) / kTile;
    if (tiles == 0) return cudaMemsetAsync(nb_out, 0, sizeof(unsigned long long), st);
    count_launches(2);
    pbm_tile_count_kernel<<<(unsigned)tiles, kScanThreads, 0, st>>>(flags, n_postings, scratch);
    pbm_scan_kernel<<<1, 1024, 0, st>>>(scratch, tiles, nb_out);
    return cudaGetLastError();
}

// Block b = tile base + rank of the start among the tile's starts (in order).
__global__ void __launch_bounds__(kScanThreads) pbm_write_blocks_kernel(
    const uint8_t* flags, const int32_t* __restrict__ docs, int64_t n, int block,
    const unsigned int* tile_base, int32_t* blk_range, int64_t* blk_pbeg) {
    constexpr int kPer = kTile / kScanThreads;   // consecutive postings per thread
    const int64_t base = (int64_t)blockIdx.x * kTile + (int64_t)threadIdx.x * kPer;
    unsigned int c = 0;
    for (int j = 0; j < kPer; ++j) {
        const int64_t i = base + j;
        if (i < n && flags[i] != 0) ++c;
    }
    // exclusive scan of c over the CTA
    __shared__ unsigned int ws[kScanThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned int inc = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned int y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
    }
    if (lane == 31) ws[warp] = inc;
    __syncthreads();
    unsigned int wbase = 0;
    for (int w = 0; w < warp; ++w) wbase += ws[w];
    unsigned int pos = tile_base[blockIdx.x] + wbase + inc - c;
    for (int j = 0; j < kPer; ++j) {
        const int64_t i = base + j;
        if (i < n && flags[i] != 0) {
            blk_range[pos] = docs[i] / block;
            blk_pbeg[pos] = i;
            ++pos;
        }
    }
}

cudaError_t launch_pbm_write_blocks(const uint8_t* flags, const int32_t* docs, int64_t n_postings,
                                    int block, const unsigned int* scratch, int32_t* blk_range,
                                    int64_t* blk_pbeg, cudaStream_t st) {
    const int64_t tiles = (n_postings + kTile - 1) / kTile;
    if (tiles == 0) return cudaSuccess;
    count_launches(1);
    pbm_write_blocks_kernel<<<(unsigned)tiles, kScanThreads, 0, st>>>(
        flags, docs, n_postings, block, scratch, blk_range, blk_pbeg);
    return cudaGetLastError();
}

__global__ void pbm_block_max_kernel(const int64_t* __restrict__ blk_pbeg,
                                     const float* __restrict__ imps, int64_t nb, float* blk_max) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < nb; b += stride) {
        float m = 0.0f;
        for (int64_t p = blk_pbeg[b]; p < blk_pbeg[b + 1]; ++p) m = fmaxf(m, imps[p]);
        blk_max[b] = m;
    }
}

cudaError_t launch_pbm_block_max(const int64_t* blk_pbeg, const float* imps, int64_t nb,
                                 float* blk_max, cudaStream_t st) {
    if (nb <= 0) return cudaSuccess;
    count_launches(1);
    pbm_block_max_kernel<<<grid_for(nb, 256), 256, 0, st>>>(blk_pbeg, imps, nb, blk_max);
    return cudaGetLastError();
}

__global__ void pbm_term_blocks_kernel(const int64_t* __restrict__ term_off, int n_terms,
                                       const int64_t* __restrict__ blk_pbeg, int64_t nb,
                                       int64_t* blk_off) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t > n_terms) return;
    blk_off[t] = t == n_terms ? nb : lower_bound_i64(blk_pbeg, 0, nb, term_off[t]);
}

cudaError_t launch_pbm_term_blocks(const int64_t* term_off, int n_terms, const int64_t* blk_pbeg,
                                   int64_t nb, int64_t* blk_off, cudaStream_t st) {
    count_launches(1);
    pbm_term_blocks_kernel<<<(n_terms + 1 + 255) / 256, 256, 0, st>>>(term_off, n_terms, blk_pbeg,
                                                                      nb, blk_off);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// query open: range bounds
// ---------------------------------------------------------------------------

__global__ void pbm_starts_kernel(PbmQuery q, const int64_t* __restrict__ blk_off,
                                  const int32_t* __restrict__ blk_range, int64_t nchunk,
                                  int64_t* starts) {
    const int64_t per = nchunk + 1;
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (int64_t)q.nq * per) return;
    const int i = (int)(idx / per);
    const int64_t k = idx % per;
    const int t = q.terms[i];
    starts[idx] = lower_bound_i32(blk_range, blk_off[t], blk_off[t + 1], k * kPbmChunk);
}

cudaError_t launch_pbm_starts(const PbmQuery& q, const int64_t* blk_off, const int32_t* blk_range,
                              int64_t nchunk, int64_t* starts, cudaStream_t st) {
    const int64_t n = (int64_t)q.nq * (nchunk + 1);
    if (n == 0) return cudaSuccess;
    count_launches(1);
    pbm_starts_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(q, blk_off, blk_range, nchunk,
                                                                   starts);
    return cudaGetLastError();
}

// One CTA per chunk of kPbmChunk ranges: term by term in query order,
// H[r] <- RN(H[r] + RN(q_t * m_t(r))) for the chunk's blocks of term t.
__global__ void __launch_bounds__(256) pbm_bounds_kernel(PbmQuery q,
                                                         const int64_t* __restrict__ starts,
                                                         const int32_t* __restrict__ blk_range,
                                                         const float* __restrict__ blk_max,
                                                         int64_t n_ranges, int64_t nchunk,
                                                         float* H, int* status,
                                                         unsigned long long* pos_ranges) {
    __shared__ float h[kPbmChunk];
    const int64_t k = blockIdx.x;
    const int64_t r0 = k * kPbmChunk;
    for (int x = threadIdx.x; x < kPbmChunk; x += blockDim.x) h[x] = 0.0f;
    __syncthreads();
    const int64_t per = nchunk + 1;
    for (int i = 0; i < q.nq; ++i) {
        const float w = q.weights[i];
        const int64_t s0 = starts[i * per + k], s1 = starts[i * per + k + 1];
        for (int64_t j = s0 + threadIdx.x; j < s1; j += blockDim.x) {
            const int64_t x = (int64_t)blk_range[j] - r0;
            if (x >= 0 && x < kPbmChunk)
                h[x] = __fadd_rn(h[x], __fmul_rn(w, blk_max[j]));
            else
                set_status(status, PVS_ERR_INVALID);   // metadata out of order
        }
        __syncthreads();
    }
    // kPbmChunk is a multiple of the block size: whole warps run every trip
    for (int x = threadIdx.x; x < kPbmChunk; x += blockDim.x) {
        const bool in = r0 + x < n_ranges;
        const float v = in ? h[x] : 0.0f;
        if (in) {
            if (!isfinite(v)) set_status(status, PVS_ERR_OVERFLOW);
            H[r0 + x] = v;
        }
        const unsigned int pos = __ballot_sync(0xffffffffu, in && v > 0.0f);
        if ((threadIdx.x & 31) == 0 && pos)
            atomicAdd(pos_ranges, (unsigned long long)__popc(pos));
    }
}

cudaError_t launch_pbm_bounds(const PbmQuery& q, const int64_t* starts, const int32_t* blk_range,
                              const float* blk_max, int64_t n_ranges, int64_t nchunk, float* H,
                              int* status, unsigned long long* pos_ranges, cudaStream_t st) {
    static_assert(kPbmChunk % 256 == 0, "whole warps in the bound pass's count");
    if (nchunk <= 0) return cudaSuccess;
    count_launches(1);
    pbm_bounds_kernel<<<(unsigned)nchunk, 256, 0, st>>>(q, starts, blk_range, blk_max, n_ranges,
                                                        nchunk, H, status, pos_ranges);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// pulls
// ---------------------------------------------------------------------------

__global__ void pbm_range_keys_kernel(const float* __restrict__ H, int64_t n, int block,
                                      uint64_t* rkeys) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n; r += stride)
        rkeys[r] = rank_key(H[r], (uint32_t)(r * block));
}

cudaError_t launch_pbm_range_keys(const float* H, int64_t n_ranges, int block, uint64_t* rkeys,
                                  cudaStream_t st) {
    if (n_ranges <= 0) return cudaSuccess;
    count_launches(1);
    pbm_range_keys_kernel<<<grid_for(n_ranges, 256, 152 * 4), 256, 0, st>>>(H, n_ranges, block,
                                                                            rkeys);
    return cudaGetLastError();
}

__global__ void pbm_window_kernel(const uint64_t* __restrict__ sorted, int64_t next,
                                  int64_t n_ranges, const uint64_t* __restrict__ pool,
                                  uint64_t hi, uint64_t* out, uint64_t cap, PbmCounters* ctr) {
    const unsigned long long lo = next < n_ranges ? sorted[next] : 0ull;
    if (blockIdx.x == 0 && threadIdx.x == 0) ctr->kmax = lo;
    const int64_t n = (int64_t)ctr->pool_len;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int lane = threadIdx.x & 31;
    // whole warps iterate together so that the appends can be aggregated
    for (int64_t i0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); i0 < n;
         i0 += stride) {
        const int64_t i = i0 + lane;
        uint64_t k = 0;
        bool take = false;
        if (i < n) {
            k = pool[i];
            take = k > lo && k < hi;
        }
        const unsigned int m = __ballot_sync(0xffffffffu, take);
        if (m == 0) continue;
        unsigned long long base = 0;
        if (lane == 0) base = atomicAdd(&ctr->collected, (unsigned long long)__popc(m));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (take) {
            const unsigned long long pos = base + __popc(m & ((1u << lane) - 1u));
            if (pos < cap) out[pos] = k;
        }
    }
}

cudaError_t launch_pbm_window(const uint64_t* sorted, int64_t next, int64_t n_ranges,
                              const uint64_t* pool, uint64_t hi, uint64_t* out, uint64_t cap,
                              PbmCounters* ctr, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(&ctr->collected, 0, sizeof(unsigned long long), st);
    if (e != cudaSuccess) return e;
    count_launches(1);
    pbm_window_kernel<<<152 * 4, 256, 0, st>>>(sorted, next, n_ranges, pool, hi, out, cap, ctr);
    return cudaGetLastError();
}

constexpr int kFinishThreads = 1024;

__global__ void __launch_bounds__(kFinishThreads) pbm_finish_kernel(const uint64_t* keys_in,
                                                                    const PbmCounters* ctr,
                                                                    uint64_t need, int complete,
                                                                    int64_t* h_ids,
                                                                    float* h_scores,
                                                                    PbmCounters* h_mirror) {
    extern __shared__ uint64_t keys[];
    const unsigned long long count = ctr->collected;
    if (need > 0 && count >= 1 && (count >= need || complete) &&
        count <= (unsigned long long)kPbmFastWindow) {
        int pow2 = 1;
        while ((unsigned long long)pow2 < count) pow2 <<= 1;
        for (int i = threadIdx.x; i < pow2; i += blockDim.x)
            keys[i] = (unsigned long long)i < count ? keys_in[i] : 0ull;   // 0 sorts last
        __syncthreads();
        // bitonic sort, descending
        for (int k = 2; k <= pow2; k <<= 1) {
            for (int j = k >> 1; j > 0; j >>= 1) {
                for (int i = threadIdx.x; i < pow2; i += blockDim.x) {
                    const int ixj = i ^ j;
                    if (ixj > i) {
                        const uint64_t a = keys[i], b = keys[ixj];
                        const bool swap = (i & k) == 0 ? a < b : a > b;
                        if (swap) {
                            keys[i] = b;
                            keys[ixj] = a;
                        }
                    }
                }
                __syncthreads();
            }
        }
        // the whole window, sorted: every key in it is certified, so the
        // host can serve later pulls from what lies beyond `need`
        for (int i = threadIdx.x; (unsigned long long)i < count; i += blockDim.x) {
            h_ids[i] = (int64_t)rank_key_id(keys[i]);
            h_scores[i] = rank_key_score(keys[i]);
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) *h_mirror = *ctr;
}

cudaError_t launch_pbm_finish(const uint64_t* keys, const PbmCounters* ctr, uint64_t need,
                              bool complete, int64_t* h_ids, float* h_scores,
                              PbmCounters* h_mirror, cudaStream_t st) {
    cudaError_t e = raise_smem_limit((const void*)pbm_finish_kernel,
                                     kPbmFastWindow * sizeof(uint64_t));
    if (e != cudaSuccess) return e;
    count_launches(1);
    pbm_finish_kernel<<<1, kFinishThreads, kPbmFastWindow * sizeof(uint64_t), st>>>(
        keys, ctr, need, complete ? 1 : 0, h_ids, h_scores, h_mirror);
    return cudaGetLastError();
}

// One CTA per range at a time: the range's block of every query term
// (binary search within the term's blocks of the range's chunk), then the
// postings term by term in query order into the items' float32 scores,
// then every item of the range goes to the pool with its rank key.  Items
// outside the support (S = 0, Sec. 2.1: no rank) and deleted items get key 0,
// which lies below every real key and every window bound, so no window takes
// them.
constexpr int kExpandThreads = 256;

__global__ void __launch_bounds__(kExpandThreads) pbm_expand_kernel(PbmExpandArgs a) {
    __shared__ float s[kPbmMaxBlock];
    __shared__ float w[kPbmMaxTerms];
    __shared__ int64_t pb[kPbmMaxTerms];
    __shared__ int64_t pe[kPbmMaxTerms];
    __shared__ unsigned long long base_sh;
    const int nq = a.q.nq;
    for (int i = threadIdx.x; i < nq; i += blockDim.x) w[i] = a.q.weights[i];
    const int64_t per = a.nchunk + 1;
    for (int64_t e = blockIdx.x; e < a.count; e += gridDim.x) {
        const int64_t r = (int64_t)rank_key_id(a.ranges[e]) / a.block;
        const int64_t k = r / kPbmChunk;
        const int64_t first = r * a.block;
        const int64_t rest = a.n_items - first;
        const int cnt = (int)(rest < a.block ? rest : a.block);
        for (int i = threadIdx.x; i < nq; i += blockDim.x) {
            const int64_t s0 = a.starts[i * per + k], s1 = a.starts[i * per + k + 1];
            const int64_t j = lower_bound_i32(a.blk_range, s0, s1, r);
            if (j < s1 && a.blk_range[j] == r) {
                pb[i] = a.blk_pbeg[j];
                pe[i] = a.blk_pbeg[j + 1];
            } else {
                pb[i] = pe[i] = 0;
            }
        }
        for (int x = threadIdx.x; x < cnt; x += blockDim.x) s[x] = 0.0f;
        __syncthreads();
        unsigned long long visited = 0;
        for (int i = 0; i < nq; ++i) {
            const int64_t b0 = pb[i], b1 = pe[i];
            if (b1 <= b0) continue;                    // the same for every thread
            visited += (unsigned long long)(b1 - b0);
            const float wi = w[i];
            for (int64_t p = b0 + threadIdx.x; p < b1; p += blockDim.x) {
                const int64_t x = (int64_t)a.docs[p] - first;
                if (x >= 0 && x < cnt)
                    s[x] = __fadd_rn(s[x], __fmul_rn(wi, a.imps[p]));
                else
                    set_status(&a.ctr->status, PVS_ERR_INVALID);   // metadata out of order
            }
            __syncthreads();
        }
        if (threadIdx.x == 0) {
            base_sh = atomicAdd(&a.ctr->pool_len, (unsigned long long)cnt);
            atomicAdd(&a.ctr->ranges_expanded, 1ull);
            atomicAdd(&a.ctr->postings, visited);
            atomicAdd(&a.ctr->items, (unsigned long long)cnt);
        }
        __syncthreads();
        const unsigned long long base = base_sh;
        for (int x = threadIdx.x; x < cnt; x += blockDim.x) {
            const float v = s[x];
            if (!isfinite(v)) set_status(&a.ctr->status, PVS_ERR_OVERFLOW);
            const int64_t id = first + x;
            const bool dead =
                a.tomb != nullptr && ((__ldg(a.tomb + (id >> 5)) >> (id & 31)) & 1u);
            a.pool[base + x] = (v > 0.0f && !dead) ? rank_key(v, (uint32_t)id) : 0ull;
        }
        __syncthreads();   // s, pb, pe are reused by the next range
    }
}

cudaError_t launch_pbm_expand(const PbmExpandArgs& a, int grid, cudaStream_t st) {
    if (grid < 1) grid = 1;
    count_launches(1);
    pbm_expand_kernel<<<grid, kExpandThreads, 0, st>>>(a);
    return cudaGetLastError();
}

__global__ void pbm_collect_kernel(const uint64_t* __restrict__ pool,
                                   const unsigned long long* from, uint64_t hi, uint64_t* out,
                                   uint64_t cap, PbmCounters* ctr) {
    const unsigned long long lo = ctr->kmax;
    const unsigned long long f = from ? *from : 0ull;
    const int64_t n = (int64_t)ctr->pool_len;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int lane = threadIdx.x & 31;
    // whole warps iterate together so that the appends can be aggregated
    for (int64_t i0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); i0 < n;
         i0 += stride) {
        const int64_t i = i0 + lane;
        uint64_t k = 0;
        bool take = false;
        if (i < n) {
            k = pool[i];
            take = k > lo && k < hi && k >= f;
        }
        const unsigned int m = __ballot_sync(0xffffffffu, take);
        if (m == 0) continue;
        unsigned long long base = 0;
        if (lane == 0) base = atomicAdd(&ctr->collected, (unsigned long long)__popc(m));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (take) {
            const unsigned long long pos = base + __popc(m & ((1u << lane) - 1u));
            if (pos < cap) out[pos] = k;
        }
    }
}

cudaError_t launch_pbm_collect(const uint64_t* pool, const unsigned long long* from, uint64_t hi,
                               uint64_t* out, uint64_t cap, PbmCounters* ctr, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(&ctr->collected, 0, sizeof(unsigned long long), st);
    if (e != cudaSuccess) return e;
    count_launches(1);
    pbm_collect_kernel<<<152 * 4, 256, 0, st>>>(pool, from, hi, out, cap, ctr);
    return cudaGetLastError();
}

// 64-bit radix selection of the k-th largest key in (kmax, hi): one digit of
// 8 bits per round, most significant first.  sel[0] = decided prefix,
// sel[1] = remaining rank, sel[2 ..] = histogram.
__global__ void pbm_sel_init_kernel(unsigned long long* sel, unsigned long long k) {
    for (int i = threadIdx.x; i < 258; i += blockDim.x) sel[i] = 0;
    if (threadIdx.x == 0) sel[1] = k;
}

__global__ void pbm_sel_hist_kernel(const uint64_t* __restrict__ pool, const PbmCounters* ctr,
                                    uint64_t hi, int shift, unsigned long long* sel) {
    __shared__ unsigned int h[256];
    for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = 0;
    __syncthreads();
    const unsigned long long lo = ctr->kmax;
    const int64_t n = (int64_t)ctr->pool_len;
    const unsigned long long prefix = sel[0];
    const int up = shift + 8;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const uint64_t k = pool[i];
        if (!(k > lo && k < hi)) continue;
        if (up < 64 && (k >> up) != (prefix >> up)) continue;
        atomicAdd(&h[(k >> shift) & 0xffu], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += blockDim.x)
        if (h[i]) atomicAdd(&sel[2 + i], (unsigned long long)h[i]);
}

__global__ void pbm_sel_pick_kernel(int shift, unsigned long long* sel) {
    if (threadIdx.x != 0) return;
    unsigned long long k = sel[1], cum = 0;
    for (int d = 255; d >= 0; --d) {
        const unsigned long long c = sel[2 + d];
        if (cum + c >= k) {
            sel[0] |= (unsigned long long)d << shift;
            sel[1] = k - cum;
            break;
        }
        cum += c;
    }
    for (int i = 0; i < 256; ++i) sel[2 + i] = 0;
}

cudaError_t launch_pbm_select64(const uint64_t* pool, const PbmCounters* ctr, uint64_t hi,
                                uint64_t k, unsigned long long* sel64, cudaStream_t st) {
    count_launches(1);
    pbm_sel_init_kernel<<<1, 256, 0, st>>>(sel64, (unsigned long long)k);
    for (int shift = 56; shift >= 0; shift -= 8) {
        count_launches(2);
        pbm_sel_hist_kernel<<<152 * 4, 256, 0, st>>>(pool, ctr, hi, shift, sel64);
        pbm_sel_pick_kernel<<<1, 32, 0, st>>>(shift, sel64);
    }
    return cudaGetLastError();
}

__global__ void pbm_emit_kernel(const uint64_t* __restrict__ keys, int m, int64_t* ids,
                                float* scores) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= m) return;
    const uint64_t k = keys[i];
    ids[i] = (int64_t)rank_key_id(k);
    scores[i] = rank_key_score(k);
}

cudaError_t launch_pbm_emit(const uint64_t* keys, int m, int64_t* ids, float* scores,
                            cudaStream_t st) {
    if (m <= 0) return cudaSuccess;
    count_launches(1);
    pbm_emit_kernel<<<(m + 255) / 256, 256, 0, st>>>(keys, m, ids, scores);
    return cudaGetLastError();
}

// One term's postings; a term lists an item at most once, so no two threads
// of a launch touch one accumulator, and launches in term order keep each
// item's additions in the query's order (App. A.2).
__global__ void pbm_score_term_kernel(const int64_t* __restrict__ term_off,
                                      const int32_t* __restrict__ docs,
                                      const float* __restrict__ imps, const int32_t* terms,
                                      const float* weights, int j, float* acc) {
    const int32_t t = terms[j];
    const float w = weights[j];
    const int64_t b = term_off[t], e = term_off[t + 1];
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = b + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < e; i += stride) {
        const int32_t x = docs[i];
        acc[x] = __fadd_rn(acc[x], __fmul_rn(w, imps[i]));
    }
}

cudaError_t launch_pbm_score_all(const PbmQuery& q, const int64_t* term_off, const int32_t* docs,
                                 const float* imps, float* acc, int grid, cudaStream_t st) {
    for (int j = 0; j < q.nq; ++j) {
        count_launches(1);
        pbm_score_term_kernel<<<grid, 256, 0, st>>>(term_off, docs, imps, q.terms, q.weights, j,
                                                    acc);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

__global__ void pbm_member_keys_kernel(const float* __restrict__ acc, int64_t n,
                                       const uint32_t* __restrict__ tomb, uint64_t* keys,
                                       unsigned long long* count) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < n; x += stride) {
        const float s = acc[x];
        if (s > 0.0f && !tombstoned(tomb, x))
            keys[atomicAdd(count, 1ull)] = rank_key(s, (uint32_t)x);
    }
}

cudaError_t launch_pbm_member_keys(const float* acc, int64_t n, const uint32_t* tomb,
                                   uint64_t* keys, unsigned long long* count, int grid,
                                   cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    count_launches(1);
    pbm_member_keys_kernel<<<grid, 256, 0, st>>>(acc, n, tomb, keys, count);
    return cudaGetLastError();
}

__global__ void pbm_rank_of_kernel(const uint64_t* __restrict__ keys, int64_t m, int32_t* rank_of) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < m; i += stride)
        rank_of[rank_key_id(keys[i])] = (int32_t)(i + 1);
}

cudaError_t launch_pbm_rank_of(const uint64_t* keys, int64_t m, int32_t* rank_of, int grid,
                               cudaStream_t st) {
    if (m <= 0) return cudaSuccess;
    count_launches(1);
    pbm_rank_of_kernel<<<grid, 256, 0, st>>>(keys, m, rank_of);
    return cudaGetLastError();
}

}  // namespace pvs
