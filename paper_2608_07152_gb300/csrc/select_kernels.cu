// Selection, compaction, sorting and emission for PVS certification
// (Sec. 2.3.1: candidates are taken in decreasing interval upper bound;
// Sec. 2.1: ranks are ordered by score, ties by ascending id).
//
//  * radix select over ordered 32-bit float keys (8-bit digits, MSB first):
//    histogram kernels with shared-memory counters, a one-block digit pick;
//  * ordered compaction (block counts -> scan -> in-order scatter) for the
//    working set, so its index order is the id order;
//  * candidate compaction with warp-aggregated atomics;
//  * single-CTA bitonic sort of up to 8192 64-bit rank keys in shared memory;
//  * LSD radix sort of 64-bit rank keys for large pulls (8 passes: block
//    histograms, one-block scan, stable scatter ranked with match.any).
#include "kernels.h"
#include "pvs_common.cuh"

namespace pvs {

// ---------------------------------------------------------------------------
// radix select on float keys
// ---------------------------------------------------------------------------
__global__ void select_hist_kernel(const float* __restrict__ vals, const unsigned int* len_dev,
                                   int64_t len_host, SelectState* sel, int shift) {
    __shared__ unsigned int h[256];
    for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = 0;
    __syncthreads();
    const int64_t len = len_dev ? (int64_t)*len_dev : len_host;
    const uint32_t prefix = (uint32_t)sel->prefix;
    const uint32_t hmask = shift >= 24 ? 0u : (0xffffffffu << (shift + 8));
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < len; i += stride) {
        const float v = vals[i];
        if (v == -INFINITY) continue;
        const uint32_t key = fkey(v);
        if ((key & hmask) != (prefix & hmask)) continue;
        atomicAdd(&h[(key >> shift) & 0xffu], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += blockDim.x)
        if (h[i]) atomicAdd(&sel->hist[i], h[i]);
}

// One block of 256 threads: choose the digit holding the k-th largest key.
__global__ void select_pick_kernel(SelectState* sel, int shift) {
    __shared__ unsigned long long suffix[256];
    const int t = threadIdx.x;
    // suffix[t] = count of keys with digit >= t (inclusive suffix sum)
    suffix[t] = sel->hist[255 - t];
    __syncthreads();
    for (int o = 1; o < 256; o <<= 1) {
        unsigned long long v = t >= o ? suffix[t - o] : 0ull;
        __syncthreads();
        suffix[t] += v;
        __syncthreads();
    }
    // suffix[t] now counts digits 255-t .. 255
    const uint64_t k = sel->k;
    const int d = 255 - t;
    const unsigned long long above = t > 0 ? suffix[t - 1] : 0ull;
    const unsigned long long upto = suffix[t];
    __syncthreads();
    if (above < k && k <= upto) {
        sel->prefix |= ((uint64_t)d << shift);
        sel->k = k - above;
    }
    __syncthreads();
    sel->hist[t] = 0;
}

__global__ void select_init_kernel(SelectState* sel, uint64_t k) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) sel->hist[i] = 0;
    if (threadIdx.x == 0) {
        sel->prefix = 0;
        sel->k = k;
    }
}

static cudaError_t select_f32(const float* vals, const unsigned int* len_dev, int64_t len_host,
                              uint64_t k, SelectState* sel, int grid, cudaStream_t st) {
    count_launches(1);
    select_init_kernel<<<1, 256, 0, st>>>(sel, k);
    for (int shift = 24; shift >= 0; shift -= 8) {
        count_launches(1);
        select_hist_kernel<<<grid, 256, 0, st>>>(vals, len_dev, len_host, sel, shift);
        count_launches(1);
        select_pick_kernel<<<1, 256, 0, st>>>(sel, shift);
    }
    return cudaGetLastError();
}

cudaError_t launch_select_f32(const float* vals, const unsigned int* len, uint64_t k,
                              SelectState* sel, int grid, cudaStream_t st) {
    return select_f32(vals, len, 0, k, sel, grid, st);
}

cudaError_t launch_select_f32_n(const float* vals, int64_t rows, uint64_t k, SelectState* sel,
                                int grid, cudaStream_t st) {
    return select_f32(vals, nullptr, rows, k, sel, grid, st);
}

// The same selection for a short array in one launch: one CTA copies the
// values into shared memory once (16-byte loads; when they fit) and runs the
// four digit rounds there, its histogram in shared memory too.
__device__ __forceinline__ void select_small_body(const float* __restrict__ vals, int64_t len,
                                                  uint64_t k0, SelectState* sel, int staged) {
    extern __shared__ float4 staged_vals[];
    __shared__ unsigned int h[256];
    __shared__ unsigned int suffix[256];
    __shared__ uint32_t prefix;
    __shared__ unsigned long long k;
    const int t = threadIdx.x;
    if (t == 0) {
        prefix = 0;
        k = k0;
    }
    const float* src = vals;
    if (staged) {
        const int64_t n4 = len / 4;
        const float4* v4 = reinterpret_cast<const float4*>(vals);
        for (int64_t i = t; i < n4; i += blockDim.x) staged_vals[i] = v4[i];
        float* sf = reinterpret_cast<float*>(staged_vals);
        for (int64_t i = n4 * 4 + t; i < len; i += blockDim.x) sf[i] = vals[i];
        src = sf;
    }
    for (int shift = 24; shift >= 0; shift -= 8) {
        if (t < 256) h[t] = 0;
        __syncthreads();
        const uint32_t hmask = shift >= 24 ? 0u : (0xffffffffu << (shift + 8));
        const uint32_t pre = prefix;
        // close scores share their high digits: each thread counts a run of
        // one digit in a register and adds it when the digit changes
        uint32_t run_d = 256u;
        unsigned int run_n = 0;
        for (int64_t i = t; i < len; i += blockDim.x) {
            const float v = src[i];
            if (v == -INFINITY) continue;
            const uint32_t key = fkey(v);
            if ((key & hmask) != (pre & hmask)) continue;
            const uint32_t d = (key >> shift) & 0xffu;
            if (d != run_d) {
                if (run_n) atomicAdd(&h[run_d], run_n);
                run_d = d;
                run_n = 0;
            }
            ++run_n;
        }
        if (run_n) atomicAdd(&h[run_d], run_n);
        __syncthreads();
        // suffix[u] = keys whose digit is 255 - u or above
        if (t < 256) suffix[t] = h[255 - t];
        __syncthreads();
        for (int o = 1; o < 256; o <<= 1) {
            unsigned int v = (t < 256 && t >= o) ? suffix[t - o] : 0u;
            __syncthreads();
            if (t < 256) suffix[t] += v;
            __syncthreads();
        }
        // every thread reads k before the one thread holding the digit
        // (exactly one: keys are counted once) rewrites it
        const unsigned long long kk = k;
        const unsigned long long above = (t < 256 && t > 0) ? suffix[t - 1] : 0u;
        const bool mine = t < 256 && above < kk && kk <= (unsigned long long)suffix[t];
        __syncthreads();
        if (mine) {
            prefix = pre | ((uint32_t)(255 - t) << shift);
            k = kk - above;
        }
        __syncthreads();
    }
    if (t == 0) {
        sel->prefix = prefix;
        sel->k = k;
    }
    if (t < 256) sel->hist[t] = 0;
}

__global__ void __launch_bounds__(1024) select_small_kernel(const float* __restrict__ vals,
                                                            int64_t len, uint64_t k0,
                                                            SelectState* sel, int staged) {
    select_small_body(vals, len, k0, sel, staged);
}

cudaError_t launch_select_small(const float* vals, int64_t len, uint64_t k, SelectState* sel,
                                cudaStream_t st) {
    // staged in shared memory when the values fit in 200 KB and start on a
    // 16-byte boundary (device allocations do)
    const bool staged = len > 0 && len * (int64_t)sizeof(float) <= 200 * 1024 &&
                        (reinterpret_cast<uintptr_t>(vals) & 15u) == 0;
    const size_t smem = staged ? (size_t)((len + 3) / 4) * sizeof(float4) : 0;
    if (smem > 0) {
        cudaError_t e = raise_smem_limit((const void*)select_small_kernel, smem);
        if (e != cudaSuccess) return e;
    }
    count_launches(1);
    select_small_kernel<<<1, 1024, smem, st>>>(vals, len, k, sel, staged ? 1 : 0);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// ordered compaction of the working set: {i : lo[i] live, key(hi[i]) >= tau}
// ---------------------------------------------------------------------------
constexpr int kCompactBlock = 256;
constexpr int kCompactItems = 16;
constexpr int kCompactTile = kCompactBlock * kCompactItems;

size_t compact_scratch_elems(int64_t rows) {
    return (size_t)((rows + kCompactTile - 1) / kCompactTile) + 1;
}

// A row leaves (emitted, tombstoned) with lo = hi = -inf, and refinement
// sets lo = hi = its score: lo is -inf exactly when hi is.  So a threshold
// that is the key of a finite bound (tau != 0) is reached only by live rows
// and needs hi alone; tau = 0 (every live row) reads lo.
__device__ __forceinline__ bool ws_member(const float* lo, const float* hi, int64_t i,
                                          uint32_t tau) {
    if (tau != 0u) return fkey(hi[i]) >= tau;
    return lo[i] != -INFINITY;
}

__device__ __forceinline__ void compact_count_body(const float* __restrict__ lo,
                                                   const float* __restrict__ hi, int64_t rows,
                                                   const SelectState* sel,
                                                   unsigned int* block_counts) {
    __shared__ unsigned int wsum[kCompactBlock / 32];
    const uint32_t tau = (uint32_t)sel->prefix;
    const int64_t base = (int64_t)blockIdx.x * kCompactTile;
    unsigned int c = 0;
    for (int j = 0; j < kCompactItems; ++j) {
        const int64_t i = base + (int64_t)j * kCompactBlock + threadIdx.x;
        if (i < rows && ws_member(lo, hi, i, tau)) ++c;
    }
    c = warp_sum(c);
    if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = c;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned int s = 0;
        for (int w = 0; w < kCompactBlock / 32; ++w) s += wsum[w];
        block_counts[blockIdx.x] = s;
    }
}

__global__ void compact_count_kernel(const float* __restrict__ lo, const float* __restrict__ hi,
                                     int64_t rows, const SelectState* sel,
                                     unsigned int* block_counts) {
    compact_count_body(lo, hi, rows, sel, block_counts);
}

// Exclusive scan of n block counts by one block; total to *total.
__device__ __forceinline__ void scan_counts_body(unsigned int* counts, int64_t n,
                                                 unsigned int* total) {
    __shared__ unsigned int part[1024];
    const int t = threadIdx.x;
    const int64_t per = (n + blockDim.x - 1) / blockDim.x;
    const int64_t b0 = t * per, b1 = (b0 + per < n) ? b0 + per : n;
    unsigned int s = 0;
    for (int64_t i = b0; i < b1; ++i) s += counts[i];
    part[t] = s;
    __syncthreads();
    for (int o = 1; o < (int)blockDim.x; o <<= 1) {
        unsigned int v = t >= o ? part[t - o] : 0u;
        __syncthreads();
        part[t] += v;
        __syncthreads();
    }
    unsigned int run = t > 0 ? part[t - 1] : 0u;
    for (int64_t i = b0; i < b1; ++i) {
        unsigned int c = counts[i];
        counts[i] = run;
        run += c;
    }
    if (t == (int)blockDim.x - 1) *total = part[t];
}

__global__ void scan_counts_kernel(unsigned int* counts, int64_t n, unsigned int* total) {
    scan_counts_body(counts, n, total);
}

__device__ __forceinline__ void compact_scatter_body(const float* __restrict__ lo,
                                                     const float* __restrict__ hi, int64_t rows,
                                                     const SelectState* sel,
                                                     const unsigned int* block_offsets,
                                                     int32_t* w_id, float* w_lo, float* w_hi) {
    __shared__ unsigned int wbase[kCompactBlock / 32];
    __shared__ unsigned int run;
    const uint32_t tau = (uint32_t)sel->prefix;
    const int64_t base = (int64_t)blockIdx.x * kCompactTile;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) run = block_offsets[blockIdx.x];
    __syncthreads();
    for (int j = 0; j < kCompactItems; ++j) {
        const int64_t i = base + (int64_t)j * kCompactBlock + threadIdx.x;
        const bool f = i < rows && ws_member(lo, hi, i, tau);
        const unsigned int bal = __ballot_sync(0xffffffffu, f);
        if (lane == 0) wbase[warp] = __popc(bal);
        __syncthreads();
        unsigned int before = 0, total = 0;
        for (int w = 0; w < kCompactBlock / 32; ++w) {
            const unsigned int c = wbase[w];
            if (w < warp) before += c;
            total += c;
        }
        if (f) {
            const unsigned int pos = run + before + __popc(bal & ((1u << lane) - 1u));
            w_id[pos] = (int32_t)i;
            w_lo[pos] = lo[i];
            w_hi[pos] = hi[i];
        }
        __syncthreads();
        if (threadIdx.x == 0) run += total;
        __syncthreads();
    }
}

__global__ void compact_scatter_kernel(const float* __restrict__ lo, const float* __restrict__ hi,
                                       int64_t rows, const SelectState* sel,
                                       const unsigned int* block_offsets, int32_t* w_id,
                                       float* w_lo, float* w_hi) {
    compact_scatter_body(lo, hi, rows, sel, block_offsets, w_id, w_lo, w_hi);
}

cudaError_t launch_compact_ordered(const float* lo, const float* hi, int64_t rows,
                                   const SelectState* sel, int32_t* w_id, float* w_lo,
                                   float* w_hi, unsigned int* w_len, unsigned int* scratch,
                                   cudaStream_t st) {
    const int64_t nb = (rows + kCompactTile - 1) / kCompactTile;
    if (nb == 0) return cudaMemsetAsync(w_len, 0, sizeof(unsigned int), st);
    count_launches(1);
    compact_count_kernel<<<(unsigned)nb, kCompactBlock, 0, st>>>(lo, hi, rows, sel, scratch);
    count_launches(1);
    scan_counts_kernel<<<1, 1024, 0, st>>>(scratch, nb, w_len);
    count_launches(1);
    compact_scatter_kernel<<<(unsigned)nb, kCompactBlock, 0, st>>>(lo, hi, rows, sel, scratch,
                                                                   w_id, w_lo, w_hi);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// the same steps for the cursors of a grouped pass, one launch per step
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) select_small_group_kernel(const __grid_constant__ WsGroupArgs a,
                                                                  int staged) {
    const int g = blockIdx.y;
    select_small_body(a.slot[g], a.slot_n, a.k[g], a.sel[g], staged);
}

__global__ void compact_count_group_kernel(const __grid_constant__ WsGroupArgs a) {
    const int g = blockIdx.y;
    compact_count_body(a.lo[g], a.hi[g], a.rows, a.sel[g], a.scratch[g]);
}

__global__ void scan_counts_group_kernel(const __grid_constant__ WsGroupArgs a, int64_t nb) {
    const int g = blockIdx.x;
    scan_counts_body(a.scratch[g], nb, a.w_len[g]);
}

__global__ void compact_scatter_group_kernel(const __grid_constant__ WsGroupArgs a) {
    const int g = blockIdx.y;
    compact_scatter_body(a.lo[g], a.hi[g], a.rows, a.sel[g], a.scratch[g], a.w_id[g], a.w_lo[g],
                         a.w_hi[g]);
}

// The same count and ordered scatter from the 16-row block maxima of hi: a
// thread takes one block of 16 rows (a CTA the same 4,096 rows as above, so
// the block counts and their scan are shared), and reads its rows only when
// the block's maximum reaches the threshold (for tau = 0, every live row:
// when the block holds one).
__device__ __forceinline__ bool bmax_reaches(const float* bmax, int64_t b, uint32_t tau) {
    const float m = bmax[b];
    return tau != 0u ? fkey(m) >= tau : m != -INFINITY;
}

__device__ __forceinline__ unsigned int bmax_block_members(const float* lo, const float* hi,
                                                           int64_t r0, int64_t rows,
                                                           uint32_t tau) {
    unsigned int c = 0;
    const int64_t r1 = r0 + kBmaxRows < rows ? r0 + kBmaxRows : rows;
    for (int64_t i = r0; i < r1; ++i) c += ws_member(lo, hi, i, tau) ? 1u : 0u;
    return c;
}

__global__ void compact_count_bmax_group_kernel(const __grid_constant__ WsGroupArgs a) {
    __shared__ unsigned int wsum[kCompactBlock / 32];
    const int g = blockIdx.y;
    const uint32_t tau = (uint32_t)a.sel[g]->prefix;
    const int64_t b = (int64_t)blockIdx.x * kCompactBlock + threadIdx.x;
    const int64_t r0 = b * kBmaxRows;
    unsigned int c = 0;
    if (r0 < a.rows && bmax_reaches(a.bmax[g], b, tau))
        c = bmax_block_members(a.lo[g], a.hi[g], r0, a.rows, tau);
    c = warp_sum(c);
    if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = c;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned int s = 0;
        for (int w = 0; w < kCompactBlock / 32; ++w) s += wsum[w];
        a.scratch[g][blockIdx.x] = s;
    }
}

__global__ void compact_scatter_bmax_group_kernel(const __grid_constant__ WsGroupArgs a) {
    __shared__ unsigned int wtot[kCompactBlock / 32];
    const int g = blockIdx.y;
    const uint32_t tau = (uint32_t)a.sel[g]->prefix;
    const float* lo = a.lo[g];
    const float* hi = a.hi[g];
    const int64_t b = (int64_t)blockIdx.x * kCompactBlock + threadIdx.x;
    const int64_t r0 = b * kBmaxRows;
    const bool live = r0 < a.rows && bmax_reaches(a.bmax[g], b, tau);
    const unsigned int c = live ? bmax_block_members(lo, hi, r0, a.rows, tau) : 0u;
    // exclusive prefix of c over the CTA, in thread (= row) order
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    unsigned int inc = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned int v = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += v;
    }
    if (lane == 31) wtot[warp] = inc;
    __syncthreads();
    unsigned int pos = a.scratch[g][blockIdx.x] + inc - c;
    for (int w = 0; w < warp; ++w) pos += wtot[w];
    if (c == 0) return;
    const int64_t r1 = r0 + kBmaxRows < a.rows ? r0 + kBmaxRows : a.rows;
    for (int64_t i = r0; i < r1; ++i) {
        if (!ws_member(lo, hi, i, tau)) continue;
        a.w_id[g][pos] = (int32_t)i;
        a.w_lo[g][pos] = lo[i];
        a.w_hi[g][pos] = hi[i];
        ++pos;
    }
}

cudaError_t launch_ws_group(const WsGroupArgs& a, cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    if (a.n > kGroupMax || a.slot_n <= 0) return cudaErrorInvalidValue;
    bool staged = a.slot_n * (int64_t)sizeof(float) <= 200 * 1024;
    for (int g = 0; g < a.n; ++g)
        staged = staged && (reinterpret_cast<uintptr_t>(a.slot[g]) & 15u) == 0;
    const size_t smem = staged ? (size_t)((a.slot_n + 3) / 4) * sizeof(float4) : 0;
    if (smem > 0) {
        cudaError_t e = raise_smem_limit((const void*)select_small_group_kernel, smem);
        if (e != cudaSuccess) return e;
    }
    count_launches(1);
    select_small_group_kernel<<<dim3(1, a.n), 1024, smem, st>>>(a, staged ? 1 : 0);
    const int64_t nb = (a.rows + kCompactTile - 1) / kCompactTile;
    if (nb == 0) {
        for (int g = 0; g < a.n; ++g) {
            cudaError_t e = cudaMemsetAsync(a.w_len[g], 0, sizeof(unsigned int), st);
            if (e != cudaSuccess) return e;
        }
        return cudaGetLastError();
    }
    bool by_blocks = true;
    for (int g = 0; g < a.n; ++g) by_blocks = by_blocks && a.bmax[g] != nullptr;
    count_launches(3);
    if (by_blocks) {
        compact_count_bmax_group_kernel<<<dim3((unsigned)nb, a.n), kCompactBlock, 0, st>>>(a);
        scan_counts_group_kernel<<<a.n, 1024, 0, st>>>(a, nb);
        compact_scatter_bmax_group_kernel<<<dim3((unsigned)nb, a.n), kCompactBlock, 0, st>>>(a);
    } else {
        compact_count_group_kernel<<<dim3((unsigned)nb, a.n), kCompactBlock, 0, st>>>(a);
        scan_counts_group_kernel<<<a.n, 1024, 0, st>>>(a, nb);
        compact_scatter_group_kernel<<<dim3((unsigned)nb, a.n), kCompactBlock, 0, st>>>(a);
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// candidates of a pull
// ---------------------------------------------------------------------------
__global__ void candidates_kernel(const float* __restrict__ w_lo, const float* __restrict__ w_hi,
                                  const unsigned int* w_len, const SelectState* sel,
                                  int32_t* cand, unsigned int* cand_len) {
    const uint32_t tau = (uint32_t)sel->prefix;
    const int64_t len = *w_len;
    const int lane = threadIdx.x & 31;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i0 = (int64_t)blockIdx.x * blockDim.x; i0 < len; i0 += stride) {
        const int64_t i = i0 + threadIdx.x;
        const bool f = i < len && w_lo[i] != -INFINITY && fkey(w_hi[i]) >= tau;
        const unsigned int bal = __ballot_sync(0xffffffffu, f);
        unsigned int base = 0;
        if (lane == 0 && bal) base = atomicAdd(cand_len, (unsigned int)__popc(bal));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (f) cand[base + __popc(bal & ((1u << lane) - 1u))] = (int32_t)i;
    }
}

cudaError_t launch_candidates(const float* w_lo, const float* w_hi, const unsigned int* w_len,
                              const SelectState* sel, int32_t* cand, unsigned int* cand_len,
                              int grid, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(cand_len, 0, sizeof(unsigned int), st);
    if (e != cudaSuccess) return e;
    count_launches(1);
    candidates_kernel<<<grid, 256, 0, st>>>(w_lo, w_hi, w_len, sel, cand, cand_len);
    return cudaGetLastError();
}

__global__ void make_keys_kernel(const int32_t* __restrict__ cand, const unsigned int* cand_len,
                                 const float* __restrict__ w_lo, uint64_t* keys) {
    const int64_t n = *cand_len;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const int32_t w = cand[i];
        keys[i] = rank_key(w_lo[w], (uint32_t)w);
    }
}

cudaError_t launch_make_keys(const int32_t* cand, const unsigned int* cand_len,
                             const float* w_lo, uint64_t* keys, int grid, cudaStream_t st) {
    count_launches(1);
    make_keys_kernel<<<grid, 256, 0, st>>>(cand, cand_len, w_lo, keys);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// single-CTA bitonic sort, descending
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) bitonic_desc_kernel(uint64_t* keys, int count, int pow2) {
    extern __shared__ uint64_t sk[];
    for (int i = threadIdx.x; i < pow2; i += blockDim.x) sk[i] = i < count ? keys[i] : 0ull;
    __syncthreads();
    for (int size = 2; size <= pow2; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = threadIdx.x; i < pow2 / 2; i += blockDim.x) {
                const int lo = 2 * i - (i & (stride - 1));
                const int hi = lo + stride;
                const bool desc = (lo & size) == 0;
                const uint64_t a = sk[lo], b = sk[hi];
                if ((a < b) == desc) {
                    sk[lo] = b;
                    sk[hi] = a;
                }
            }
            __syncthreads();
        }
    }
    for (int i = threadIdx.x; i < count; i += blockDim.x) keys[i] = sk[i];
}

// The same network for at most 1024 E keys with E per thread in registers
// (thread t holds positions tE .. tE + E - 1): a stride below E is a swap
// within a thread, below 32 E a shuffle within a warp, and only the larger
// strides go through shared memory (15 of the 78 stages at 4,096 keys).
template <int E>
__device__ __forceinline__ void bitonic_keep(uint64_t& v, uint64_t w, int i, int j, int size) {
    const bool desc = (i & size) == 0;
    const bool keep_max = (i < j) == desc;
    v = keep_max ? (v > w ? v : w) : (v < w ? v : w);
}

template <int E>
__global__ void __launch_bounds__(1024) bitonic_desc_reg_kernel(uint64_t* keys, int count) {
    __shared__ uint64_t sk[1024 * E];
    const int t = threadIdx.x;
    constexpr int n = 1024 * E;
    uint64_t v[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int i = t * E + e;
        v[e] = i < count ? keys[i] : 0ull;
    }
    for (int size = 2; size <= n; size <<= 1) {
        for (int s = size >> 1; s > 0; s >>= 1) {
            if (s >= 32 * E) {   // another warp's element
#pragma unroll
                for (int e = 0; e < E; ++e) sk[t * E + e] = v[e];
                __syncthreads();
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    const int i = t * E + e;
                    bitonic_keep<E>(v[e], sk[i ^ s], i, i ^ s, size);
                }
                __syncthreads();
            } else if (s >= E) {   // another lane's element
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    const int i = t * E + e;
                    const uint64_t w = __shfl_xor_sync(0xffffffffu, v[e], s / E);
                    bitonic_keep<E>(v[e], w, i, i ^ s, size);
                }
            } else {   // this thread's element: s is 1 or 2 (E = 2 or 4)
                auto ex = [&](uint64_t& a, uint64_t& b, int e) {
                    const bool desc = ((t * E + e) & size) == 0;
                    const bool swap = (a < b) == desc;
                    const uint64_t x = a;
                    a = swap ? b : a;
                    b = swap ? x : b;
                };
                if (E >= 2 && s == 1) {
                    ex(v[0], v[E >= 2 ? 1 : 0], 0);
                    if (E == 4) ex(v[E == 4 ? 2 : 0], v[E == 4 ? 3 : 0], 2);
                } else if (E == 4 && s == 2) {
                    ex(v[0], v[E == 4 ? 2 : 0], 0);
                    ex(v[E == 4 ? 1 : 0], v[E == 4 ? 3 : 0], 1);
                }
            }
        }
    }
#pragma unroll
    for (int e = 0; e < E; ++e) {
        const int i = t * E + e;
        if (i < count) keys[i] = v[e];
    }
}

cudaError_t launch_bitonic_desc(uint64_t* keys, int count, cudaStream_t st) {
    if (count <= 1) return cudaSuccess;
    if (count <= 4096) {
        count_launches(1);
        if (count <= 1024)
            bitonic_desc_reg_kernel<1><<<1, 1024, 0, st>>>(keys, count);
        else if (count <= 2048)
            bitonic_desc_reg_kernel<2><<<1, 1024, 0, st>>>(keys, count);
        else
            bitonic_desc_reg_kernel<4><<<1, 1024, 0, st>>>(keys, count);
        return cudaGetLastError();
    }
    int pow2 = 2;
    while (pow2 < count) pow2 <<= 1;
    const size_t smem = (size_t)pow2 * sizeof(uint64_t);
    cudaError_t e = raise_smem_limit((const void*)bitonic_desc_kernel, smem);
    if (e != cudaSuccess) return e;
    count_launches(1);
    bitonic_desc_kernel<<<1, 1024, smem, st>>>(keys, count, pow2);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// LSD radix sort of 64-bit keys, descending (digit = 255 - byte)
// ---------------------------------------------------------------------------
constexpr int kSortBlock = 256;
constexpr int kSortRounds = 16;
constexpr int kSortTile = kSortBlock * kSortRounds;

size_t radix_sort_scratch_bytes(int64_t count) {
    const int64_t nb = (count + kSortTile - 1) / kSortTile;
    return (size_t)(256 * nb + 1 + 256) * sizeof(unsigned int);   // counts, total, digit sums
}

// Exclusive scan of the digit-major block counts (count[d nb + b]) in two
// parallel steps: each digit's total, then one CTA per digit adds the totals
// of the digits before it and scans its nb counts.  (One CTA scanning all
// 256 nb counts took ~94 us per pass at 8.8M keys.)
__global__ void __launch_bounds__(256) digit_sum_kernel(const unsigned int* __restrict__ counts,
                                                        int64_t nb, unsigned int* digit_total) {
    __shared__ unsigned int ws[8];
    const unsigned int* c = counts + (int64_t)blockIdx.x * nb;
    unsigned int s = 0;
    for (int64_t i = threadIdx.x; i < nb; i += blockDim.x) s += c[i];
    s = warp_sum(s);
    if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned int t = 0;
        for (int w = 0; w < 8; ++w) t += ws[w];
        digit_total[blockIdx.x] = t;
    }
}

__global__ void __launch_bounds__(1024) digit_scan_kernel(unsigned int* counts, int64_t nb,
                                                          const unsigned int* digit_total,
                                                          unsigned int* total) {
    __shared__ unsigned int part[1024];
    __shared__ unsigned int base_sh;
    const int t = threadIdx.x;
    const int d = blockIdx.x;
    if (t < 32) {   // the totals of the digits before d
        unsigned int b = 0;
        for (int i = t; i < d; i += 32) b += digit_total[i];
        b = warp_sum(b);
        if (t == 0) base_sh = b;
    }
    unsigned int* c = counts + (int64_t)d * nb;
    const int64_t per = (nb + blockDim.x - 1) / blockDim.x;
    const int64_t b0 = t * per, b1 = (b0 + per < nb) ? b0 + per : nb;
    unsigned int s = 0;
    for (int64_t i = b0; i < b1; ++i) s += c[i];
    part[t] = s;
    __syncthreads();
    for (int o = 1; o < (int)blockDim.x; o <<= 1) {
        const unsigned int v = t >= o ? part[t - o] : 0u;
        __syncthreads();
        part[t] += v;
        __syncthreads();
    }
    unsigned int run = base_sh + (t > 0 ? part[t - 1] : 0u);
    for (int64_t i = b0; i < b1; ++i) {
        const unsigned int x = c[i];
        c[i] = run;
        run += x;
    }
    if (d == 255 && t == (int)blockDim.x - 1) *total = base_sh + part[t];
}

__device__ __forceinline__ int sort_digit(uint64_t k, int shift) {
    return 255 - (int)((k >> shift) & 0xffu);
}

__global__ void sort_upsweep_kernel(const uint64_t* __restrict__ keys, int64_t count, int shift,
                                    unsigned int* block_hist, int64_t nb) {
    __shared__ unsigned int h[256];
    h[threadIdx.x] = 0;
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * kSortTile;
    for (int r = 0; r < kSortRounds; ++r) {
        const int64_t i = base + (int64_t)r * kSortBlock + threadIdx.x;
        if (i < count) atomicAdd(&h[sort_digit(keys[i], shift)], 1u);
    }
    __syncthreads();
    block_hist[(int64_t)threadIdx.x * nb + blockIdx.x] = h[threadIdx.x];
}

__global__ void sort_downsweep_kernel(const uint64_t* __restrict__ keys, uint64_t* out,
                                      int64_t count, int shift, const unsigned int* block_off,
                                      int64_t nb) {
    constexpr int W = kSortBlock / 32;
    __shared__ unsigned int warp_cnt[W][256];
    __shared__ unsigned int warp_off[W][256];
    __shared__ unsigned int run[256];
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    run[t] = block_off[(int64_t)t * nb + blockIdx.x];
    for (int w = 0; w < W; ++w) warp_cnt[w][t] = 0;
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * kSortTile;
    for (int r = 0; r < kSortRounds; ++r) {
        const int64_t i = base + (int64_t)r * kSortBlock + t;
        const bool valid = i < count;
        const uint64_t k = valid ? keys[i] : 0ull;
        const int d = valid ? sort_digit(k, shift) : 256 + lane;  // unique dummy digit
        const unsigned int peers = __match_any_sync(0xffffffffu, d);
        const int rank = __popc(peers & ((1u << lane) - 1u));
        const int leader = __ffs(peers) - 1;
        if (valid && lane == leader) warp_cnt[warp][d] = __popc(peers);
        __syncthreads();
        {
            unsigned int acc = run[t];
            for (int w = 0; w < W; ++w) {
                const unsigned int c = warp_cnt[w][t];
                warp_off[w][t] = acc;
                acc += c;
                warp_cnt[w][t] = 0;
            }
            run[t] = acc;
        }
        __syncthreads();
        if (valid) out[warp_off[warp][d] + rank] = k;
        __syncthreads();
    }
}

cudaError_t launch_radix_sort_desc(uint64_t* keys, uint64_t* tmp, int64_t count, void* scratch,
                                   cudaStream_t st) {
    if (count <= 1) return cudaSuccess;
    const int64_t nb = (count + kSortTile - 1) / kSortTile;
    unsigned int* hist = static_cast<unsigned int*>(scratch);
    unsigned int* total = hist + 256 * nb;
    unsigned int* digit_total = total + 1;
    const bool wide = nb >= 64;   // many block counts: the digit-parallel scan
    uint64_t* src = keys;
    uint64_t* dst = tmp;
    for (int pass = 0; pass < 8; ++pass) {
        const int shift = 8 * pass;
        count_launches(1);
        sort_upsweep_kernel<<<(unsigned)nb, kSortBlock, 0, st>>>(src, count, shift, hist, nb);
        if (wide) {
            count_launches(2);
            digit_sum_kernel<<<256, 256, 0, st>>>(hist, nb, digit_total);
            digit_scan_kernel<<<256, 1024, 0, st>>>(hist, nb, digit_total, total);
        } else {
            count_launches(1);
            scan_counts_kernel<<<1, 1024, 0, st>>>(hist, 256 * nb, total);
        }
        count_launches(1);
        sort_downsweep_kernel<<<(unsigned)nb, kSortBlock, 0, st>>>(src, dst, count, shift, hist,
                                                                   nb);
        uint64_t* x = src;
        src = dst;
        dst = x;
    }
    // 8 passes: the result is back in `keys`
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// emit the first n sorted keys and mark them emitted
// ---------------------------------------------------------------------------
__global__ void emit_kernel(const uint64_t* __restrict__ keys, int n, const int32_t* w_id,
                            float* w_lo, float* w_hi, float* lo, float* hi, int64_t* out_ids,
                            float* out_scores) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const uint64_t k = keys[i];
    const uint32_t w = rank_key_id(k);
    const int32_t id = w_id[w];
    out_ids[i] = id;
    out_scores[i] = rank_key_score(k);
    w_lo[w] = -INFINITY;
    w_hi[w] = -INFINITY;
    if (lo) {
        lo[id] = -INFINITY;
        hi[id] = -INFINITY;
    }
}

cudaError_t launch_emit(const uint64_t* keys, int n, const int32_t* w_id, float* w_lo,
                        float* w_hi, float* lo, float* hi, int64_t* out_ids, float* out_scores,
                        cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    count_launches(1);
    emit_kernel<<<(n + 255) / 256, 256, 0, st>>>(keys, n, w_id, w_lo, w_hi, lo, hi, out_ids,
                                                 out_scores);
    return cudaGetLastError();
}

}  // namespace pvs
