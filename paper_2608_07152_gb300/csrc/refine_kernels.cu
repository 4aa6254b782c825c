// Authoritative float32 scores of PVS candidates (Sec. 2.3.1: raw vectors are
// read only for candidates the intervals do not order; App. A.1: a score
// outside its interval fails the request).  The score itself is computed by
// exact_dot_warp_eft (exact_dot.cuh): RN_f32 of the exact inner product.
#include "exact_dot.cuh"
#include "kernels.h"
#include "pvs_common.cuh"

namespace pvs {

// Warps warp0, warp0 + nwarps, ... of the launch score candidates of one
// cursor.  lo / hi (bounds of every row) may be null for a cursor that only
// holds a working set.  A warp fetches the metadata of its next 32
// candidates at once (lane j holds candidate j) and broadcasts it with
// shuffles, so each candidate waits on its row alone.
__device__ inline void refine_warps(const int32_t* __restrict__ cand, const unsigned int* cand_len,
                                    const int32_t* __restrict__ w_id, float* w_lo, float* w_hi,
                                    float* lo, float* hi, const float* __restrict__ qraw,
                                    const float* __restrict__ raw, int m_raw, int* status,
                                    DevCounters* ctr, int64_t warp0, int64_t nwarps) {
    const int lane = threadIdx.x & 31;
    const int64_t n = *cand_len;
    unsigned long long refined = 0, fallbacks = 0;
#pragma unroll 1
    for (int64_t base = warp0; base < n; base += 32 * nwarps) {
        const int64_t mine = base + lane * nwarps;
        int32_t w = 0, id = 0;
        float l = 0.0f, h = 0.0f;   // l == h: nothing to do
        if (mine < n) {
            w = cand[mine];
            l = w_lo[w];
            h = w_hi[w];
            id = w_id[w];
        }
        const int64_t left = (n - base + nwarps - 1) / nwarps;   // candidates of this warp left
        const int cnt = left < 32 ? (int)left : 32;
#pragma unroll 1
        for (int j = 0; j < cnt; ++j) {
            const float lj = __shfl_sync(0xffffffffu, l, j);
            const float hj = __shfl_sync(0xffffffffu, h, j);
            const int32_t wj = __shfl_sync(0xffffffffu, w, j);
            const int32_t idj = __shfl_sync(0xffffffffu, id, j);
            if (!(lj < hj)) continue;    // resolved: lo == hi is the exact score
            bool fb;
            const float s = exact_dot_warp_eft(qraw, raw + (int64_t)idj * m_raw, m_raw, &fb);
            if (lane == 0) {
                ++refined;
                fallbacks += fb;
                if (!isfinite(s)) set_status(status, PVS_ERR_OVERFLOW);
                else if (s < lj || s > hj) set_status(status, PVS_ERR_INTERVAL);
                w_lo[wj] = s;
                w_hi[wj] = s;
                if (lo) {
                    lo[idj] = s;
                    hi[idj] = s;
                }
            }
        }
    }
    if (lane == 0 && refined) {
        atomicAdd(&ctr->refined, refined);
        if (fallbacks) atomicAdd(&ctr->exact_fallbacks, fallbacks);
    }
}

__global__ void __launch_bounds__(256) refine_kernel(
    const int32_t* __restrict__ cand, const unsigned int* cand_len, const int32_t* __restrict__ w_id,
    float* w_lo, float* w_hi, float* lo, float* hi, const float* __restrict__ qraw,
    const float* __restrict__ raw, int m_raw, int* status, DevCounters* ctr) {
    refine_warps(cand, cand_len, w_id, w_lo, w_hi, lo, hi, qraw, raw, m_raw, status, ctr,
                 (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5),
                 (int64_t)gridDim.x * (blockDim.x >> 5));
}

// Many cursors at once: blocks_per_cursor consecutive blocks serve cursor
// blockIdx.x / blocks_per_cursor.
__global__ void __launch_bounds__(256) refine_batch_kernel(const PullArgs* args,
                                                           int blocks_per_cursor) {
    const PullArgs& a = args[blockIdx.x / blocks_per_cursor];
    const int64_t warps_per_block = blockDim.x >> 5;
    refine_warps(a.cand, &a.ctr->cand, a.w_id, a.w_lo, a.w_hi, a.lo, a.hi, a.qraw, a.raw,
                 a.m_raw, a.status, a.ctr,
                 (int64_t)(blockIdx.x % blocks_per_cursor) * warps_per_block + (threadIdx.x >> 5),
                 (int64_t)blocks_per_cursor * warps_per_block);
}

cudaError_t launch_refine_batch(const PullArgs* args_dev, int ncursors, int blocks_per_cursor,
                                cudaStream_t st) {
    if (ncursors <= 0) return cudaSuccess;
    count_launches(1);
    refine_batch_kernel<<<ncursors * blocks_per_cursor, 256, 0, st>>>(args_dev,
                                                                       blocks_per_cursor);
    return cudaGetLastError();
}

cudaError_t launch_refine(const int32_t* cand, const unsigned int* cand_len,
                          const int32_t* w_id, float* w_lo, float* w_hi, float* lo, float* hi,
                          const float* qraw, const float* raw, int m_raw, int* status,
                          DevCounters* ctr, int grid, cudaStream_t st) {
    count_launches(1);
    refine_kernel<<<grid, 256, 0, st>>>(cand, cand_len, w_id, w_lo, w_hi, lo, hi, qraw, raw,
                                        m_raw, status, ctr);
    return cudaGetLastError();
}

__global__ void score_ids_kernel(const int64_t* ids, int n, const float* qraw, const float* raw,
                                 int m_raw, float* out, DevCounters* ctr) {
    const int lane = threadIdx.x & 31;
    const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (i >= n) return;
    bool fb;
    const float s = exact_dot_warp_eft(qraw, raw + ids[i] * m_raw, m_raw, &fb);
    if (lane == 0) {
        out[i] = s;
        if (fb) atomicAdd(&ctr->exact_fallbacks, 1ull);
    }
}

cudaError_t launch_score_ids(const int64_t* ids, int n, const float* qraw, const float* raw,
                             int m_raw, float* out, DevCounters* ctr, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    count_launches(1);
    score_ids_kernel<<<(n + 7) / 8, 256, 0, st>>>(ids, n, qraw, raw, m_raw, out, ctr);
    return cudaGetLastError();
}

}  // namespace pvs
