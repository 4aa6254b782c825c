// Exhaustive float32 scanning, the dense rank generator that PVS is compared
// with in the rank-generator ablation (arXiv 2608.07152 Sec. 3.5, 4.4): the
// authoritative score of every visible row (the same exact dot product as
// PVS refinement, Sec. 2.3.1), then one full sort by (score desc, id asc);
// pulls read the sorted keys in order.
#include "exact_dot.cuh"
#include "kernels.h"
#include "pvs_common.cuh"

namespace pvs {

constexpr int kScanWarps = 8;

__global__ void __launch_bounds__(kScanWarps * 32) scan_scores_kernel(
    const float* __restrict__ qraw, const float* __restrict__ raw, int m_raw, int64_t rows,
    const uint32_t* __restrict__ tomb, uint64_t* keys, int* status, DevCounters* ctr) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * kScanWarps;
    unsigned long long scored = 0, fallbacks = 0;
    for (int64_t row = (int64_t)blockIdx.x * kScanWarps + (threadIdx.x >> 5); row < rows;
         row += warps) {
        const bool live = !tomb || ((tomb[row >> 5] >> (row & 31)) & 1u) == 0;
        if (!live) {
            if (lane == 0) keys[row] = 0;
            continue;
        }
        bool fb = false;
        const float s = exact_dot_warp_eft(qraw, qraw, raw + row * (int64_t)m_raw, m_raw, &fb);
        if (lane == 0) {
            if (!isfinite(s)) set_status(status, PVS_ERR_OVERFLOW);
            keys[row] = rank_key(s, (uint32_t)row);
            ++scored;
            fallbacks += fb ? 1 : 0;
        }
    }
    if (lane == 0 && scored) {
        atomicAdd(&ctr->refined, scored);
        if (fallbacks) atomicAdd(&ctr->exact_fallbacks, fallbacks);
    }
}

cudaError_t launch_scan_scores(const float* qraw, const float* raw, int m_raw, int64_t rows,
                               const uint32_t* tomb, uint64_t* keys, int* status,
                               DevCounters* ctr, cudaStream_t st) {
    if (rows <= 0) return cudaSuccess;
    int64_t blocks = (rows + kScanWarps - 1) / kScanWarps;
    if (blocks > 152 * 16) blocks = 152 * 16;
    count_launches(1);
    scan_scores_kernel<<<(unsigned)blocks, kScanWarps * 32, 0, st>>>(qraw, raw, m_raw, rows, tomb,
                                                                    keys, status, ctr);
    return cudaGetLastError();
}

__global__ void scan_emit_kernel(const uint64_t* __restrict__ keys, int64_t n, int64_t* ids,
                                 float* scores, const int* status, int* mirror) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        ids[i] = (int64_t)rank_key_id(keys[i]);
        scores[i] = rank_key_score(keys[i]);
    }
    // the status word is published last (the host may poll it): a launch that
    // publishes is one block, and its writes are made visible to the host first
    if (mirror) {
        __syncthreads();
        if (threadIdx.x == 0) {
            __threadfence_system();
            *reinterpret_cast<volatile int*>(mirror) = *reinterpret_cast<const volatile int*>(status);
        }
    }
}

cudaError_t launch_scan_emit(const uint64_t* keys, int64_t n, int64_t* ids, float* scores,
                             const int* status, int* mirror, cudaStream_t st) {
    int64_t blocks = (n + 255) / 256;
    if (blocks < 1) blocks = 1;
    if (blocks > 152 * 4) blocks = 152 * 4;
    if (mirror) blocks = 1;   // one block publishes after all of its writes
    count_launches(1);
    scan_emit_kernel<<<(unsigned)blocks, 256, 0, st>>>(keys, n, ids, scores, status, mirror);
    return cudaGetLastError();
}

}  // namespace pvs
