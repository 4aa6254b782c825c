// Authoritative float32 scores of PVS candidates (Sec. 2.3.1: raw vectors are
// read only for candidates the intervals do not order; App. A.1: a score
// outside its interval fails the request).  The score itself is computed by
// exact_dot_warp_eft (exact_dot.cuh): RN_f32 of the exact inner product.
#include "exact_dot.cuh"
#include "kernels.h"
#include "pipeline.cuh"
#include "pvs_common.cuh"

namespace pvs {

// Warps warp0, warp0 + nwarps, ... of the launch score candidates of one
// cursor.  lo / hi (bounds of every row) may be null for a cursor that only
// holds a working set.  A warp fetches the metadata of its next 32
// candidates at once (lane j holds candidate j) and broadcasts it with
// shuffles, so each candidate waits on its row alone.
__device__ inline void refine_warps(const int32_t* __restrict__ cand, const unsigned int* cand_len,
                                    const int32_t* __restrict__ w_id, float* w_lo, float* w_hi,
                                    float* lo, float* hi, const float* q_fast,
                                    const float* __restrict__ qraw,
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
            const float s = exact_dot_warp_eft(q_fast, qraw, raw + (int64_t)idj * m_raw, m_raw, &fb);
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

// The query in shared memory when it fits (stage_q: m_raw floats of dynamic
// shared memory), else read from global memory.
__device__ inline const float* stage_query(const float* qraw, int m_raw, int stage_q) {
    extern __shared__ float4 q_sh[];
    if (!stage_q) return qraw;
    const float4* src = reinterpret_cast<const float4*>(qraw);
    for (int i = threadIdx.x; i < (m_raw >> 2); i += blockDim.x) q_sh[i] = src[i];
    __syncthreads();
    return reinterpret_cast<const float*>(q_sh);
}

__global__ void __launch_bounds__(256, 3) refine_kernel(
    const int32_t* __restrict__ cand, const unsigned int* cand_len, const int32_t* __restrict__ w_id,
    float* w_lo, float* w_hi, float* lo, float* hi, const float* __restrict__ qraw,
    const float* __restrict__ raw, int m_raw, int* status, DevCounters* ctr, int stage_q) {
    const float* qf = stage_query(qraw, m_raw, stage_q);
    refine_warps(cand, cand_len, w_id, w_lo, w_hi, lo, hi, qf, qraw, raw, m_raw, status, ctr,
                 (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5),
                 (int64_t)gridDim.x * (blockDim.x >> 5));
}

// Many cursors at once: blocks_per_cursor consecutive blocks serve cursor
// blockIdx.x / blocks_per_cursor.
__global__ void __launch_bounds__(256, 3)
    refine_batch_kernel(const __grid_constant__ PullArgsPack args, int blocks_per_cursor,
                        int stage_q) {
    const PullArgs& a = args.a[blockIdx.x / blocks_per_cursor];
    const float* qf = stage_query(a.qraw, a.m_raw, stage_q);
    const int64_t warps_per_block = blockDim.x >> 5;
    refine_warps(a.cand, &a.ctr->cand, a.w_id, a.w_lo, a.w_hi, a.lo, a.hi, qf, a.qraw, a.raw,
                 a.m_raw, a.status, a.ctr,
                 (int64_t)(blockIdx.x % blocks_per_cursor) * warps_per_block + (threadIdx.x >> 5),
                 (int64_t)blocks_per_cursor * warps_per_block);
}

// ---- bulk-copy ring: rows stream into shared memory ---------------------------
// Each warp owns `stages` row buffers with one mbarrier each.  Lane 0 issues a
// 1-D bulk copy (cp.async.bulk, L2 evict-first) of the next candidate's row
// into a free buffer while the warp scores the row in the oldest one, so a
// warp keeps up to `stages` rows in flight without holding them in registers.
// Candidate metadata is fetched 32 at a time (lane j holds candidate j) and
// rows already resolved (lo == hi) are skipped before any copy.
constexpr int kRingWarps = 8;
constexpr int kRingMaxStages = 4;
constexpr size_t kRingSmemBudget = 110 * 1024;   // two blocks per SM

struct RingRefs {
    const int32_t* cand;
    const unsigned int* cand_len;
    const int32_t* w_id;
    float* w_lo;
    float* w_hi;
    float* lo;
    float* hi;
    const float* qraw;
    const float* raw;
    int m_raw;
    int* status;
    DevCounters* ctr;
};

// Dynamic shared memory: q [m_raw] | rows [kRingWarps][stages][m_raw] |
// bars [kRingWarps][stages] | meta [kRingWarps][stages] (int4: w, lo, hi, id).
__host__ __device__ inline size_t ring_smem_bytes(int m_raw, int stages) {
    const size_t row = (size_t)m_raw * sizeof(float);
    return row + (size_t)kRingWarps * stages * (row + sizeof(uint64_t) + sizeof(int4));
}

__device__ inline void refine_ring(const RingRefs& a, int stages, int64_t warp0, int64_t nwarps) {
    extern __shared__ float4 ring_sh[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n4 = a.m_raw >> 2;
    float4* q_sh = ring_sh;
    float4* rows = ring_sh + n4 + (size_t)warp * stages * n4;
    uint64_t* bars = reinterpret_cast<uint64_t*>(ring_sh + n4 + (size_t)kRingWarps * stages * n4) +
                     warp * stages;
    int4* meta = reinterpret_cast<int4*>(reinterpret_cast<uint64_t*>(
                     ring_sh + n4 + (size_t)kRingWarps * stages * n4) + kRingWarps * stages) +
                 warp * stages;
    const float4* q4 = reinterpret_cast<const float4*>(a.qraw);
    for (int i = threadIdx.x; i < n4; i += blockDim.x) q_sh[i] = q4[i];
    if (lane == 0) {
        for (int st = 0; st < stages; ++st) mbar_init(&bars[st], 1);
        mbar_fence_init();
    }
    __syncthreads();

    const int64_t n = *a.cand_len;
    const uint32_t row_bytes = (uint32_t)a.m_raw * sizeof(float);
    const uint64_t pol = l2_evict_first_policy();
    // producer cursor over this warp's candidates warp0, warp0 + nwarps, ...
    int64_t pbase = warp0;
    unsigned int pmask = 0;
    int32_t pw = 0, pid = 0;
    float pl = 0.0f, ph = 0.0f;
    auto issue = [&](int st) -> bool {
        while (pmask == 0) {
            if (pbase >= n) return false;
            const int64_t mine = pbase + lane * nwarps;
            bool need = false;
            if (mine < n) {
                pw = a.cand[mine];
                pl = a.w_lo[pw];
                ph = a.w_hi[pw];
                pid = a.w_id[pw];
                need = pl < ph;   // lo == hi: already the exact score
            }
            pmask = __ballot_sync(0xffffffffu, need);
            pbase += 32 * nwarps;
        }
        const int j = __ffs(pmask) - 1;
        pmask &= pmask - 1;
        const int32_t wj = __shfl_sync(0xffffffffu, pw, j);
        const int32_t idj = __shfl_sync(0xffffffffu, pid, j);
        const float lj = __shfl_sync(0xffffffffu, pl, j);
        const float hj = __shfl_sync(0xffffffffu, ph, j);
        if (lane == 0) {
            meta[st] = make_int4(wj, __float_as_int(lj), __float_as_int(hj), idj);
            fence_proxy_async_smem();   // the warp's reads of this buffer come first
            mbar_arrive_expect_tx(&bars[st], row_bytes);
            bulk_g2s(rows + (size_t)st * n4, a.raw + (int64_t)idj * a.m_raw, row_bytes, &bars[st],
                     pol);
        }
        return true;
    };

    int issued = 0;
    while (issued < stages && issue(issued)) ++issued;
    __syncwarp();
    unsigned long long refined = 0, fallbacks = 0;
    int k = 0;
    for (; k < issued; ++k) {
        const int st = k % stages;
        // warp-uniform: every lane must agree before the warp-wide steps below
        if (!__all_sync(0xffffffffu, mbar_wait(&bars[st], (uint32_t)((k / stages) & 1)))) break;
        const int4 md = meta[st];
        const float lj = __int_as_float(md.y), hj = __int_as_float(md.z);
        const float* vg = a.raw + (int64_t)md.w * a.m_raw;
        bool fb;
        const float s = exact_dot_warp_eft_smem(reinterpret_cast<const float*>(q_sh), a.qraw,
                                                reinterpret_cast<const float*>(rows + (size_t)st * n4),
                                                vg, a.m_raw, &fb);
        if (lane == 0) {
            ++refined;
            fallbacks += fb;
            if (!isfinite(s)) set_status(a.status, PVS_ERR_OVERFLOW);
            else if (s < lj || s > hj) set_status(a.status, PVS_ERR_INTERVAL);
            a.w_lo[md.x] = s;
            a.w_hi[md.x] = s;
            if (a.lo) {
                a.lo[md.w] = s;
                a.hi[md.w] = s;
            }
        }
        __syncwarp();
        if (issue(st)) ++issued;
    }
    if (k < issued) {   // a copy did not arrive in time: record it, drain every copy in flight
        if (lane == 0) set_status(a.status, PVS_ERR_TIMEOUT);
        for (int k2 = k; k2 < issued; ++k2)
            mbar_wait(&bars[k2 % stages], (uint32_t)((k2 / stages) & 1));
    }
    if (lane == 0 && refined) {
        atomicAdd(&a.ctr->refined, refined);
        if (fallbacks) atomicAdd(&a.ctr->exact_fallbacks, fallbacks);
    }
}

__global__ void __launch_bounds__(kRingWarps * 32, 2) refine_ring_kernel(RingRefs a, int stages) {
    refine_ring(a, stages, (int64_t)blockIdx.x * kRingWarps + (threadIdx.x >> 5),
                (int64_t)gridDim.x * kRingWarps);
}

__global__ void __launch_bounds__(kRingWarps * 32, 2) refine_ring_batch_kernel(
    const __grid_constant__ PullArgsPack args, int blocks_per_cursor, int stages) {
    const PullArgs& p = args.a[blockIdx.x / blocks_per_cursor];
    const RingRefs a{p.cand, &p.ctr->cand, p.w_id, p.w_lo, p.w_hi, p.lo, p.hi,
                     p.qraw, p.raw, p.m_raw, p.status, p.ctr};
    refine_ring(a, stages, (int64_t)(blockIdx.x % blocks_per_cursor) * kRingWarps +
                               (threadIdx.x >> 5),
                (int64_t)blocks_per_cursor * kRingWarps);
}

// Ring depth for rows of m_raw floats within the shared-memory budget; 0 when
// fewer than two buffers per warp fit (then the register path runs).
static int ring_stages(int m_raw) {
    for (int st = kRingMaxStages; st >= 2; --st)
        if (ring_smem_bytes(m_raw, st) <= kRingSmemBudget) return st;
    return 0;
}

static cudaError_t ring_attr(const void* fn, size_t smem) {
    return raise_smem_limit(fn, smem);
}

// Staging the query takes m_raw floats of shared memory; up to 48 KB.
static int query_stage_bytes(int m_raw) {
    const size_t b = (size_t)m_raw * sizeof(float);
    return b <= 48 * 1024 ? (int)b : 0;
}

cudaError_t launch_refine_batch(const PullArgsPack& args_dev, int ncursors, int blocks_per_cursor,
                                int m_raw, cudaStream_t st) {
    if (ncursors <= 0) return cudaSuccess;
    const int stages = ring_stages(m_raw);
    if (stages) {
        const size_t smem = ring_smem_bytes(m_raw, stages);
        cudaError_t e = ring_attr((const void*)refine_ring_batch_kernel, smem);
        if (e != cudaSuccess) return e;
        count_launches(1);
        refine_ring_batch_kernel<<<ncursors * blocks_per_cursor, kRingWarps * 32, smem, st>>>(
            args_dev, blocks_per_cursor, stages);
        return cudaGetLastError();
    }
    const int smem = query_stage_bytes(m_raw);
    count_launches(1);
    refine_batch_kernel<<<ncursors * blocks_per_cursor, 256, smem, st>>>(args_dev,
                                                                          blocks_per_cursor,
                                                                          smem > 0);
    return cudaGetLastError();
}

cudaError_t launch_refine(const int32_t* cand, const unsigned int* cand_len,
                          const int32_t* w_id, float* w_lo, float* w_hi, float* lo, float* hi,
                          const float* qraw, const float* raw, int m_raw, int* status,
                          DevCounters* ctr, int grid, cudaStream_t st) {
    const int stages = ring_stages(m_raw);
    if (stages) {
        const size_t smem = ring_smem_bytes(m_raw, stages);
        cudaError_t e = ring_attr((const void*)refine_ring_kernel, smem);
        if (e != cudaSuccess) return e;
        count_launches(1);
        const RingRefs a{cand, cand_len, w_id, w_lo, w_hi, lo, hi, qraw, raw, m_raw, status, ctr};
        refine_ring_kernel<<<grid, kRingWarps * 32, smem, st>>>(a, stages);
        return cudaGetLastError();
    }
    const int smem = query_stage_bytes(m_raw);
    count_launches(1);
    refine_kernel<<<grid, 256, smem, st>>>(cand, cand_len, w_id, w_lo, w_hi, lo, hi, qraw, raw,
                                           m_raw, status, ctr, smem > 0);
    return cudaGetLastError();
}

__global__ void score_ids_kernel(const int64_t* ids, int n, const float* qraw, const float* raw,
                                 int m_raw, float* out, DevCounters* ctr) {
    const int lane = threadIdx.x & 31;
    const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (i >= n) return;
    bool fb;
    const float s = exact_dot_warp_eft(qraw, qraw, raw + ids[i] * m_raw, m_raw, &fb);
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
