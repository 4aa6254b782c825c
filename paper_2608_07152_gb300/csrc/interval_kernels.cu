// PVS interval pass (Sec. 2.3.1, App. A.1): one streaming pass over the Int8
// codes that writes the outward-rounded score interval [lo, hi] of every
// visible vector.
//
// Single query = an HBM-bound GEMV.  Persistent CTAs (one per SM) own a
// strided sequence of 64-row tiles.  A producer warp stages each tile (codes
// plus the three per-vector parameters) into shared memory with 1-D bulk
// copies (the TMA engine's cp.async.bulk) through an S-deep mbarrier ring,
// with an L2 evict-first hint because every code byte is read exactly once.
// Eight consumer warps compute: a quad of lanes owns one row, each lane
// accumulates dp4a over a quarter of the row's 16-byte chunks against the
// query codes held in registers, two shuffles reduce the quad, and lane 0 of
// the quad evaluates the interval epilogue and writes (lo, hi).
//
// Shared-memory banks: a quarter-warp (8 lanes) reads 2 rows x 4 chunks.
// When a code row spans a multiple of 8 chunks, odd rows walk their chunks
// rotated by one step of 4 so the 8 addresses hit 8 distinct 16-byte bank
// groups.
#include "kernels.h"
#include "pipeline.cuh"
#include "pvs_common.cuh"

namespace pvs {

constexpr int kConsumerWarps = 8;
constexpr int kIntervalThreads = (kConsumerWarps + 1) * 32;

// CPL = 16-byte chunks per lane per row = m_pad / 64 (compile-time), or 0 for
// a runtime count with the query chunks read from global memory.
template <int CPL>
__global__ void __launch_bounds__(kIntervalThreads, 1)
    interval_pass_kernel(IntervalArgs a, int stages, int rotate, int cpl_rt) {
    extern __shared__ __align__(128) uint8_t smem[];
    constexpr int TR = kTileRows;
    const int m_pad = a.m_pad;
    const int stage_bytes = TR * m_pad + 3 * TR * 4;
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)stages * stage_bytes);
    uint64_t* empty = full + stages;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t ntiles = (a.rows + TR - 1) / TR;

    if (threadIdx.x == 0) {
        for (int s = 0; s < stages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kConsumerWarps);
        }
        mbar_fence_init();
    }
    __syncthreads();

    if (warp == kConsumerWarps) {
        // ---------------- producer ----------------
        if (lane == 0) {
            const uint64_t pol = l2_evict_first_policy();
            int k = 0;
            bool ok = true;
            for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++k) {
                const int s = k % stages;
                const uint32_t ph = (uint32_t)(k / stages) & 1u;
                if (!mbar_wait(&empty[s], ph ^ 1u, a.wait_ns)) {
                    set_status(a.status, PVS_ERR_TIMEOUT);
                    ok = false;
                    break;
                }
                const int64_t r0 = t * TR;
                const int rows_t = (int)(a.rows - r0 < TR ? a.rows - r0 : TR);
                const uint32_t cb = (uint32_t)rows_t * (uint32_t)m_pad;
                const uint32_t pb = (uint32_t)((rows_t + 3) & ~3) * 4u;
                uint8_t* dst = smem + (size_t)s * stage_bytes;
                mbar_arrive_expect_tx(&full[s], cb + 3u * pb);
                bulk_g2s(dst, a.codes + r0 * m_pad, cb, &full[s], pol);
                bulk_g2s(dst + TR * m_pad, a.scale + r0, pb, &full[s], pol);
                bulk_g2s(dst + TR * m_pad + TR * 4, a.vnorm + r0, pb, &full[s], pol);
                bulk_g2s(dst + TR * m_pad + 2 * TR * 4, a.enorm + r0, pb, &full[s], pol);
            }
            // drain: the last copy into every used stage has landed before exit
            const int issued = k;
            for (int s = 0; s < stages && s < issued; ++s) {
                const int last = issued - 1 - ((issued - 1 - s) % stages);
                if (!mbar_wait(&full[s], (uint32_t)(last / stages) & 1u) && ok)
                    set_status(a.status, PVS_ERR_TIMEOUT);
            }
        }
        return;
    }

    // ---------------- consumers ----------------
    const int quad = lane >> 2, p = lane & 3;
    const int r_in_tile = warp * 8 + quad;
    const int par = rotate ? (quad & 1) : 0;
    const int cpl = CPL > 0 ? CPL : cpl_rt;
    const QueryScalars q = *a.qs;
    const int4* zq4 = reinterpret_cast<const int4*>(a.zq);

    int4 qreg[CPL > 0 ? CPL : 1];
    if constexpr (CPL > 0) {
#pragma unroll
        for (int j = 0; j < CPL; ++j) {
            int jj = j + par;
            if (jj >= CPL) jj -= CPL;
            qreg[j] = zq4[4 * jj + p];
        }
    }

    // the slot's kSlotTop largest live lower bounds, descending
    float top[kSlotTop];
#pragma unroll
    for (int j = 0; j < kSlotTop; ++j) top[j] = -INFINITY;

    int k = 0;
    for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++k) {
        const int s = k % stages;
        const uint32_t ph = (uint32_t)(k / stages) & 1u;
        if (!mbar_wait(&full[s], ph, a.wait_ns)) {
            if (lane == 0) set_status(a.status, PVS_ERR_TIMEOUT);
            break;
        }
        const uint8_t* stage = smem + (size_t)s * stage_bytes;
        const int64_t row = t * TR + r_in_tile;
        const int4* rowp = reinterpret_cast<const int4*>(stage + r_in_tile * m_pad);
        int acc0 = 0, acc1 = 0;
        if (row < a.rows) {
            if constexpr (CPL > 0) {
#pragma unroll
                for (int j = 0; j < CPL; ++j) {
                    int jj = j + par;
                    if (jj >= CPL) jj -= CPL;
                    const int4 cv = rowp[4 * jj + p];
                    acc0 = __dp4a(cv.x, qreg[j].x, acc0);
                    acc1 = __dp4a(cv.y, qreg[j].y, acc1);
                    acc0 = __dp4a(cv.z, qreg[j].z, acc0);
                    acc1 = __dp4a(cv.w, qreg[j].w, acc1);
                }
            } else {
                for (int j = 0; j < cpl; ++j) {
                    int jj = j + par;
                    if (jj >= cpl) jj -= cpl;
                    const int4 cv = rowp[4 * jj + p];
                    const int4 qv = zq4[4 * jj + p];
                    acc0 = __dp4a(cv.x, qv.x, acc0);
                    acc1 = __dp4a(cv.y, qv.y, acc1);
                    acc0 = __dp4a(cv.z, qv.z, acc0);
                    acc1 = __dp4a(cv.w, qv.w, acc1);
                }
            }
        }
        int dot = acc0 + acc1;
        dot += __shfl_xor_sync(0xffffffffu, dot, 1);
        dot += __shfl_xor_sync(0xffffffffu, dot, 2);
        if (p == 0 && row < a.rows) {
            const float* ps = reinterpret_cast<const float*>(stage + TR * m_pad);
            float lo, hi;
            interval_epilogue(dot, q, ps[r_in_tile], ps[TR + r_in_tile], ps[2 * TR + r_in_tile],
                              lo, hi);
            if (!isfinite(lo) || !isfinite(hi)) set_status(a.status, PVS_ERR_OVERFLOW);
            if (tombstoned(a.tomb, row)) lo = hi = -INFINITY;
            a.lo[row] = lo;
            a.hi[row] = hi;
            if (lo > top[kSlotTop - 1]) {   // insertion into the descending list
                top[kSlotTop - 1] = lo;
#pragma unroll
                for (int j = kSlotTop - 1; j > 0; --j)
                    if (top[j] > top[j - 1]) {
                        const float x = top[j];
                        top[j] = top[j - 1];
                        top[j - 1] = x;
                    }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[s]);
    }
    if (a.slot_top && p == 0) {
        float* o = a.slot_top + ((size_t)blockIdx.x * TR + (size_t)r_in_tile) * kSlotTop;
#pragma unroll
        for (int j = 0; j < kSlotTop; ++j) o[j] = top[j];
    }
}

template <int CPL>
static cudaError_t launch_tpl(const IntervalArgs& a, int num_sms, cudaStream_t st) {
    const int stage_bytes = kTileRows * a.m_pad + 3 * kTileRows * 4;
    int stages = (200 * 1024) / stage_bytes;
    if (stages > 8) stages = 8;
    if (stages < 2) return cudaErrorInvalidValue;
    const size_t smem = (size_t)stages * stage_bytes + 2 * stages * sizeof(uint64_t);
    cudaError_t e = raise_smem_limit((const void*)interval_pass_kernel<CPL>, smem);
    if (e != cudaSuccess) return e;
    const int64_t ntiles = (a.rows + kTileRows - 1) / kTileRows;
    const int grid = (int)(ntiles < num_sms ? ntiles : num_sms);
    const int chunks = a.m_pad / 16;
    const int rotate = (chunks % 8) == 0 ? 1 : 0;
    count_launches(1);
    interval_pass_kernel<CPL><<<grid, kIntervalThreads, smem, st>>>(a, stages, rotate,
                                                                     a.m_pad / 64);
    return cudaGetLastError();
}

// The staged kernel serves these row widths (the others take the unstaged one).
static bool staged_width(int m_pad) {
    switch (m_pad / 64) {
        case 1: case 2: case 4: case 6: case 8: case 12: case 16: return true;
        default: break;
    }
    return kTileRows * m_pad + 3 * kTileRows * 4 <= 100 * 1024;
}

int64_t interval_slots(int64_t rows, int m_pad, int num_sms, int64_t* min_rows_per_slot) {
    *min_rows_per_slot = 0;
    if (rows <= 0 || !staged_width(m_pad)) return 0;
    const int64_t ntiles = (rows + kTileRows - 1) / kTileRows;
    const int64_t grid = ntiles < num_sms ? ntiles : num_sms;
    // CTA b scans tiles b, b + grid, ...: at least ntiles / grid of them, of
    // which only the very last tile of the pass can be partial
    *min_rows_per_slot = ntiles / grid - 1;
    return grid * kTileRows;
}

cudaError_t launch_interval_pass(const IntervalArgs& a, int num_sms, cudaStream_t st) {
    if (a.rows <= 0) return cudaSuccess;
    switch (a.m_pad / 64) {
        case 1: return launch_tpl<1>(a, num_sms, st);
        case 2: return launch_tpl<2>(a, num_sms, st);
        case 4: return launch_tpl<4>(a, num_sms, st);
        case 6: return launch_tpl<6>(a, num_sms, st);
        case 8: return launch_tpl<8>(a, num_sms, st);
        case 12: return launch_tpl<12>(a, num_sms, st);
        case 16: return launch_tpl<16>(a, num_sms, st);
        default: break;
    }
    if (kTileRows * a.m_pad + 3 * kTileRows * 4 <= 100 * 1024) return launch_tpl<0>(a, num_sms, st);
    return launch_interval_simple(a, st);
}

// Unstaged variant: one warp per row, lane-strided 4-byte code words.  Used
// for code rows too long for two shared-memory stages.
__global__ void interval_simple_kernel(IntervalArgs a) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    const QueryScalars q = *a.qs;
    const int words = a.m_pad / 4;
    const int* zq = reinterpret_cast<const int*>(a.zq);
    for (int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
         row < a.rows; row += warps) {
        const int* cw = reinterpret_cast<const int*>(a.codes + row * a.m_pad);
        int acc = 0;
        for (int j = lane; j < words; j += kWarp) acc = __dp4a(cw[j], zq[j], acc);
        acc = warp_sum(acc);
        if (lane == 0) {
            float lo, hi;
            interval_epilogue(acc, q, a.scale[row], a.vnorm[row], a.enorm[row], lo, hi);
            if (!isfinite(lo) || !isfinite(hi)) set_status(a.status, PVS_ERR_OVERFLOW);
            if (tombstoned(a.tomb, row)) lo = hi = -INFINITY;
            a.lo[row] = lo;
            a.hi[row] = hi;
        }
    }
}

cudaError_t launch_interval_simple(const IntervalArgs& a, cudaStream_t st) {
    if (a.rows <= 0) return cudaSuccess;
    int64_t blocks = (a.rows + 7) / 8;
    if (blocks > 152 * 16) blocks = 152 * 16;
    count_launches(1);
    interval_simple_kernel<<<(unsigned)blocks, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace pvs
