// Grouped PVS interval pass (Sec. 2.3.1, App. A.1): the score intervals of
// up to kGroupMax = 16 queries from one streaming read of the Int8 codes.
//
// A single query's pass is an HBM-bound GEMV at about one Int8 operation per
// byte; queries answered together can share its code stream.  For 8
// queries the exact Int8 dot products are a [rows x m] x [m x 8] product,
// done here on the tensor cores with warp-level mma.sync m16n8k16 (16 rows x
// 8 queries per instruction, f16 operands, f32 accumulation).  GB300 has no
// Int8 tcgen05 MMA, and its legacy Int8 mma.sync runs at about a quarter of
// the f16 rate; the codes are converted to f16 in registers instead, which
// is exact: |z| <= 127, every product is an integer below 2^14 and every
// partial sum an integer below 2^24, so the f32 accumulator holds the exact
// Int8 dot product.  (dp4a on the CUDA cores, at two warp instructions per
// clock per SM, made the 8-query pass compute-bound at 1.7 ms; s8 mma.sync
// on the codes as they are, with eight consumer warps per SM, bound by the
// tensor pipe at 1.49 ms.)  The conversion and the epilogue make the
// consumers' arithmetic about as long as the code stream at 8 queries, so
// 16 queries (split, below) take twice as long per pass: no gain per query.
//
// Structure: a persistent CTA per SM; a producer thread stages 64-row tiles
// (codes, then the three per-vector parameter arrays) with four 1-D bulk
// copies (the TMA engine's cp.async.bulk) through an mbarrier ring, as the
// single-query pass does.  Eight consumer warps form two groups of four;
// warp b of a group owns rows 16b .. 16b+15 of the tiles it takes.  With up
// to 8 queries the groups take alternate tiles, each for every query; with
// 9 .. 16 (split) both take every tile, group 0 for queries 0 .. 7 and
// group 1 for queries 8 .. 15, so a tile is released once all eight warps
// have read it (query fragments in registers: m_pad up to 768).
// (Rows staged one bulk copy each, into a padded pitch free of bank
// conflicts, made the TMA issue rate the limit: 2.4 ms per pass.  With
// unpadded rows the fragment loads below are 2-way bank conflicted, which
// costs far less.)
//
// K order inside an MMA: a dot product may sum its terms in any order, so
// the 16 code bytes of one MMA step are chosen for conflict-free 16-byte
// loads rather than in the natural order.  In step (j, s) lane (g, q) (g =
// lane / 4, q = lane % 4) supplies, for rows g and g + 8, the four code
// bytes at offset 16 (4j + q) + 4s of the row -- A elements (2q, 2q + 1) and
// (2q + 8, 2q + 9) -- and, for query g, the same four bytes of that query's
// codes as B elements; every byte of the row is used by exactly one step.
// The query fragments are converted once: kept in registers for the whole
// pass (2 registers per step: 8 m_pad / 64 in all) up to m_pad = 768, and in
// shared memory for wider rows (16 KB at m_pad = 1024).  Each warp's MMA
// chain alternates between two accumulators, halving its dependent length;
// both halves are exact integers below 2^24, and so is their sum.
//
// Epilogue: lane (g, q) holds the dot products of rows g and g + 8 with
// queries 2q and 2q + 1; it evaluates their App. A.1 intervals in the
// single-query pass's operation order (bit-identical bounds), writes them to
// the queries' arrays and keeps, per query, its slot's four largest lower
// bounds (slot = CTA x consumer warp x g) for the first working set.
#include "kernels.h"
#include "pipeline.cuh"
#include "pvs_common.cuh"

namespace pvs {
namespace {

constexpr int kGroupWarps = 8;                        // consumer warps
constexpr int kGroupHalf = 8;                         // queries of one consumer group
constexpr int kGroupThreads = (kGroupWarps + 1) * 32;
constexpr int kGroupSmemMax = 220 * 1024;             // stage ring budget

__host__ __device__ inline int group_stage_bytes(int m_pad) {
    return kTileRows * m_pad + 3 * kTileRows * 4;
}

// Four signed Int8 codes -> two f16x2 (bytes 0,1 and bytes 2,3), exact:
// x = w ^ 0x80808080 holds the codes + 128 as unsigned bytes u; the byte
// u placed under the f16 exponent byte 0x64 reads as 1024 + u, and
// subtracting 1152 leaves u - 128, the code.
__device__ __forceinline__ void codes_to_f16x2(uint32_t w, uint32_t& lo, uint32_t& hi) {
    const uint32_t x = w ^ 0x80808080u;
    const uint32_t l = __byte_perm(x, 0x64646464u, 0x4140);
    const uint32_t h = __byte_perm(x, 0x64646464u, 0x4342);
    const uint32_t bias = 0x64806480u;   // (1152, 1152) in f16
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(lo) : "r"(l), "r"(bias));
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(hi) : "r"(h), "r"(bias));
}

__device__ __forceinline__ void mma_16x8x16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                            uint32_t a3, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, "
        "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void top_insert(float (&top)[kSlotTop], float lo) {
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

// One query's side of a lane's epilogue: its index, scalars and slot list
// (its output arrays are read from the kernel's parameters when written).
struct LaneQuery {
    QueryScalars q;
    float top[kSlotTop];
    int n;
    bool on;
};

// Returns the row's upper bound (-inf for a deleted row).
__device__ __forceinline__ float eval_row(const IntervalGroupArgs& a, LaneQuery& Q, float dot_f,
                                          float sv, float vn, float en, int64_t row) {
    float lo, hi;
    interval_epilogue(__float2int_rn(dot_f), Q.q, sv, vn, en, lo, hi);
    if (!isfinite(lo) || !isfinite(hi)) set_status(a.status[Q.n], PVS_ERR_OVERFLOW);
    if (tombstoned(a.tomb, row)) lo = hi = -INFINITY;
    a.lo[Q.n][row] = lo;
    a.hi[Q.n][row] = hi;
    top_insert(Q.top, lo);
    return hi;
}

// B fragments in shared memory for rows wider than this many 64-byte groups.
constexpr int kGroupRegCPJ = 12;

__host__ __device__ inline int group_bfrag_bytes(int m_pad) {
    return m_pad / 64 > kGroupRegCPJ ? (m_pad / 16) * 32 * 8 : 0;   // steps x lanes x 8 B
}

// CPJ = m_pad / 64: groups of four 16-byte chunks per row.
template <int CPJ>
__global__ void __launch_bounds__(kGroupThreads, 1)
    interval_group_kernel(const __grid_constant__ IntervalGroupArgs a, int stages) {
    extern __shared__ __align__(128) uint8_t smem[];
    constexpr int TR = kTileRows;
    constexpr int STEPS = 4 * CPJ;                     // MMA steps per 16-row block
    constexpr bool kRegB = CPJ <= kGroupRegCPJ;        // query fragments in registers
    const int m_pad = a.m_pad;                         // == 64 * CPJ
    const int pitch = m_pad;
    const int stage_bytes = group_stage_bytes(m_pad);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)stages * stage_bytes);
    uint64_t* empty = full + stages;
    uint2* bsm = reinterpret_cast<uint2*>(empty + stages);   // [STEPS][32] when !kRegB
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t ntiles = (a.rows + TR - 1) / TR;

    if (threadIdx.x == 0) {
        for (int s = 0; s < stages; ++s) {
            mbar_init(&full[s], 1);
            // the warps that read a tile: one group, or both when split
            mbar_init(&empty[s], a.nq > kGroupHalf ? kGroupWarps : kGroupWarps / 2);
        }
        mbar_fence_init();
    }
    __syncthreads();

    if (warp == kGroupWarps) {
        // ---------------- producer ----------------
        if (lane != 0) return;
        const uint64_t pol = l2_evict_first_policy();
        int k = 0;
        bool ok = true;
        for (int64_t t = blockIdx.x; t < ntiles; t += gridDim.x, ++k) {
            const int s = k % stages;
            const uint32_t ph = (uint32_t)(k / stages) & 1u;
            if (!mbar_wait(&empty[s], ph ^ 1u, a.wait_ns)) {
                for (int g = 0; g < a.nq; ++g) set_status(a.status[g], PVS_ERR_TIMEOUT);
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
            uint8_t* pd = dst + (size_t)TR * pitch;
            bulk_g2s(pd, a.scale + r0, pb, &full[s], pol);
            bulk_g2s(pd + TR * 4, a.vnorm + r0, pb, &full[s], pol);
            bulk_g2s(pd + 2 * TR * 4, a.enorm + r0, pb, &full[s], pol);
        }
        // drain: the last copy into every used stage has landed before exit
        // (with the full wait limit, whatever a.wait_ns is)
        {
            const int issued = k;
            for (int s = 0; s < stages && s < issued; ++s) {
                const int last = issued - 1 - ((issued - 1 - s) % stages);
                if (!mbar_wait(&full[s], (uint32_t)(last / stages) & 1u) && ok)
                    for (int g = 0; g < a.nq; ++g) set_status(a.status[g], PVS_ERR_TIMEOUT);
            }
        }
        return;
    }

    // ---------------- consumers ----------------
    const bool split = a.nq > kGroupHalf;
    const int grp = warp / (kGroupWarps / 2);          // tiles k = grp, grp + 2, ... (or all)
    const int blk = warp % (kGroupWarps / 2);          // rows 16 blk .. 16 blk + 15
    const int g = lane >> 2, q = lane & 3;
    const int qb = split ? kGroupHalf * grp : 0;       // this group's first query

    // query qb + g's B fragments for every step, converted once
    uint32_t bf[kRegB ? STEPS : 1][2];
    {
        const int qg = qb + g;
        const uint32_t* zq = reinterpret_cast<const uint32_t*>(a.zq[qg < a.nq ? qg : 0]);
#pragma unroll
        for (int j = 0; j < CPJ; ++j)
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                const uint32_t w = qg < a.nq ? zq[4 * (4 * j + q) + s] : 0u;
                if constexpr (kRegB) {
                    codes_to_f16x2(w, bf[4 * j + s][0], bf[4 * j + s][1]);
                } else if (warp == 0) {
                    uint32_t b0, b1;
                    codes_to_f16x2(w, b0, b1);
                    bsm[(4 * j + s) * 32 + lane] = make_uint2(b0, b1);
                }
            }
        if constexpr (!kRegB)   // the consumer warps only (the producer never waits here)
            asm volatile("bar.sync 1, %0;" ::"n"(kGroupWarps * 32) : "memory");
    }
    LaneQuery Q[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
        Q[u].n = qb + 2 * q + u;
        Q[u].on = Q[u].n < a.nq;
        Q[u].q = Q[u].on ? *a.qs[Q[u].n] : QueryScalars{};
#pragma unroll
        for (int j = 0; j < kSlotTop; ++j) Q[u].top[j] = -INFINITY;
    }

    const int kstep = split ? 1 : 2;
    int k = split ? 0 : grp;
    for (int64_t t = blockIdx.x + (split ? 0 : (int64_t)grp * gridDim.x); t < ntiles;
         t += (int64_t)kstep * gridDim.x, k += kstep) {
        const int s = k % stages;
        const uint32_t ph = (uint32_t)(k / stages) & 1u;
        if (!mbar_wait(&full[s], ph, a.wait_ns)) {
            if (lane == 0)
                for (int m = 0; m < a.nq; ++m) set_status(a.status[m], PVS_ERR_TIMEOUT);
            break;
        }
        const uint8_t* stage = smem + (size_t)s * stage_bytes;
        const uint8_t* ra = stage + (size_t)(16 * blk + g) * pitch;
        const uint8_t* rb = ra + (size_t)8 * pitch;
        float d[2][4] = {{0.0f, 0.0f, 0.0f, 0.0f}, {0.0f, 0.0f, 0.0f, 0.0f}};
#pragma unroll
        for (int j = 0; j < CPJ; ++j) {
            const uint4 u = *reinterpret_cast<const uint4*>(ra + 16 * (4 * j + q));
            const uint4 v = *reinterpret_cast<const uint4*>(rb + 16 * (4 * j + q));
            const uint32_t uw[4] = {u.x, u.y, u.z, u.w};
            const uint32_t vw[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int s4 = 0; s4 < 4; ++s4) {
                uint32_t a0, a1, a2, a3;
                codes_to_f16x2(uw[s4], a0, a2);   // row g: elements (2q, 2q+1), (2q+8, 2q+9)
                codes_to_f16x2(vw[s4], a1, a3);   // row g + 8: the same elements
                uint32_t b0, b1;
                if constexpr (kRegB) {
                    b0 = bf[4 * j + s4][0];
                    b1 = bf[4 * j + s4][1];
                } else {
                    const uint2 b = bsm[(4 * j + s4) * 32 + lane];
                    b0 = b.x;
                    b1 = b.y;
                }
                mma_16x8x16(d[s4 & 1], a0, a1, a2, a3, b0, b1);
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) d[0][i] += d[1][i];   // exact: integers below 2^24
        // the rows' parameters, then the stage goes back to the producer
        const float* ps = reinterpret_cast<const float*>(stage + (size_t)TR * pitch);
        const int ia = 16 * blk + g, ib = ia + 8;
        const float sa = ps[ia], va = ps[TR + ia], ea = ps[2 * TR + ia];
        const float sb = ps[ib], vb = ps[TR + ib], eb = ps[2 * TR + ib];
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[s]);
        const int64_t row_a = t * TR + ia, row_b = t * TR + ib;
        float bm[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            if (!Q[u].on) continue;
            if (row_a < a.rows) bm[u] = eval_row(a, Q[u], d[0][u], sa, va, ea, row_a);
            if (row_b < a.rows)
                bm[u] = fmaxf(bm[u], eval_row(a, Q[u], d[0][2 + u], sb, vb, eb, row_b));
        }
        // the warp's 16 rows: the lanes of one query pair differ in bits 2-4
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            bm[u] = fmaxf(bm[u], __shfl_xor_sync(0xffffffffu, bm[u], 4));
            bm[u] = fmaxf(bm[u], __shfl_xor_sync(0xffffffffu, bm[u], 8));
            bm[u] = fmaxf(bm[u], __shfl_xor_sync(0xffffffffu, bm[u], 16));
        }
        if (g == 0) {
            const int64_t b = t * (TR / kBmaxRows) + blk;
#pragma unroll
            for (int u = 0; u < 2; ++u)
                if (Q[u].on && a.bmax[Q[u].n] && b * kBmaxRows < a.rows) a.bmax[Q[u].n][b] = bm[u];
        }
    }
    const size_t slot = ((size_t)blockIdx.x * kGroupWarps + warp) * 8 + g;
#pragma unroll
    for (int u = 0; u < 2; ++u) {
        float* dst = Q[u].on ? a.slot_top[Q[u].n] : nullptr;
        if (dst) {
#pragma unroll
            for (int j = 0; j < kSlotTop; ++j) dst[slot * kSlotTop + j] = Q[u].top[j];
        }
        // split: this slot scanned nothing for the other group's queries
        const int other = kGroupHalf * (1 - grp) + 2 * q + u;
        float* dso = split && other < a.nq ? a.slot_top[other] : nullptr;
        if (dso) {
#pragma unroll
            for (int j = 0; j < kSlotTop; ++j) dso[slot * kSlotTop + j] = -INFINITY;
        }
    }
}

template <int CPJ>
cudaError_t launch_group_tpl(const IntervalGroupArgs& a, int num_sms, cudaStream_t st) {
    const int stage_bytes = group_stage_bytes(a.m_pad);
    const int bbytes = group_bfrag_bytes(a.m_pad);
    int stages = (kGroupSmemMax - bbytes - 256) / stage_bytes;
    if (stages > 8) stages = 8;
    if (stages < 2) return cudaErrorInvalidValue;
    const size_t smem = (size_t)stages * stage_bytes + 2 * stages * sizeof(uint64_t) + bbytes;
    cudaError_t e = raise_smem_limit((const void*)interval_group_kernel<CPJ>, smem);
    if (e != cudaSuccess) return e;
    const int64_t ntiles = (a.rows + kTileRows - 1) / kTileRows;
    const int grid = (int)(ntiles < num_sms ? ntiles : num_sms);
    count_launches(1);
    interval_group_kernel<CPJ><<<grid, kGroupThreads, smem, st>>>(a, stages);
    return cudaGetLastError();
}

}  // namespace

bool interval_group_supported(int m_pad, int nq) {
    if (nq < 1 || nq > kGroupMax || m_pad < 64 || m_pad % 64 != 0) return false;
    if (nq > kGroupHalf && m_pad / 64 > kGroupRegCPJ) return false;   // split: fragments in registers
    switch (m_pad / 64) {
        case 1: case 2: case 3: case 4: case 6: case 8: case 12: case 16: return true;
        default: return false;
    }
}

int64_t interval_group_slots(int64_t rows, int m_pad, int nq, int num_sms,
                             int64_t* min_rows_per_slot) {
    *min_rows_per_slot = 0;
    if (rows <= 0 || !interval_group_supported(m_pad, nq)) return 0;
    const int64_t ntiles = (rows + kTileRows - 1) / kTileRows;
    const int64_t grid = ntiles < num_sms ? ntiles : num_sms;
    // CTA b scans tiles b, b + grid, ... (at least ntiles / grid of them);
    // its two warp groups take alternate ones (or, split, both take every
    // one), and only the pass's very last tile can be partial; a slot sees
    // two rows of each tile of its group
    const int64_t per_group = nq > kGroupHalf ? ntiles / grid : (ntiles / grid) / 2;
    *min_rows_per_slot = per_group > 0 ? (per_group - 1) * 2 : 0;
    return grid * kGroupWarps * 8;
}

cudaError_t launch_interval_group(const IntervalGroupArgs& a, int num_sms, cudaStream_t st) {
    if (a.rows <= 0) return cudaSuccess;
    if (!interval_group_supported(a.m_pad, a.nq)) return cudaErrorNotSupported;
    switch (a.m_pad / 64) {
        case 1: return launch_group_tpl<1>(a, num_sms, st);
        case 2: return launch_group_tpl<2>(a, num_sms, st);
        case 3: return launch_group_tpl<3>(a, num_sms, st);
        case 4: return launch_group_tpl<4>(a, num_sms, st);
        case 6: return launch_group_tpl<6>(a, num_sms, st);
        case 8: return launch_group_tpl<8>(a, num_sms, st);
        case 12: return launch_group_tpl<12>(a, num_sms, st);
        case 16: return launch_group_tpl<16>(a, num_sms, st);
        default: return cudaErrorNotSupported;
    }
}

}  // namespace pvs
