// Batched PVS interval pass on the tensor cores (Sec. 2.3.1 intervals for
// many queries at once; App. A.1 bound arithmetic).
//
// For Q <= 256 queries the exact Int8 dot products <z_q, z_v> of every corpus
// row v are one GEMM: D[rows x Qp] = A[rows x m] * B[Qp x m]^T.  Codes are
// integers in [-127, 127], exact in bf16; every product is <= 16129 and every
// partial sum stays below 2^24, so fp32 accumulation is exact and D holds the
// exact integers.
//
// Persistent kernel, CTA pairs (a cluster of two CTAs on the two SMs of a TPC)
// with one CTA per SM, 18 warps per CTA.  A pair computes 256 rows x Qp per
// tile slot with tcgen05.mma.cta_group::2 (M = 256): each CTA holds its own
// 128 rows of A and HALF of the query chunk (Qp/2 rows of B), so every SM
// takes in 32 KB per K chunk instead of the 48 KB a lone CTA needs (A 16 KB +
// all of B 32 KB), and six stages fit where four did.
//   warp 0     TMA producer (both CTAs): its A tile (128 rows x 64 bf16) and
//              its half of the B tile (Qp/2 x 64) per K chunk into a 6-stage
//              ring, 128-byte swizzle; the bytes of BOTH CTAs are counted on
//              the even CTA's full barrier;
//   warp 1     allocates 512 TMEM columns in both CTAs; in the even CTA one
//              thread issues the pair's MMAs (M=256, N=Qp, K=16) x 4 per chunk
//              and commits each stage back to both producers and each finished
//              tile to both epilogues;
//   warps 2-17 epilogue (both CTAs): one TMEM lane (= one corpus row) per
//              thread; the four warps that share a TMEM lane quarter split
//              the query columns (32 at a time, tcgen05.ld); then the interval
//              arithmetic of App. A.1 in the same operation order as the
//              single-query pass.  Both CTAs' epilogues release an
//              accumulator on the even CTA's barrier.
// Two TMEM accumulators (2 x 256 columns) let the epilogue of tile i run
// under the MMAs of tile i+1.  Where no CTA pair can be scheduled the same
// kernel runs one CTA per tile (M = 128, whole B chunk per CTA, 4 stages).
//
// Modes:
//   dump    every sampled tile writes lo/hi of all (row, query) pairs; used to
//           pick per-query thresholds from a sample of rows and by tests;
//   filter  rows whose interval upper bound reaches the query's threshold
//           tau_q are appended to that query's working set; rows whose lower
//           bound reaches tau_q are counted (they fix the horizon).  A cheap
//           upper bound c + rmax_q < tau_q rejects most pairs before the full
//           interval is computed.
#include <cuda.h>
#include <mutex>

#include "kernels.h"
#include "pvs_common.cuh"
#include "tc.cuh"

namespace pvs {

constexpr int kBM = 128;          // corpus rows per tile and CTA
constexpr int kBK = 64;           // bf16 per K chunk (128 bytes: one swizzle row)
constexpr int kMaxBN = 256;       // queries per pass
constexpr int kStageA = kBM * kBK * 2;        // 16 KB
constexpr int kEpiWarps = 16;   // 4 per TMEM lane quarter: latency hiding for the epilogue
constexpr int kBatchThreads = (2 + kEpiWarps) * 32;
constexpr uint32_t kTmemCols = 512;
constexpr int kMaxStages = 6;

// Ring geometry for kCta CTAs per tile slot (1: lone CTA, 2: CTA pair).
template <int kCta> struct Ring {
    static constexpr int kStageB = kMaxBN / kCta * kBK * 2;   // this CTA's share of B
    static constexpr int kStageBytes = kStageA + kStageB;
    static constexpr int kStages = kCta == 2 ? 6 : 4;
};
static_assert(Ring<1>::kStages <= kMaxStages && Ring<2>::kStages <= kMaxStages, "ring");

struct BatchShared {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint32_t tmem_base;
    int abort;
    QueryScalars qs[kMaxBN];
    // filter: s_q, rmax_q (upper bound of the half-width), tau_q per query
    alignas(16) float fs[kMaxBN];
    alignas(16) float frm[kMaxBN];
    alignas(16) float ftau[kMaxBN];
};

template <int kCta>
constexpr size_t batch_smem_bytes() {
    return 1024 + (size_t)Ring<kCta>::kStages * Ring<kCta>::kStageBytes + sizeof(BatchShared);
}
static_assert(batch_smem_bytes<1>() <= 227 * 1024 && batch_smem_bytes<2>() <= 227 * 1024, "smem");

// The abort flag is written and polled by different warps.
__device__ __forceinline__ bool abort_set(BatchShared& sh) {
    return *reinterpret_cast<volatile int*>(&sh.abort) != 0;
}
__device__ __forceinline__ void raise_abort(BatchShared& sh) {
    *reinterpret_cast<volatile int*>(&sh.abort) = 1;
}

// fdot: the exact dot product as the fp32 accumulator holds it (an integer
// below 2^24, so it equals the float conversion of the int32 dot product).
__device__ __forceinline__ void interval_of(float fdot, const QueryScalars& q, float sv, float vn,
                                            float en, float& lo, float& hi) {
    const float c = __fmul_rn(__fmul_rn(q.s, sv), fdot);
    const float E = __fadd_ru(__fmul_ru(q.enorm, vn), __fmul_ru(q.qhat, en));
    const float G = __fmul_ru(__fadd_ru(__fadd_ru(fabsf(c), E), __fmul_ru(q.qnorm, vn)), q.gamma);
    const float r = __fadd_ru(E, G);
    lo = __fsub_rd(c, r);
    hi = __fadd_ru(c, r);
}

// Two fp32 lanes per instruction (f32x2), each lane rounded as its scalar
// counterpart.
__device__ __forceinline__ uint64_t pack2(float x, float y) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(x), "f"(y));
    return r;
}
__device__ __forceinline__ void unpack2(uint64_t v, float& x, float& y) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(x), "=f"(y) : "l"(v));
}
__device__ __forceinline__ uint64_t mul2_rn(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t add2_ru(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rp.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

// kCta = 2: the two CTAs of each cluster form a pair (cluster rank 0 is the
// even CTA that issues the MMAs); kCta = 1: no clusters.  Every CTA of a pair
// runs the same number of tile slots; a slot past the last tile loads an
// out-of-range A box (zero fill), still supplies its half of B, and writes
// nothing.
template <int kCta>
__global__ void __launch_bounds__(kBatchThreads, 1)
    batch_interval_kernel(const __grid_constant__ CUtensorMap tmA,
                          const __grid_constant__ CUtensorMap tmB, BatchArgs a) {
    using R = Ring<kCta>;
    extern __shared__ uint8_t smem_raw[];
    // stage buffers 1024-B aligned (128-byte swizzle atoms); the layout is the
    // same in both CTAs of a pair (the pair MMA and the barriers are
    // addressed by offset)
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* stages = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
    BatchShared& sh = *reinterpret_cast<BatchShared*>(stages + R::kStages * R::kStageBytes);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nq = a.nq, nqp = a.nq_pad;
    const int kchunks = a.m_pad / kBK;
    const int64_t ntiles_total = (a.rows + kBM - 1) / kBM;
    const int64_t niter = (ntiles_total + a.tile_stride - 1) / a.tile_stride;
    const uint32_t crank = kCta == 2 ? cluster_ctarank() : 0u;
    const bool leader = crank == 0;
    const int64_t slot0 = blockIdx.x / kCta, nslots = gridDim.x / kCta;

    for (int i = threadIdx.x; i < kMaxBN; i += blockDim.x) {
        if (i < nq) {
            sh.qs[i] = a.qs[i];
            sh.fs[i] = a.qs[i].s;
            sh.frm[i] = a.rmax ? a.rmax[i] : INFINITY;
            sh.ftau[i] = a.tau ? a.tau[i] : -INFINITY;
        } else {   // padding columns: never candidates
            sh.fs[i] = 0.0f;
            sh.frm[i] = 0.0f;
            sh.ftau[i] = INFINITY;
        }
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < R::kStages; ++s) {
            mbar_init(&sh.full[s], 1);
            mbar_init(&sh.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sh.tfull[b], 1);
            mbar_init(&sh.tempty[b], kCta * kEpiWarps);   // both CTAs' epilogue warps
        }
        sh.abort = 0;
        mbar_fence_init();
    }
    if (warp == 1) {
        if (kCta == 2)
            tc::tmem_alloc_pair(&sh.tmem_base, kTmemCols);
        else
            tc::tmem_alloc(&sh.tmem_base, kTmemCols);
        tc::fence_before_sync();
    }
    __syncthreads();
    if (kCta == 2) cluster_barrier();   // both CTAs' barriers and TMEM are ready
    tc::fence_after_sync();
    const uint32_t tmem = sh.tmem_base;

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            tc::prefetch_tmap(&tmA);
            tc::prefetch_tmap(&tmB);
            // the pair's bytes per stage, all counted on the even CTA's barrier
            const uint32_t bytes = (uint32_t)kStageA * kCta + (uint32_t)nqp * kBK * 2u;
            const int bhalf = nqp / kCta;   // query rows this CTA supplies
            uint32_t g = 0;
            for (int64_t t = slot0; t * kCta < niter && !abort_set(sh); t += nslots) {
                const int64_t i = t * kCta + crank;
                int64_t r0 = i * a.tile_stride * kBM;
                if (r0 > a.rows) r0 = a.rows;   // a slot past the end: all rows out of range
                const int row0 = (int)r0;
                for (int kc = 0; kc < kchunks; ++kc, ++g) {
                    const int s = g % R::kStages;
                    const uint32_t ph = (g / R::kStages) & 1u;
                    if (!mbar_wait(&sh.empty[s], ph ^ 1u)) {
                        set_status(a.status, PVS_ERR_TIMEOUT);
                        raise_abort(sh);
                        break;
                    }
                    uint8_t* sa = stages + s * R::kStageBytes;
                    if (kCta == 2) {
                        if (leader) mbar_arrive_expect_tx(&sh.full[s], bytes);
                        const uint32_t fb = cluster_map(&sh.full[s], 0);
                        tc::tma_load_2d_pair(sa, &tmA, kc * kBK, row0, fb);
                        tc::tma_load_2d_pair(sa + kStageA, &tmB, kc * kBK, (int)crank * bhalf, fb);
                    } else {
                        mbar_arrive_expect_tx(&sh.full[s], bytes);
                        tc::tma_load_2d(sa, &tmA, kc * kBK, row0, &sh.full[s]);
                        tc::tma_load_2d(sa + kStageA, &tmB, kc * kBK, 0, &sh.full[s]);
                    }
                }
            }
            // drain: the MMAs have consumed the last fill of every used stage,
            // so no copy into this CTA and no commit to its barriers is still
            // in flight
            for (int s = 0; s < R::kStages && (uint32_t)s < g; ++s) {
                const uint32_t last = g - 1 - ((g - 1 - s) % R::kStages);
                if (!mbar_wait(&sh.empty[s], (last / R::kStages) & 1u))
                    set_status(a.status, PVS_ERR_TIMEOUT);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer (the even CTA of a pair) ----------------
        if (lane == 0 && leader) {
            const uint32_t idesc = tc::idesc_bf16_f32(kBM * kCta, nqp);
            uint32_t g = 0;
            int it = 0;
            for (int64_t t = slot0; t * kCta < niter && !abort_set(sh); t += nslots, ++it) {
                const int b = it & 1;
                const uint32_t phb = (uint32_t)(it >> 1) & 1u;
                if (!mbar_wait(&sh.tempty[b], phb ^ 1u)) {
                    set_status(a.status, PVS_ERR_TIMEOUT);
                    raise_abort(sh);
                    break;
                }
                tc::fence_after_sync();
                const uint32_t d = tmem + (uint32_t)(b * kMaxBN);
                for (int kc = 0; kc < kchunks; ++kc, ++g) {
                    const int s = g % R::kStages;
                    const uint32_t ph = (g / R::kStages) & 1u;
                    if (!mbar_wait(&sh.full[s], ph)) {
                        set_status(a.status, PVS_ERR_TIMEOUT);
                        raise_abort(sh);
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t sa = smem_u32(stages + s * R::kStageBytes);
                    const uint32_t sb = sa + kStageA;
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k) {
                        const uint64_t ad = tc::smem_desc_sw128_kmajor(sa + k * 32);
                        const uint64_t bd = tc::smem_desc_sw128_kmajor(sb + k * 32);
                        if (kCta == 2)
                            tc::mma_bf16_pair(d, ad, bd, idesc, (kc | k) != 0 ? 1u : 0u);
                        else
                            tc::mma_bf16(d, ad, bd, idesc, (kc | k) != 0 ? 1u : 0u);
                    }
                    if (kCta == 2)
                        tc::commit_pair(&sh.empty[s]);   // the stage is free in both CTAs
                    else
                        tc::commit(&sh.empty[s]);
                }
                if (abort_set(sh)) break;
                if (kCta == 2)
                    tc::commit_pair(&sh.tfull[b]);
                else
                    tc::commit(&sh.tfull[b]);
            }
            // every MMA issued has completed before TMEM is released: wait for
            // the last tile's commit (the epilogue also waits on it)
            if (it > 0) {
                const int lb = (it - 1) & 1;
                if (!mbar_wait(&sh.tfull[lb], (uint32_t)((it - 1) >> 1) & 1u))
                    set_status(a.status, PVS_ERR_TIMEOUT);
            }
        }
    } else {
        // ---------------- epilogue ----------------
        const int quarter = warp & 3;               // TMEM lanes 32*quarter ..
        const int cgroup = (warp - 2) >> 2;         // this warp's share of the 32-column chunks
        const int r_in_tile = quarter * 32 + lane;
        const uint32_t lanemask_lt = (1u << lane) - 1u;
        const uint32_t tempty_at[2] = {kCta == 2 ? cluster_map(&sh.tempty[0], 0) : 0u,
                                       kCta == 2 ? cluster_map(&sh.tempty[1], 0) : 0u};
        // this thread's row parameters, loaded one tile slot ahead so that the
        // loads are in flight while the previous tile is processed
        float sv, vn, en;
        uint32_t tw;    // tombstone word of the row
        bool inside;
        auto fetch = [&](int64_t tt, float& psv, float& pvn, float& pen, uint32_t& ptw,
                         bool& pin) {
            const int64_t ii = tt * kCta + crank;
            const int64_t rw = ii * a.tile_stride * kBM + r_in_tile;
            pin = ii < niter && rw < a.rows;
            psv = pvn = pen = 0.f;
            ptw = 0u;
            if (pin) {
                psv = __ldg(a.scale + rw);
                pvn = __ldg(a.vnorm + rw);
                pen = __ldg(a.enorm + rw);
                if (a.tomb) ptw = __ldg(a.tomb + (rw >> 5));
            }
        };
        fetch(slot0, sv, vn, en, tw, inside);
        int it = 0;
        for (int64_t t = slot0; t * kCta < niter; t += nslots, ++it) {
            float nsv, nvn, nen;
            uint32_t ntw;
            bool nin;
            fetch(t + nslots, nsv, nvn, nen, ntw, nin);
            const int64_t i = t * kCta + crank;
            const int b = it & 1;
            const uint32_t phb = (uint32_t)(it >> 1) & 1u;
            if (!mbar_wait(&sh.tfull[b], phb)) {
                if (lane == 0) set_status(a.status, PVS_ERR_TIMEOUT);
                raise_abort(sh);
                break;
            }
            tc::fence_after_sync();
            const bool real = i < niter;
            const int64_t row = i * a.tile_stride * kBM + r_in_tile;
            const bool live = inside && ((tw >> (row & 31)) & 1u) == 0;
            const int64_t srow = i * kBM + r_in_tile;   // row of the dump arrays
            const uint32_t tcol = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(b * kMaxBN);
            for (int cc = cgroup; real && cc < nqp / 32; cc += kEpiWarps / 4) {
                if (a.mode == 0) {
                    // 32 query columns, read from TMEM 8 at a time
                    for (int g = 0; g < 4; ++g) {
                        uint32_t r[8];
                        tc::ld_32x32b_x8(tcol + (uint32_t)(cc * 32 + g * 8), r);
                        tc::wait_ld();
#pragma unroll
                        for (int k = 0; k < 8; ++k) {
                            const int q = cc * 32 + g * 8 + k;
                            if (q >= nq) continue;
                            float lo = -INFINITY, hi = -INFINITY;
                            if (live) interval_of(__uint_as_float(r[k]), sh.qs[q], sv, vn, en, lo, hi);
                            if (live && (!isfinite(lo) || !isfinite(hi)))
                                set_status(a.status, PVS_ERR_OVERFLOW);
                            a.dump_lo[(int64_t)q * a.dump_ld + srow] = lo;
                            if (a.dump_hi) a.dump_hi[(int64_t)q * a.dump_ld + srow] = hi;
                        }
                    }
                    continue;
                }
                // filter, step 1: which of the 32 queries keep this row (bit
                // k of pmask); rows whose lower bound reaches tau are counted
                // at once (no result is waited for).  A branch-free test
                // RU(c + rmax_q) >= tau_q marks the candidates (every other
                // pair has hi < tau for sure), two queries per f32x2
                // instruction with the roundings of c in the interval; only
                // the candidates get the full interval.
                uint32_t cand = 0;
                {
                    uint32_t r[32];
                    tc::ld_32x32b_x32(tcol + (uint32_t)(cc * 32), r);
                    tc::wait_ld();
                    const uint64_t sv2 = pack2(sv, sv);
#pragma unroll
                    for (int k = 0; k < 32; k += 4) {
                        const int q = cc * 32 + k;
                        const float4 s4 = *reinterpret_cast<const float4*>(&sh.fs[q]);
                        const float4 m4 = *reinterpret_cast<const float4*>(&sh.frm[q]);
                        const float4 t4 = *reinterpret_cast<const float4*>(&sh.ftau[q]);
                        const uint64_t c01 = mul2_rn(mul2_rn(pack2(s4.x, s4.y), sv2),
                                                     pack2(__uint_as_float(r[k]),
                                                           __uint_as_float(r[k + 1])));
                        const uint64_t c23 = mul2_rn(mul2_rn(pack2(s4.z, s4.w), sv2),
                                                     pack2(__uint_as_float(r[k + 2]),
                                                           __uint_as_float(r[k + 3])));
                        float u0, u1, u2, u3;
                        unpack2(add2_ru(c01, pack2(m4.x, m4.y)), u0, u1);
                        unpack2(add2_ru(c23, pack2(m4.z, m4.w)), u2, u3);
                        cand |= ((uint32_t)!(u0 < t4.x) << k) | ((uint32_t)!(u1 < t4.y) << (k + 1)) |
                                ((uint32_t)!(u2 < t4.z) << (k + 2)) |
                                ((uint32_t)!(u3 < t4.w) << (k + 3));
                    }
                }
                if (!live) cand = 0;
                uint32_t pmask = 0;
                uint32_t rest = __reduce_or_sync(0xffffffffu, cand);
                while (rest != 0) {   // the same for the whole warp; rare
                    const int k = __ffs(rest) - 1;
                    rest &= rest - 1u;
                    const uint32_t v = tc::ld_32x32b_x1(tcol + (uint32_t)(cc * 32 + k));
                    tc::wait_ld();
                    const int q = cc * 32 + k;
                    if (!((cand >> k) & 1u) || q >= nq) continue;
                    const float tau = sh.ftau[q];
                    float lo, hi;
                    interval_of(__uint_as_float(v), sh.qs[q], sv, vn, en, lo, hi);
                    if (!isfinite(lo) || !isfinite(hi)) set_status(a.status, PVS_ERR_OVERFLOW);
                    if (hi < tau) continue;
                    pmask |= 1u << k;
                    if (lo >= tau) atomicAdd(&a.h_eff[q], 1u);
                }
                // step 2: lane j reserves room for every row of the warp that
                // query cc*32+j keeps (one atomic round trip for the chunk)
                if (!__any_sync(0xffffffffu, pmask != 0)) continue;
                uint32_t my_keep = 0;
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    const uint32_t bj = __ballot_sync(0xffffffffu, (pmask >> j) & 1u);
                    if (lane == j) my_keep = bj;
                }
                unsigned int base = 0;
                if (my_keep != 0)
                    base = atomicAdd(&a.w_len[cc * 32 + lane], (unsigned int)__popc(my_keep));
                // step 3: every kept row is written at its reserved position
                // (its dot product read again from TMEM)
                uint32_t kept = __ballot_sync(0xffffffffu, my_keep != 0);
                while (kept != 0) {   // the same for the whole warp
                    const int j = __ffs(kept) - 1;
                    kept &= kept - 1u;
                    const uint32_t bj = __shfl_sync(0xffffffffu, my_keep, j);
                    const unsigned int b0 = __shfl_sync(0xffffffffu, base, j);
                    const uint32_t v = tc::ld_32x32b_x1(tcol + (uint32_t)(cc * 32 + j));
                    tc::wait_ld();
                    if ((pmask >> j) & 1u) {
                        const int q = cc * 32 + j;
                        float lo, hi;
                        interval_of(__uint_as_float(v), sh.qs[q], sv, vn, en, lo, hi);
                        const unsigned int pos = b0 + (unsigned int)__popc(bj & lanemask_lt);
                        if (pos < (unsigned int)a.w_cap) {
                            const int64_t o = (int64_t)q * a.w_cap + pos;
                            a.w_id[o] = (int32_t)row;
                            a.w_lo[o] = lo;
                            a.w_hi[o] = hi;
                        }
                    }
                }
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) {
                if (kCta == 2)
                    mbar_arrive_remote(tempty_at[b]);   // the even CTA's barrier (or its own)
                else
                    mbar_arrive(&sh.tempty[b]);
            }
            sv = nsv;
            vn = nvn;
            en = nen;
            tw = ntw;
            inside = nin;
        }
    }
    __syncthreads();
    if (kCta == 2) cluster_barrier();   // no CTA leaves while its peer may still address it
    if (warp == 1) {
        tc::fence_after_sync();
        if (kCta == 2)
            tc::tmem_dealloc_pair(tmem, kTmemCols);
        else
            tc::tmem_dealloc(tmem, kTmemCols);
    }
}

// ---- host side ---------------------------------------------------------------
namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static std::once_flag once;
    static EncodeTiledFn fn = nullptr;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
        else
            cudaGetLastError();
    });
    return fn;
}

// bf16 matrix [rows][cols] (row stride cols), box = [64 cols x box_rows], 128B swizzle.
bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}


cudaLaunchConfig_t pair_config(int grid, cudaStream_t st, cudaLaunchAttribute* attr) {
    cudaLaunchConfig_t cfg{};
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kBatchThreads);
    cfg.dynamicSmemBytes = batch_smem_bytes<2>();
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cfg;
}

// CTA pairs that run at once on the current device (0: pairs unavailable).
// The kernels' shared-memory limits are raised on the way.
int pairs_on_device(int num_sms) {
    static std::mutex mu;
    static int pairs[64];
    static bool known[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return 0;
    }
    std::lock_guard<std::mutex> lock(mu);
    if (!known[dev]) {
        int n = 0;
        if (cudaFuncSetAttribute(batch_interval_kernel<1>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)batch_smem_bytes<1>()) != cudaSuccess ||
            cudaFuncSetAttribute(batch_interval_kernel<2>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)batch_smem_bytes<2>()) != cudaSuccess) {
            cudaGetLastError();
        } else {
            cudaLaunchAttribute attr[1];
            const cudaLaunchConfig_t cfg = pair_config(2 * num_sms, nullptr, attr);
            if (cudaOccupancyMaxActiveClusters(&n, batch_interval_kernel<2>, &cfg) != cudaSuccess) {
                cudaGetLastError();
                n = 0;
            }
        }
        pairs[dev] = n;
        known[dev] = true;
    }
    return pairs[dev];
}

}  // namespace

cudaError_t launch_batch_intervals(const BatchArgs& a, const uint16_t* codes_bf16,
                                   const uint16_t* qcodes_bf16, int num_sms, cudaStream_t st) {
    if (a.rows <= 0 || a.nq <= 0) return cudaSuccess;
    if (a.nq > kMaxBN || a.nq_pad % 32 != 0 || a.nq_pad < a.nq || a.nq_pad > kMaxBN ||
        a.m_pad % kBK != 0 || a.tile_stride < 1)
        return cudaErrorInvalidValue;
    const int pairs = pairs_on_device(num_sms);
    const int cta = pairs > 0 ? 2 : 1;
    // B boxes: the whole query chunk (lone CTA) or half of it (pair); Qp/2 is
    // a multiple of 16 rows, so each half starts on a 1024-B swizzle atom
    CUtensorMap ta, tb;
    if (!make_map(&ta, codes_bf16, (uint64_t)a.rows, (uint64_t)a.m_pad, kBM) ||
        !make_map(&tb, qcodes_bf16, (uint64_t)a.nq_pad, (uint64_t)a.m_pad,
                  (uint32_t)(a.nq_pad / cta)))
        return cudaErrorInvalidValue;
    const int64_t ntiles = (a.rows + kBM - 1) / kBM;
    const int64_t niter = (ntiles + a.tile_stride - 1) / a.tile_stride;
    const int64_t slots = (niter + cta - 1) / cta;
    count_launches(1);
    if (cta == 1) {
        const int grid = (int)(slots < num_sms ? slots : num_sms);
        batch_interval_kernel<1><<<grid, kBatchThreads, batch_smem_bytes<1>(), st>>>(ta, tb, a);
        return cudaGetLastError();
    }
    const int grid = 2 * (int)(slots < pairs ? slots : pairs);
    cudaLaunchAttribute attr[1];
    const cudaLaunchConfig_t cfg = pair_config(grid, st, attr);
    return cudaLaunchKernelEx(&cfg, batch_interval_kernel<2>, ta, tb, a);
}

// bf16 copy of int8 codes (exact: |z| <= 127).
__global__ void codes_to_bf16_kernel(const int8_t* __restrict__ src, uint16_t* __restrict__ dst,
                                     int64_t count) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count; i += stride) {
        const float f = (float)src[i];
        dst[i] = (uint16_t)(__float_as_uint(f) >> 16);   // exact: at most 8 significant bits
    }
}

cudaError_t launch_codes_to_bf16(const int8_t* src, uint16_t* dst, int64_t count,
                                 cudaStream_t st) {
    if (count <= 0) return cudaSuccess;
    int64_t blocks = (count + 255) / 256;
    if (blocks > 152 * 32) blocks = 152 * 32;
    count_launches(1);
    codes_to_bf16_kernel<<<(unsigned)blocks, 256, 0, st>>>(src, dst, count);
    return cudaGetLastError();
}

}  // namespace pvs
