// Batched PVS interval pass on the tensor cores (Sec. 2.3.1 intervals for
// many queries at once; App. A.1 bound arithmetic).
//
// For Q <= 256 queries the exact Int8 dot products <z_q, z_v> of every corpus
// row v are one GEMM: D[128 rows x Qp] = A[128 x m] * B[Qp x m]^T per tile.
// Codes are integers in [-127, 127], exact in bf16; every product is <= 16129
// and every partial sum stays below 2^24, so fp32 accumulation is exact and
// D holds the exact integers.
//
// Persistent kernel, one CTA per SM, 18 warps:
//   warp 0     TMA producer: A tile (128 rows x 64 bf16) and B tile (Qp x 64)
//              per K chunk into a 4-stage ring, 128-byte swizzle;
//   warp 1     allocates 512 TMEM columns, issues tcgen05.mma (M=128, N=Qp,
//              K=16) x 4 per chunk, commits each stage back to the producer
//              and each finished tile to the epilogue;
//   warps 2-17 epilogue: one TMEM lane (= one corpus row) per thread; the
//              four warps that share a TMEM lane quarter split the query
//              columns (32 at a time, tcgen05.ld), so every scheduler has
//              four epilogue warps to hide load and arithmetic latency; then
//              the interval arithmetic of App. A.1 in the same operation
//              order as the single-query pass.
// Two TMEM accumulators (2 x 256 columns) let the epilogue of tile i run
// under the MMAs of tile i+1.
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

constexpr int kBM = 128;          // corpus rows per tile
constexpr int kBK = 64;           // bf16 per K chunk (128 bytes: one swizzle row)
constexpr int kMaxBN = 256;       // queries per pass
constexpr int kStages = 4;
constexpr int kStageA = kBM * kBK * 2;        // 16 KB
constexpr int kStageB = kMaxBN * kBK * 2;     // 32 KB
constexpr int kStageBytes = kStageA + kStageB;
constexpr int kEpiWarps = 16;   // 4 per TMEM lane quarter: latency hiding for the epilogue
constexpr int kBatchThreads = (2 + kEpiWarps) * 32;
constexpr uint32_t kTmemCols = 512;

struct BatchShared {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint32_t tmem_base;
    int abort;
    QueryScalars qs[kMaxBN];
    float4 flt[kMaxBN];   // filter: (s_q, rmax_q, tau_q, 0)
};

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

__global__ void __launch_bounds__(kBatchThreads, 1)
    batch_interval_kernel(const __grid_constant__ CUtensorMap tmA,
                          const __grid_constant__ CUtensorMap tmB, BatchArgs a) {
    extern __shared__ uint8_t smem_raw[];
    // stage buffers 1024-B aligned (128-byte swizzle atoms)
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* stages = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
    BatchShared& sh = *reinterpret_cast<BatchShared*>(stages + kStages * kStageBytes);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nq = a.nq, nqp = a.nq_pad;
    const int kchunks = a.m_pad / kBK;
    const int64_t ntiles_total = (a.rows + kBM - 1) / kBM;
    const int64_t niter = (ntiles_total + a.tile_stride - 1) / a.tile_stride;
    const uint32_t idesc = tc::idesc_bf16_f32(kBM, nqp);

    for (int i = threadIdx.x; i < kMaxBN; i += blockDim.x) {
        if (i < nq) {
            sh.qs[i] = a.qs[i];
            sh.flt[i] = make_float4(a.qs[i].s, a.rmax ? a.rmax[i] : INFINITY,
                                    a.tau ? a.tau[i] : -INFINITY, 0.0f);
        }
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&sh.full[s], 1);
            mbar_init(&sh.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sh.tfull[b], 1);
            mbar_init(&sh.tempty[b], kEpiWarps);
        }
        sh.abort = 0;
        mbar_fence_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(&sh.tmem_base, kTmemCols);
        tc::fence_before_sync();
    }
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = sh.tmem_base;

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            tc::prefetch_tmap(&tmA);
            tc::prefetch_tmap(&tmB);
            const uint32_t bytes = (uint32_t)kStageA + (uint32_t)nqp * kBK * 2u;
            uint32_t g = 0;
            for (int64_t i = blockIdx.x; i < niter && !abort_set(sh); i += gridDim.x) {
                const int row0 = (int)(i * a.tile_stride * kBM);
                for (int kc = 0; kc < kchunks; ++kc, ++g) {
                    const int s = g % kStages;
                    const uint32_t ph = (g / kStages) & 1u;
                    if (!mbar_wait(&sh.empty[s], ph ^ 1u)) {
                        set_status(a.status, PVS_ERR_TIMEOUT);
                        raise_abort(sh);
                        break;
                    }
                    uint8_t* sa = stages + s * kStageBytes;
                    mbar_arrive_expect_tx(&sh.full[s], bytes);
                    tc::tma_load_2d(sa, &tmA, kc * kBK, row0, &sh.full[s]);
                    tc::tma_load_2d(sa + kStageA, &tmB, kc * kBK, 0, &sh.full[s]);
                }
            }
            // drain: the last copy into every used stage has landed
            for (int s = 0; s < kStages && (uint32_t)s < g; ++s) {
                const uint32_t last = g - 1 - ((g - 1 - s) % kStages);
                if (!mbar_wait(&sh.full[s], (last / kStages) & 1u)) set_status(a.status, PVS_ERR_TIMEOUT);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            uint32_t g = 0;
            int it = 0;
            for (int64_t i = blockIdx.x; i < niter && !abort_set(sh); i += gridDim.x, ++it) {
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
                    const int s = g % kStages;
                    const uint32_t ph = (g / kStages) & 1u;
                    if (!mbar_wait(&sh.full[s], ph)) {
                        set_status(a.status, PVS_ERR_TIMEOUT);
                        raise_abort(sh);
                        break;
                    }
                    tc::fence_after_sync();
                    const uint32_t sa = smem_u32(stages + s * kStageBytes);
                    const uint32_t sb = sa + kStageA;
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k) {
                        const uint64_t ad = tc::smem_desc_sw128_kmajor(sa + k * 32);
                        const uint64_t bd = tc::smem_desc_sw128_kmajor(sb + k * 32);
                        tc::mma_bf16(d, ad, bd, idesc, (kc | k) != 0 ? 1u : 0u);
                    }
                    tc::commit(&sh.empty[s]);
                }
                if (abort_set(sh)) break;
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
        int it = 0;
        for (int64_t i = blockIdx.x; i < niter; i += gridDim.x, ++it) {
            const int b = it & 1;
            const uint32_t phb = (uint32_t)(it >> 1) & 1u;
            if (!mbar_wait(&sh.tfull[b], phb)) {
                if (lane == 0) set_status(a.status, PVS_ERR_TIMEOUT);
                raise_abort(sh);
                break;
            }
            tc::fence_after_sync();
            const int64_t row = i * a.tile_stride * kBM + r_in_tile;
            const bool inside = row < a.rows;
            bool live = inside;
            if (inside && a.tomb) live = ((__ldg(a.tomb + (row >> 5)) >> (row & 31)) & 1u) == 0;
            float sv = 0.f, vn = 0.f, en = 0.f;
            if (inside) {
                sv = __ldg(a.scale + row);
                vn = __ldg(a.vnorm + row);
                en = __ldg(a.enorm + row);
            }
            const int64_t srow = i * kBM + r_in_tile;   // row of the dump arrays
            for (int cc = cgroup; cc < nqp / 32; cc += kEpiWarps / 4) {
                uint32_t r[32];
                tc::ld_32x32b_x32(tmem + ((uint32_t)(quarter * 32) << 16) +
                                      (uint32_t)(b * kMaxBN + cc * 32),
                                  r);
                tc::wait_ld();
#pragma unroll 4
                for (int j = 0; j < 32; ++j) {
                    const int q = cc * 32 + j;
                    if (q >= nq) break;
                    const float fdot = __uint_as_float(r[j]);
                    const QueryScalars& qs = sh.qs[q];
                    if (a.mode == 0) {
                        float lo = -INFINITY, hi = -INFINITY;
                        if (live) interval_of(fdot, qs, sv, vn, en, lo, hi);
                        if (live && (!isfinite(lo) || !isfinite(hi)))
                            set_status(a.status, PVS_ERR_OVERFLOW);
                        a.dump_lo[(int64_t)q * a.dump_ld + srow] = lo;
                        if (a.dump_hi) a.dump_hi[(int64_t)q * a.dump_ld + srow] = hi;
                    } else if (live) {
                        const float4 f = sh.flt[q];
                        const float c = __fmul_rn(__fmul_rn(f.x, sv), fdot);
                        const float tau = f.z;
                        if (__fadd_ru(c, f.y) < tau) continue;   // hi < tau for sure
                        float lo, hi;
                        interval_of(fdot, qs, sv, vn, en, lo, hi);
                        if (!isfinite(lo) || !isfinite(hi)) set_status(a.status, PVS_ERR_OVERFLOW);
                        if (hi < tau) continue;
                        const unsigned int pos = atomicAdd(&a.w_len[q], 1u);
                        if (pos < (unsigned int)a.w_cap) {
                            const int64_t o = (int64_t)q * a.w_cap + pos;
                            a.w_id[o] = (int32_t)row;
                            a.w_lo[o] = lo;
                            a.w_hi[o] = hi;
                        }
                        if (lo >= tau) atomicAdd(&a.h_eff[q], 1u);
                    }
                }
            }
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.tempty[b]);
        }
    }
    __syncthreads();
    if (warp == 1) {
        tc::fence_after_sync();
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

}  // namespace

cudaError_t launch_batch_intervals(const BatchArgs& a, const uint16_t* codes_bf16,
                                   const uint16_t* qcodes_bf16, int num_sms, cudaStream_t st) {
    if (a.rows <= 0 || a.nq <= 0) return cudaSuccess;
    if (a.nq > kMaxBN || a.nq_pad % 32 != 0 || a.nq_pad < a.nq || a.nq_pad > kMaxBN ||
        a.m_pad % kBK != 0 || a.tile_stride < 1)
        return cudaErrorInvalidValue;
    CUtensorMap ta, tb;
    if (!make_map(&ta, codes_bf16, (uint64_t)a.rows, (uint64_t)a.m_pad, kBM) ||
        !make_map(&tb, qcodes_bf16, (uint64_t)a.nq_pad, (uint64_t)a.m_pad, (uint32_t)a.nq_pad))
        return cudaErrorInvalidValue;
    const size_t smem = 1024 + (size_t)kStages * kStageBytes + sizeof(BatchShared);
    cudaError_t e = cudaFuncSetAttribute(batch_interval_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t ntiles = (a.rows + kBM - 1) / kBM;
    const int64_t niter = (ntiles + a.tile_stride - 1) / a.tile_stride;
    const int grid = (int)(niter < num_sms ? niter : num_sms);
    count_launches(1);
    batch_interval_kernel<<<grid, kBatchThreads, smem, st>>>(ta, tb, a);
    return cudaGetLastError();
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
