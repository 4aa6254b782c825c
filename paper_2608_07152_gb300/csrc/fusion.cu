// Complete-list weighted RRF on the device: the finishes of EAHR's adaptive
// policy when both ranked lists would have to be read deep (arXiv 2608.07152,
// Sec. 2.1 defines T*_K over the complete lists; Sec. 2.2's last paragraph
// notes that when early determination is impossible, fusing the complete
// lists gives the same result).
//
// fuse_complete, one request, on the dense cursor's stream:
//   1. the complete dense ranking: the authoritative score of every visible
//      row (the exhaustive scanning generator's kernel) and one sort by
//      (score desc, id asc); rank_d[x] = position + 1;
//   2. the caller's sparse list, copied to the device on a second stream
//      while step 1 runs: rank_s[x] = position + 1, each id checked (inside
//      the snapshot, visible, not repeated);
//   3. a 64-bit key per visible item: the binary32 value of its fused score
//      F = g_d(rank_d) + g_s(rank_s), computed in binary64 and rounded to
//      nearest (monotone in F), above the complement of its id; one sort;
//   4. on the host, the items whose binary32 value is at least the one just
//      below the K-th key's: every item of T*_K is among them (the binary64
//      error of F is far below a binary32 step), and the caller orders them
//      with exact rational arithmetic.
//
// rank_queries, the cheaper finish: the exact ranks of a few items only, in
// the list they have not been read from.
//   dense  the item's authoritative score s_x fixes its key (s_x, x); its
//          rank is one plus the number of visible rows whose key is larger.
//          Every row's interval [lo, hi] (App. A.1) decides that comparison
//          unless s_x lies inside it; only such rows are scored exactly.
//          Rows the cursor has delivered (bounds set to -inf) rank before
//          every item not yet delivered.  One pass over the bounds counts
//          for all items at once: a row adds one to the items whose keys
//          are below its own, a prefix of the items' sorted keys;
//   sparse one scatter of the host list (as step 2 above), read at the
//          items' ids.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <vector>

#include "exact_dot.cuh"
#include "kernels.h"
#include "pvs_common.cuh"
#include "runtime.h"

namespace pvs {
namespace {

__global__ void list_rank_kernel(const int64_t* __restrict__ ids, int64_t n, int64_t rows,
                                 const uint32_t* __restrict__ tomb, int32_t* rank_of,
                                 int* status) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const int64_t x = ids[i];
        if (x < 0 || x >= rows || tombstoned(tomb, x)) {
            set_status(status, PVS_ERR_INVALID);
            continue;
        }
        if (atomicExch(&rank_of[x], (int32_t)(i + 1)) != 0) set_status(status, PVS_ERR_INVALID);
    }
}

__global__ void dense_rank_kernel(const uint64_t* __restrict__ keys, int64_t visible,
                                  int32_t* rank_of) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < visible; i += stride)
        rank_of[rank_key_id(keys[i])] = (int32_t)(i + 1);
}

__global__ void fused_key_kernel(const int32_t* __restrict__ rd, const int32_t* __restrict__ rs,
                                 int64_t rows, const uint32_t* __restrict__ tomb, FuseWeights w,
                                 uint64_t* keys) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < rows; x += stride) {
        double F = 0.0;
        const int32_t a = rd[x], b = rs[x];
        if (a > 0 && w.a[0] != 0.0) F += w.a[0] / (w.b[0] * (double)a + w.c[0]);
        if (b > 0 && w.a[1] != 0.0) F += w.a[1] / (w.b[1] * (double)b + w.c[1]);
        uint64_t key = 0;
        if (F > 0.0 && !tombstoned(tomb, x))
            key = ((uint64_t)__float_as_uint(__double2float_rn(F)) << 32) |
                  (uint64_t)(0xffffffffu - (uint32_t)x);
        keys[x] = key;
    }
}

__global__ void top_entries_kernel(const uint64_t* __restrict__ keys, int64_t m,
                                   const int32_t* __restrict__ rd,
                                   const int32_t* __restrict__ rs, FusedCand* out) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < m; i += stride) {
        const uint64_t k = keys[i];
        FusedCand e;
        e.fbits = (uint32_t)(k >> 32);
        e.id = k ? (int32_t)(0xffffffffu - (uint32_t)(k & 0xffffffffu)) : -1;
        e.rd = k ? rd[e.id] : 0;
        e.rs = k ? rs[e.id] : 0;
        out[i] = e;
    }
}

int grid_of(int64_t n) {
    const int64_t g = (n + 255) / 256;
    return (int)std::max<int64_t>(1, std::min<int64_t>(g, 152 * 8));
}

// The queried items' keys (score, id) in ascending order, in one CTA:
// keys[i] = rank_key(score of ids[i], ids[i]), bitonic sort in shared memory.
__global__ void __launch_bounds__(kRankQueryMax) query_keys_kernel(const int64_t* __restrict__ ids,
                                                                   const float* __restrict__ scores,
                                                                   int n, uint64_t* keys,
                                                                   int* status) {
    __shared__ uint64_t sk[kRankQueryMax];
    int pow2 = 1;
    while (pow2 < n) pow2 <<= 1;
    for (int i = threadIdx.x; i < pow2; i += blockDim.x) {
        uint64_t k = ~0ull;   // padding sorts last
        if (i < n) {
            const float s = scores[i];
            if (!isfinite(s)) set_status(status, PVS_ERR_OVERFLOW);
            k = rank_key(s, (uint32_t)ids[i]);
        }
        sk[i] = k;
    }
    __syncthreads();
    for (int size = 2; size <= pow2; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = threadIdx.x; i < pow2; i += blockDim.x) {
                const int j = i ^ stride;
                if (j > i) {
                    const bool up = (i & size) == 0;
                    const uint64_t a = sk[i], b = sk[j];
                    if ((a > b) == up) {
                        sk[i] = b;
                        sk[j] = a;
                    }
                }
            }
            __syncthreads();
        }
    }
    for (int i = threadIdx.x; i < n; i += blockDim.x) keys[i] = sk[i];
}

// Number of keys below x, and at most x (keys ascending).
__device__ __forceinline__ int keys_below(const uint64_t* k, int n, uint64_t x) {
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (k[mid] < x) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}
__device__ __forceinline__ int keys_at_most(const uint64_t* k, int n, uint64_t x) {
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (k[mid] <= x) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

constexpr int kCountWarps = 8;
// Rows a block classifies per step (four per lane), and the straddling rows
// it queues for the residual level (and for the fp32 rows after it), flushed
// before a tile could overflow the queue.
constexpr int kCountTile = kCountWarps * 32 * 4;
constexpr int kPlaceQueue = 2048;
static_assert(kPlaceQueue >= 2 * kCountTile, "queue");

// Pinned staging of one rank query: ids in (8 B dense, 4 B sparse), per dense
// item two 8-byte counts (plus one) and its key, per sparse item its rank,
// two status words.
constexpr size_t kRankQueryPinned = size_t(64) << 10;
static_assert((size_t)kRankQueryMax * 12 + ((size_t)kRankQueryMax + 1) * 16 +
                      (size_t)kRankQueryMax * 12 + 8 <=
                  kRankQueryPinned,
              "rank-query staging");

// fp32 inner product of q and v (m_raw floats, 16-byte aligned, zero padded)
// by one warp: each lane a chain of FMAs over its float4s, then a butterfly
// sum; every lane returns the same f and the same *err >= |f - q.v|.  Each
// product is exact inside its FMA and then takes part in at most
// n = 4 ceil(n4 / 32) + 5 roundings, so (Higham, Accuracy and Stability of
// Numerical Algorithms, Sec. 3.1 and 3.3; gamma_n = n u / (1 - n u), u = 2^-24)
//   |f - q.v| <= gamma_n S + k 2^-150,   S = sum |q_j v_j|,
// k the roundings that may fall in the subnormal range (32 n + 32 at most;
// 2^-149 per rounding below covers the growth of those terms).  S is bounded
// the same way from its own fp32 chain g:  S <= (g + k 2^-149) / (1 - gamma_n).
// Nothing here relies on a stored norm.
__device__ __forceinline__ float fast_dot_warp(const float* __restrict__ q,
                                               const float* __restrict__ v, int m_raw,
                                               float* err) {
    const int lane = threadIdx.x & 31;
    const float4* q4 = reinterpret_cast<const float4*>(q);
    const float4* v4 = reinterpret_cast<const float4*>(v);
    const int n4 = m_raw >> 2;
    constexpr int kBatch = 8;   // float4 of the row in flight per lane: one round trip
    float f = 0.0f, g = 0.0f;
#pragma unroll 1
    for (int j0 = lane; j0 < n4; j0 += 32 * kBatch) {
        float4 y[kBatch];
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
            const int j = j0 + 32 * b;
            y[b] = j < n4 ? __ldg(v4 + j) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        }
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
            const int j = j0 + 32 * b;
            if (j < n4) {
                const float4 a = q4[j];
                f = fmaf(a.x, y[b].x, f);
                g = fmaf(fabsf(a.x), fabsf(y[b].x), g);
                f = fmaf(a.y, y[b].y, f);
                g = fmaf(fabsf(a.y), fabsf(y[b].y), g);
                f = fmaf(a.z, y[b].z, f);
                g = fmaf(fabsf(a.z), fabsf(y[b].z), g);
                f = fmaf(a.w, y[b].w, f);
                g = fmaf(fabsf(a.w), fabsf(y[b].w), g);
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        f += __shfl_xor_sync(0xffffffffu, f, o);
        g += __shfl_xor_sync(0xffffffffu, g, o);
    }
    const int n = 4 * ((n4 + 31) / 32) + 5;
    const float nu = (float)n * 0x1p-24f;
    const float gamma = __fdiv_ru(nu, __fsub_rd(1.0f, nu));
    const float tiny = (float)(32 * n + 32) * 0x1p-149f;
    const float S = __fdiv_ru(__fadd_ru(g, tiny), __fsub_rd(1.0f, gamma));
    *err = __fadd_ru(__fmul_ru(gamma, S), tiny);
    return f;
}

// Upper bound of |x|, x the exact value that y = RN(x) rounds (a single
// binary32 rounding: |x - y| <= 2^-23 |y| + 2^-149 covers the relative error
// u |x| <= u (|y| + |x - y|) and the subnormal range).
__device__ __forceinline__ float abs_before_rn(float y) {
    return __fadd_ru(__fadd_ru(fabsf(y), __fmul_ru(fabsf(y), 0x1p-23f)), 0x1p-149f);
}

// Residual codes of rows [r0, r0 + n), one warp per row, in binary32 with
// directed rounding.  e_j = RN(v_j - s z_j) (one FMA; v the authoritative
// row, s and z its scale and codes), s2 = RN(max_j |e_j| / 7), z2_j =
// clip(rint(e_j / s2), -7, 7), r2_j = RN(e_j - s2 z2_j) (one FMA).  The true
// residual v_j - s z_j - s2 z2_j is at most a_j = |r2_j|^ + (|e_j|^ -
// |e_j|) in magnitude (^: the bound of abs_before_rn), so rnorm =
// RU(sqrt(sum a_j^2)) with every operation rounded up, and wnorm =
// RU(||v||^ + rnorm) bounds ||s z + s2 z2|| = ||v - r2||.  Both hold whatever
// the stored codes are.
__global__ void __launch_bounds__(256) resid_build_kernel(
    const float* __restrict__ raw, const int8_t* __restrict__ codes,
    const float* __restrict__ scale, int64_t r0, int64_t n, int m, int m_pad, int m_raw,
    uint8_t* __restrict__ resid, float4* __restrict__ rparam, int* status) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    const int nw = m_pad >> 3;   // 32-bit words of nibbles per row
    for (int64_t i = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); i < n;
         i += warps) {
        const int64_t row = r0 + i;
        const float* v = raw + row * (int64_t)m_raw;
        const int8_t* z = codes + row * (int64_t)m_pad;
        const float s = scale[row];
        auto e_of = [&](int d) { return d < m ? fmaf(-s, (float)z[d], v[d]) : 0.0f; };
        float emax = 0.0f;
        for (int d = lane; d < m; d += kWarp) emax = fmaxf(emax, fabsf(e_of(d)));
        emax = warp_max(emax);
        float s2 = 0.0f;
        if (emax > 0.0f) {
            s2 = __fdiv_rn(emax, 7.0f);
            if (s2 == 0.0f) s2 = __uint_as_float(1u);   // 2^-149
        }
        if (!isfinite(s2)) s2 = 0.0f;
        auto z2_of = [&](float e) {
            if (s2 == 0.0f) return 0;
            return (int)fminf(fmaxf(rintf(__fdiv_rn(e, s2)), -7.0f), 7.0f);
        };
        float ss = 0.0f, sv = 0.0f;   // sums of squares, rounded up
        for (int t = lane; t < nw; t += kWarp) {
            uint32_t w = 0;
            for (int k = 0; k < 8; ++k) {
                const int d = 8 * t + k;
                const float e = e_of(d);
                const int c = z2_of(e);
                w |= (uint32_t)(c + 8) << (8 * (k >> 1) + 4 * (k & 1));
                if (d < m) {
                    const float r = fmaf(-s2, (float)c, e);
                    const float a = __fadd_ru(abs_before_rn(r),
                                              __fsub_ru(abs_before_rn(e), fabsf(e)));
                    ss = __fadd_ru(ss, __fmul_ru(a, a));
                    sv = __fadd_ru(sv, __fmul_ru(v[d], v[d]));
                }
            }
            reinterpret_cast<uint32_t*>(resid + row * (int64_t)(m_pad >> 1))[t] = w;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            ss = __fadd_ru(ss, __shfl_xor_sync(0xffffffffu, ss, o));
            sv = __fadd_ru(sv, __shfl_xor_sync(0xffffffffu, sv, o));
        }
        if (lane == 0) {
            const float nb = __fsqrt_ru(ss);
            const float wb = __fadd_ru(__fsqrt_ru(sv), nb);
            if (!isfinite(wb)) set_status(status, PVS_ERR_OVERFLOW);
            rparam[row] = make_float4(s, s2, nb, wb);
        }
    }
}

// Rows of at most this many padded dimensions get residual codes (the
// query's 16-bit codes then fit in 16 KB of shared memory).
constexpr int kResidMaxPad = 4096;

// The residual codes of every row of the index, extended on stream st; st
// then waits for the last build, whichever stream ran it.
pvs_status ensure_resid(pvs_index* x, cudaStream_t st, int* status) {
    std::lock_guard<std::mutex> lock(x->resid_mutex);
    if (!x->resid) {
        const size_t cap = (size_t)std::max<int64_t>(x->cap, 1);
        if (cudaMalloc(reinterpret_cast<void**>(&x->resid), cap * (size_t)(x->m_pad >> 1)) !=
                cudaSuccess ||
            cudaMalloc(reinterpret_cast<void**>(&x->rparam), cap * sizeof(float4)) !=
                cudaSuccess) {
            const cudaError_t e = cudaGetLastError();
            cudaFree(x->resid), cudaFree(x->rparam);
            x->resid = nullptr, x->rparam = nullptr;
            return e == cudaErrorMemoryAllocation ? PVS_ERR_OOM : PVS_ERR_CUDA;
        }
        x->resid_rows = 0;
    }
    if (!x->resid_ready &&
        cudaEventCreateWithFlags(&x->resid_ready, cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        return PVS_ERR_CUDA;
    }
    cudaError_t e = cudaSuccess;
    if (x->resid_rows < x->size) {
        const int64_t r0 = x->resid_rows, n = x->size - r0;
        count_launches(1);
        resid_build_kernel<<<(unsigned)std::min<int64_t>((n + 7) / 8, 152 * 64), 256, 0, st>>>(
            x->raw, x->codes, x->scale, r0, n, x->m, x->m_pad, x->m_raw, x->resid, x->rparam,
            status);
        e = cudaGetLastError();
        if (e == cudaSuccess) e = cudaEventRecord(x->resid_ready, st);
        if (e == cudaSuccess) x->resid_rows = x->size;
    } else {
        e = cudaStreamWaitEvent(st, x->resid_ready, 0);
    }
    if (e != cudaSuccess) {
        cudaGetLastError();
        return PVS_ERR_CUDA;
    }
    return PVS_OK;
}

// The query in integers for the residual level, computed by every block of
// a rank count into shared memory: q = s_q zq + e_q with |zq_j| <= Q (Q
// keeps every integer dot product below 2^31), zq as 16-bit pairs twice,
// in dimension order (for the int8 codes) and in the residual codes' nibble
// order (dims 8t + 0, 2, 4, 6, 1, 3, 5, 7: the pairs (0,2) (4,6) of the low
// nibbles, (1,3) (5,7) of the high ones), each as 16-byte slots: the first
// half of every 16-dim chunk, then the second halves; eq >= ||e_q|| and
// bias = sum zq_j.
struct ResidQuery {
    float sq, eq;
    int bias;
};

// D1 = zq.z and D2 = zq.z2 over one row, exact integers, by the eight
// lanes of an aligned group (dp2a): lane sl of the group takes the 16-dim
// chunks sl, sl + 8, ..., so the group reads whole 128-byte lines of codes;
// every lane of the group returns the same sums.  Lanes whose row is not
// valid take part in the shuffles with zero sums.
__device__ __forceinline__ void resid_dots_group8(const int32_t* __restrict__ zqn,
                                                  const int32_t* __restrict__ zqp, int bias,
                                                  const int8_t* __restrict__ z,
                                                  const uint8_t* __restrict__ z2, int m_pad,
                                                  bool valid, int* D1, int* D2) {
    const int sl = threadIdx.x & 7;
    const int n16 = m_pad >> 4;   // 16 dims per chunk: 16 code bytes, 8 residual bytes
    const uint4* zc = reinterpret_cast<const uint4*>(z);
    const uint2* rc = reinterpret_cast<const uint2*>(z2);
    const int4* qn = reinterpret_cast<const int4*>(zqn);
    const int4* qp = reinterpret_cast<const int4*>(zqp);
    int acc1 = 0, acc2 = 0;
    if (valid) {
#pragma unroll 1
        for (int c0 = sl; c0 < n16; c0 += 24) {
            uint4 a[3];
            uint2 b[3];
#pragma unroll
            for (int u = 0; u < 3; ++u) {
                const int c = c0 + 8 * u;
                a[u] = c < n16 ? __ldg(zc + c) : make_uint4(0, 0, 0, 0);
                b[u] = c < n16 ? __ldg(rc + c) : make_uint2(0x88888888u, 0x88888888u);
            }
#pragma unroll
            for (int u = 0; u < 3; ++u) {
                const int c = c0 + 8 * u;
                if (c >= n16) break;
                const int4 n0 = qn[c], n1 = qn[n16 + c];
                const int4 p0 = qp[c], p1 = qp[n16 + c];
                acc1 = __dp2a_lo(n0.x, (int)a[u].x, acc1);
                acc1 = __dp2a_hi(n0.y, (int)a[u].x, acc1);
                acc1 = __dp2a_lo(n0.z, (int)a[u].y, acc1);
                acc1 = __dp2a_hi(n0.w, (int)a[u].y, acc1);
                acc1 = __dp2a_lo(n1.x, (int)a[u].z, acc1);
                acc1 = __dp2a_hi(n1.y, (int)a[u].z, acc1);
                acc1 = __dp2a_lo(n1.z, (int)a[u].w, acc1);
                acc1 = __dp2a_hi(n1.w, (int)a[u].w, acc1);
                const int l0 = (int)(b[u].x & 0x0F0F0F0Fu), h0 = (int)((b[u].x >> 4) & 0x0F0F0F0Fu);
                const int l1 = (int)(b[u].y & 0x0F0F0F0Fu), h1 = (int)((b[u].y >> 4) & 0x0F0F0F0Fu);
                acc2 = __dp2a_lo(p0.x, l0, acc2);
                acc2 = __dp2a_hi(p0.y, l0, acc2);
                acc2 = __dp2a_lo(p0.z, h0, acc2);
                acc2 = __dp2a_hi(p0.w, h0, acc2);
                acc2 = __dp2a_lo(p1.x, l1, acc2);
                acc2 = __dp2a_hi(p1.y, l1, acc2);
                acc2 = __dp2a_lo(p1.z, h1, acc2);
                acc2 = __dp2a_hi(p1.w, h1, acc2);
            }
        }
    }
#pragma unroll
    for (int o = 4; o > 0; o >>= 1) {   // within the aligned group of eight
        acc1 += __shfl_xor_sync(0xffffffffu, acc1, o);
        acc2 += __shfl_xor_sync(0xffffffffu, acc2, o);
    }
    *D1 = acc1;
    *D2 = acc2 - 8 * bias;   // nibbles hold z2 + 8
}

// The exact inner product q.v lies in [*fl, *fh], from the row's dots
// D1 = zq.z and D2 = zq.z2 and rp = (s, s2, rnorm, wnorm).  With
// w = s z + s2 z2 (so v = w + r2) and q = s_q zq + e_q:
//   q.v = s_q (s D1 + s2 D2) + e_q.w + q.r2,
// |e_q.w| <= eq wnorm, |q.r2| <= ||q|| rnorm.  The binary32 evaluation
// c = RN(s_q RN(RN(s RN(D1)) + RN(s2 RN(D2)))) has six roundings of relative
// error u = 2^-24 each, so |c - s_q (s D1 + s2 D2)| <= 8 u s_q (|s D1'| +
// |s2 D2'|) with room (' the rounded terms), plus (s_q + 1) 2^-147 for the
// subnormal range.  False when the bounds are not finite.
__device__ __forceinline__ bool resid_bounds(int D1, int D2, const float4 rp,
                                             const ResidQuery& rq, float qnorm, float* fl,
                                             float* fh) {
    const float a = __fmul_rn(rp.x, __int2float_rn(D1));
    const float b = __fmul_rn(rp.y, __int2float_rn(D2));
    const float c = __fmul_rn(rq.sq, __fadd_rn(a, b));
    float E = __fmul_ru(__fmul_ru(rq.sq, __fadd_ru(fabsf(a), fabsf(b))), 0x1p-21f);
    E = __fadd_ru(E, __fadd_ru(__fmul_ru(rq.sq, 0x1p-147f), 0x1p-147f));
    E = __fadd_ru(E, __fmul_ru(rq.eq, rp.w));
    E = __fadd_ru(E, __fmul_ru(qnorm, rp.z));
    *fl = __fsub_rd(c, E);
    *fh = __fadd_ru(c, E);
    return isfinite(*fl) && isfinite(*fh);
}

// hist[j] = number of visible rows whose key lies above exactly j of the
// queried keys (sorted ascending); the rank of the item with the j-th
// smallest key is then 1 + sum of hist[t] for t > j.  A row's key lies in
// [key(lo, y), key(hi, y)]; when no queried key falls in that range the
// count is fixed by the bounds.  Otherwise, with `exact`, the row's
// authoritative score is placed: first by the bounds of its residual codes
// (resid_dots_group8 and resid_bounds, 1.5 B per dimension; the block queues
// such rows and places them eight lanes per row), else by the fp32 dot with
// its error bound, else exactly (and it must lie in its interval, App. A.1);
// without, the row counts in hist[a] (a = the queried keys below key(lo, y):
// it is surely above those) and may lie above the keys a .. b-1 (b = the
// keys at most key(hi, y)): maybe[a] += 1, maybe[b] -= 1, so that the prefix
// sum of `maybe` at j counts the rows that may lie above the j-th key.  A
// row with hi = -inf has been delivered and lies above every queried key.
__global__ void __launch_bounds__(kCountWarps * 32, 4) rank_count_kernel(
    const float* __restrict__ lo, const float* __restrict__ hi, int64_t rows,
    const uint32_t* __restrict__ tomb, const float* __restrict__ qraw,
    const float* __restrict__ raw, int m_raw, const uint64_t* __restrict__ qkeys, int nq, int exact,
    const int8_t* __restrict__ codes, const uint8_t* __restrict__ resid,
    const float4* __restrict__ rparam, int m_pad, int qrange,
    const QueryScalars* __restrict__ qs, unsigned long long* hist, unsigned long long* maybe,
    int* status, DevCounters* ctr) {
    __shared__ uint64_t sk[kRankQueryMax];
    __shared__ unsigned int sh[kRankQueryMax + 1];
    __shared__ int sm[kRankQueryMax + 1];
    for (int i = threadIdx.x; i < nq; i += blockDim.x) sk[i] = qkeys[i];
    for (int i = threadIdx.x; i <= nq; i += blockDim.x) {
        sh[i] = 0;
        sm[i] = 0;
    }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int64_t step = (int64_t)gridDim.x * kCountTile;
    unsigned long long scored = 0, fallbacks = 0;
    // the query's integer form for the residual level (every block computes
    // the same): s_q = RN(max |q_j| / Q), zq_j = clip(rint(RN(q_j / s_q)),
    // -Q, Q), e_j = RN(q_j - s_q zq_j) (one FMA), eq = RU(sqrt(sum of the
    // bounds of |q_j - s_q zq_j| squared)) with every operation rounded up
    extern __shared__ int4 rq_smem[];
    int32_t* zqn = reinterpret_cast<int32_t*>(rq_smem);   // m_pad / 2 pairs
    int32_t* zqp = zqn + (m_pad >> 1);
    __shared__ ResidQuery srq;
    __shared__ float red_f[kCountWarps];
    __shared__ int red_i[kCountWarps];
    const bool use_resid = exact && resid != nullptr;
    float qnorm = 0.0f;
    if (use_resid) {
        const int w = threadIdx.x >> 5;
        const float Qf = (float)qrange;
        float mq = 0.0f;
        for (int j = threadIdx.x; j < m_raw; j += blockDim.x) mq = fmaxf(mq, fabsf(qraw[j]));
        mq = warp_max(mq);
        if (lane == 0) red_f[w] = mq;
        __syncthreads();
        mq = red_f[0];
        for (int i = 1; i < kCountWarps; ++i) mq = fmaxf(mq, red_f[i]);
        __syncthreads();   // red_f is written again below
        float sq = 1.0f;
        if (mq > 0.0f) {
            sq = __fdiv_rn(mq, Qf);
            if (sq == 0.0f) sq = __uint_as_float(1u);   // 2^-149
        }
        int16_t* zn16 = reinterpret_cast<int16_t*>(zqn);
        int16_t* zp16 = reinterpret_cast<int16_t*>(zqp);
        float ss = 0.0f;
        int bias = 0;
        for (int j = threadIdx.x; j < m_pad; j += blockDim.x) {
            int c = 0;
            if (j < m_raw && mq > 0.0f) {
                c = (int)fminf(fmaxf(rintf(__fdiv_rn(qraw[j], sq)), -Qf), Qf);
                const float a = abs_before_rn(fmaf(-sq, (float)c, qraw[j]));
                ss = __fadd_ru(ss, __fmul_ru(a, a));
            } else if (j < m_raw) {
                ss = __fadd_ru(ss, __fmul_ru(qraw[j], qraw[j]));
            }
            // half h of chunk j / 16 (dims 8h .. 8h + 7 of the chunk) sits at
            // 16-byte slot h * (m_pad / 16) + j / 16, so that the eight lanes
            // of a group read consecutive slots
            const int k = j & 7, slot = ((j >> 3) & 1) * (m_pad >> 4) + (j >> 4);
            zn16[slot * 8 + k] = (int16_t)c;
            zp16[slot * 8 + ((k & 1) ? 4 + (k >> 1) : (k >> 1))] = (int16_t)c;
            bias += c;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss = __fadd_ru(ss, __shfl_xor_sync(0xffffffffu, ss, o));
        bias = __reduce_add_sync(0xffffffffu, bias);
        if (lane == 0) {
            red_f[w] = ss;
            red_i[w] = bias;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            float st = 0.0f;
            int bt = 0;
            for (int i = 0; i < kCountWarps; ++i) {
                st = __fadd_ru(st, red_f[i]);
                bt += red_i[i];
            }
            srq.sq = sq;
            srq.eq = __fsqrt_ru(st);
            srq.bias = bt;
        }
        __syncthreads();
        qnorm = qs->qnorm;
    }
    const int64_t rbytes = m_pad >> 1;
    const int warp = threadIdx.x >> 5;
    // row r's bin from its fp32 row, by the whole warp: first a plain fp32
    // dot with its error bound, which places the authoritative score RN(q.v)
    // in [fl, fh] and fixes the bin unless a queried key falls in that range;
    // then the exact dot
    auto place_fp32 = [&](int64_t r, float lr, float hr) {
        float err;
        const float f = fast_dot_warp(qraw, raw + r * (int64_t)m_raw, m_raw, &err);
        int fast_bin = -1;
        if (lane == 0 && isfinite(f) && isfinite(err)) {
            // a score of zero is reported as +0, whose key is above -0's
            const float fl = __fsub_rd(f, err);
            const float fh = __fadd_ru(f, err) == 0.0f ? 0.0f : __fadd_ru(f, err);
            const int a = keys_below(sk, nq, rank_key(fl, (uint32_t)r));
            const int b = keys_at_most(sk, nq, rank_key(fh, (uint32_t)r));
            if (a == b) {
                fast_bin = a;
                if (fh < lr || fl > hr) set_status(status, PVS_ERR_INTERVAL);
                atomicAdd(&sh[a], 1u);
                ++scored;
            }
        }
        if (__shfl_sync(0xffffffffu, fast_bin, 0) >= 0) return;
        bool fb = false;
        const float s = exact_dot_warp_eft(qraw, qraw, raw + r * (int64_t)m_raw, m_raw, &fb);
        if (lane == 0) {
            if (!isfinite(s)) set_status(status, PVS_ERR_OVERFLOW);
            else if (s < lr || s > hr) set_status(status, PVS_ERR_INTERVAL);
            atomicAdd(&sh[keys_below(sk, nq, rank_key(s, (uint32_t)r))], 1u);
            ++scored;
            fallbacks += fb ? 1 : 0;
        }
    };
    // with the residual codes, the block queues its straddling rows and
    // places them eight lanes per row; the rows they leave open are queued
    // again and scored one warp per row
    __shared__ int32_t q_rows[kPlaceQueue];
    __shared__ int32_t f_rows[kPlaceQueue];
    __shared__ int q_n, f_n;
    if (threadIdx.x == 0) q_n = f_n = 0;
    __syncthreads();
    // a block tile: kCountWarps warps x 32 lanes x 4 consecutive rows, the
    // bounds read as float4 (scalars at a ragged end or unaligned buffers)
    const bool vec_ok =
        ((reinterpret_cast<uintptr_t>(lo) | reinterpret_cast<uintptr_t>(hi)) & 15) == 0;
    const unsigned int lanemask_lt = (1u << lane) - 1u;
    for (int64_t tb = (int64_t)blockIdx.x * kCountTile;; tb += step) {
        const int64_t base = tb + (int64_t)warp * 32 * 4;
        if (base < rows) {
            const int64_t y0 = base + 4 * lane;
            float lv[4] = {0.f, 0.f, 0.f, 0.f}, hv[4] = {0.f, 0.f, 0.f, 0.f};
            if (vec_ok && y0 + 3 < rows) {
                const float4 L = *reinterpret_cast<const float4*>(lo + y0);
                const float4 H = *reinterpret_cast<const float4*>(hi + y0);
                lv[0] = L.x, lv[1] = L.y, lv[2] = L.z, lv[3] = L.w;
                hv[0] = H.x, hv[1] = H.y, hv[2] = H.z, hv[3] = H.w;
            } else {
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (y0 + u < rows) {
                        lv[u] = lo[y0 + u];
                        hv[u] = hi[y0 + u];
                    }
            }
            // the four rows share one tombstone word
            const uint32_t tw = (tomb && y0 < rows) ? tomb[y0 >> 5] >> (y0 & 31) : 0u;
            unsigned int strad[4] = {0u, 0u, 0u, 0u};   // straddling lanes per row slot
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int64_t y = y0 + u;
                const float l = lv[u], h = hv[u];
                int bin = -1;   // -1: nothing to count from the bounds
                int mb = -1;    // bounds mode: the row may lie above keys bin .. mb - 1
                bool straddle = false;
                if (y < rows && !((tw >> u) & 1u)) {
                    if (h == -INFINITY) {
                        bin = nq;
                    } else {
                        const int a = keys_below(sk, nq, rank_key(l, (uint32_t)y));
                        const int b = keys_at_most(sk, nq, rank_key(h, (uint32_t)y));
                        if (a == b) {
                            bin = a;
                        } else if (exact) {
                            straddle = true;
                        } else {
                            bin = a;
                            mb = b;
                        }
                    }
                }
                // one shared-memory add per distinct bin of the warp
                const unsigned int live = __ballot_sync(0xffffffffu, bin >= 0);
                if (bin >= 0) {
                    const unsigned int same = __match_any_sync(live, bin);
                    if (lane == __ffs(same) - 1) atomicAdd(&sh[bin], (unsigned int)__popc(same));
                }
                // bounds mode: maybe[a] += 1, maybe[b] -= 1, per distinct key of the warp
                const unsigned int mlive = __ballot_sync(0xffffffffu, mb >= 0);
                if (mb >= 0) {
                    const unsigned int sa = __match_any_sync(mlive, bin);
                    if (lane == __ffs(sa) - 1) atomicAdd(&sm[bin], __popc(sa));
                    const unsigned int sb = __match_any_sync(mlive, mb);
                    if (lane == __ffs(sb) - 1) atomicAdd(&sm[mb], -__popc(sb));
                }
                const unsigned int todo = __ballot_sync(0xffffffffu, straddle);
                if (use_resid) {   // one queue reservation per warp
                    if (todo) {
                        int qb = 0;
                        if (lane == __ffs(todo) - 1) qb = atomicAdd(&q_n, __popc(todo));
                        qb = __shfl_sync(0xffffffffu, qb, __ffs(todo) - 1);
                        if (straddle) q_rows[qb + __popc(todo & lanemask_lt)] = (int32_t)y;
                    }
                } else {
                    strad[u] = todo;
                }
            }
            // without the residual codes, each straddling row from its fp32 row
#pragma unroll 1
            for (int u = 0; u < 4 && !use_resid; ++u) {
                unsigned int rest = strad[u];
                while (rest) {
                    const int src = __ffs(rest) - 1;
                    rest &= rest - 1;
                    if (rest) {   // the next row to score, into L2 while this one is scored
                        const char* nrow = reinterpret_cast<const char*>(
                            raw + (base + 4 * (__ffs(rest) - 1) + u) * (int64_t)m_raw);
                        for (int off = lane * 128; off < m_raw * 4; off += 32 * 128)
                            asm volatile("prefetch.global.L2 [%0];" ::"l"(nrow + off));
                    }
                    const int64_t r = base + 4 * src + u;
                    place_fp32(r, lo[r], hi[r]);
                }
            }
        }
        const bool last = tb + step >= rows;   // the same in every thread of the block
        if (!use_resid) {
            if (last) break;
            continue;
        }
        __syncthreads();
        const int n = q_n;
        if (n > kPlaceQueue - kCountTile || last) {
            // four rows per warp, eight lanes per row
            const int sl = lane & 7;
            for (int i0 = warp * 4; i0 < n; i0 += kCountWarps * 4) {
                const int i = i0 + (lane >> 3);
                const bool valid = i < n;
                const int64_t r = valid ? q_rows[i] : 0;
                const int inext = i + kCountWarps * 4;   // the group's next row, into L2
                if (inext < n) {
                    const int64_t pr = q_rows[inext];
                    const char* zc = reinterpret_cast<const char*>(codes + pr * (int64_t)m_pad);
                    const char* rc = reinterpret_cast<const char*>(resid + pr * rbytes);
                    for (int off = sl * 128; off < m_pad; off += 8 * 128)
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(zc + off));
                    for (int off = sl * 128; off < rbytes; off += 8 * 128)
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(rc + off));
                    if (sl == 7) asm volatile("prefetch.global.L2 [%0];" ::"l"(rparam + pr));
                }
                int D1, D2;
                resid_dots_group8(zqn, zqp, srq.bias, codes + r * (int64_t)m_pad,
                                  resid + r * rbytes, m_pad, valid, &D1, &D2);
                int open = 0;   // the row needs its fp32 row
                if (valid && sl == 0) {
                    float rl, rh;
                    bool placed = false;
                    if (resid_bounds(D1, D2, rparam[r], srq, qnorm, &rl, &rh)) {
                        // RN(q.v) lies in [rl, rh] as q.v does; a score of
                        // zero is reported as +0, whose key is above -0's
                        const float rh0 = rh == 0.0f ? 0.0f : rh;
                        const int a = keys_below(sk, nq, rank_key(rl, (uint32_t)r));
                        const int b = keys_at_most(sk, nq, rank_key(rh0, (uint32_t)r));
                        if (a == b) {
                            placed = true;
                            if (rh < lo[r] || rl > hi[r]) set_status(status, PVS_ERR_INTERVAL);
                            atomicAdd(&sh[a], 1u);
                        }
                    }
                    if (!placed) {
                        f_rows[atomicAdd(&f_n, 1)] = (int32_t)r;
                        open = 1;
                    }
                }
                if (__shfl_sync(0xffffffffu, open, lane & ~7)) {   // its fp32 row, into L2
                    const char* vr = reinterpret_cast<const char*>(raw + r * (int64_t)m_raw);
                    for (int off = sl * 128; off < m_raw * 4; off += 8 * 128)
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(vr + off));
                }
            }
            __syncthreads();
            const int nf = f_n;
            for (int i = warp; i < nf; i += kCountWarps) {
                const int64_t r = f_rows[i];
                place_fp32(r, lo[r], hi[r]);
            }
            __syncthreads();
            if (threadIdx.x == 0) q_n = f_n = 0;
            __syncthreads();
        }
        if (last) break;
    }
    __syncthreads();
    for (int i = threadIdx.x; i <= nq; i += blockDim.x) {
        if (sh[i]) atomicAdd(&hist[i], (unsigned long long)sh[i]);
        if (sm[i]) atomicAdd(&maybe[i], (unsigned long long)(long long)sm[i]);   // mod 2^64
    }
    if (lane == 0 && scored) {
        atomicAdd(&ctr->refined, scored);
        if (fallbacks) atomicAdd(&ctr->exact_fallbacks, fallbacks);
    }
}

__global__ void gather_ranks_kernel(const int32_t* __restrict__ rank_of,
                                    const int32_t* __restrict__ ids, int n, int32_t* out) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) out[i] = rank_of[ids[i]];
}

// Every id of a sparse list: inside the snapshot, not deleted, not repeated
// (one bit per id in `seen`, zeroed before; the second setter of a bit finds
// it set).  The verdict goes to *status.
__global__ void list_check_kernel(const int64_t* __restrict__ ids, int64_t n, int64_t rows,
                                  const uint32_t* __restrict__ tomb, uint32_t* seen, int* status) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const int64_t x = ids[i];
        if (x < 0 || x >= rows || tombstoned(tomb, x)) {
            set_status(status, PVS_ERR_INVALID);
            continue;
        }
        const uint32_t bit = 1u << (x & 31);
        if (atomicOr(&seen[x >> 5], bit) & bit) set_status(status, PVS_ERR_INVALID);
    }
}

// out[k] = position + 1 of q[k] in the list (0: absent), q ascending and
// distinct (nq <= kRankQueryMax), one pass over the list.
__global__ void list_find_kernel(const int64_t* __restrict__ ids, int64_t n,
                                 const int32_t* __restrict__ q, int nq, int32_t* out) {
    __shared__ int32_t sq[kRankQueryMax];
    for (int i = threadIdx.x; i < nq; i += blockDim.x) sq[i] = q[i];
    __syncthreads();
    if (nq == 0) return;
    const int64_t qlo = sq[0], qhi = sq[nq - 1];
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const int64_t x = ids[i];
        if (x < qlo || x > qhi) continue;
        int lo = 0, hi = nq - 1;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (sq[mid] < x) lo = mid + 1;
            else hi = mid;
        }
        if (sq[lo] == x) out[lo] = (int32_t)(i + 1);
    }
}

}  // namespace

pvs_status fuse_complete(pvs_cursor* c, const int64_t* sparse, int64_t ns, const FuseWeights& w,
                         int32_t K, std::vector<FusedCand>* out) {
    out->clear();
    if (!c || !c->index || K < 1 || ns < 0 || (ns > 0 && !sparse)) return PVS_ERR_INVALID;
    pvs_index* x = c->index;
    int prev = -1;
    cudaGetDevice(&prev);
    if (prev != x->device) cudaSetDevice(x->device);
    struct Restore {
        int dev;
        ~Restore() {
            if (dev >= 0) cudaSetDevice(dev);
        }
    } restore{prev != x->device ? prev : -1};

    const SnapData* sd = c->snap.get();
    const int64_t rows = sd->rows, visible = sd->visible;
    const uint32_t* tomb = sd->d_tomb;
    cudaStream_t st = c->stream;
    cudaStream_t st2 = nullptr;
    cudaEvent_t ev = nullptr;
    std::vector<void*> held;
    pvs_status result = PVS_OK;
    auto alloc = [&](size_t bytes, cudaStream_t s) -> void* {
        void* p = nullptr;
        if (cudaMallocFromPoolAsync(&p, std::max<size_t>(bytes, 16), x->scratch_pool, s) !=
            cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        held.push_back(p);
        return p;
    };
    auto cleanup = [&]() {
        // st frees everything, after whatever st2 still has queued
        if (st2 && ev && cudaEventRecord(ev, st2) == cudaSuccess) cudaStreamWaitEvent(st, ev, 0);
        for (void* p : held) cudaFreeAsync(p, st);
        if (ev) cudaEventDestroy(ev);
        if (st2) cudaStreamDestroy(st2);
        cudaGetLastError();
    };
#define FUSE_CUDA(expr)                                            \
    do {                                                           \
        cudaError_t e_ = (expr);                                   \
        if (e_ != cudaSuccess) {                                   \
            cudaGetLastError();                                    \
            cleanup();                                             \
            return e_ == cudaErrorMemoryAllocation ? PVS_ERR_OOM   \
                                                   : PVS_ERR_CUDA; \
        }                                                          \
    } while (0)
    if (cudaStreamCreateWithFlags(&st2, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        cleanup();
        return PVS_ERR_CUDA;
    }
    const size_t n = (size_t)std::max<int64_t>(rows, 1);
    uint64_t* keys = static_cast<uint64_t*>(alloc(n * 8, st));
    uint64_t* tmp = static_cast<uint64_t*>(alloc(n * 8, st));
    void* sort_scratch = alloc(radix_sort_scratch_bytes((int64_t)n), st);
    int32_t* rd = static_cast<int32_t*>(alloc(n * 4, st));
    int* status = static_cast<int*>(alloc(2 * sizeof(int), st));
    DevCounters* ctr = static_cast<DevCounters*>(alloc(sizeof(DevCounters), st));
    // the sparse side lives on st2 until the join
    int32_t* rs = static_cast<int32_t*>(alloc(n * 4, st2));
    int64_t* d_sparse = static_cast<int64_t*>(alloc((size_t)std::max<int64_t>(ns, 1) * 8, st2));
    if (!keys || !tmp || !sort_scratch || !rd || !status || !ctr || !rs || !d_sparse) {
        cleanup();
        return PVS_ERR_OOM;
    }
    // 1. dense: every visible row's authoritative score, one sort
    FUSE_CUDA(cudaMemsetAsync(status, 0, 2 * sizeof(int), st));
    FUSE_CUDA(cudaMemsetAsync(ctr, 0, sizeof(DevCounters), st));
    FUSE_CUDA(cudaMemsetAsync(rd, 0, n * 4, st));
    FUSE_CUDA(launch_scan_scores(c->qraw, x->raw, x->m_raw, rows, tomb, keys, status, ctr, st));
    if (rows > 1) FUSE_CUDA(launch_radix_sort_desc(keys, tmp, rows, sort_scratch, st));
    count_launches(1);
    dense_rank_kernel<<<grid_of(visible), 256, 0, st>>>(keys, visible, rd);
    FUSE_CUDA(cudaGetLastError());
    // 2. sparse: the caller's list, on st2 (its host copy overlaps step 1)
    FUSE_CUDA(cudaMemsetAsync(rs, 0, n * 4, st2));
    if (ns > 0) {
        FUSE_CUDA(cudaMemcpyAsync(d_sparse, sparse, (size_t)ns * 8, cudaMemcpyHostToDevice, st2));
        count_launches(1);
        list_rank_kernel<<<grid_of(ns), 256, 0, st2>>>(d_sparse, ns, rows, tomb, rs, status + 1);
        FUSE_CUDA(cudaGetLastError());
    }
    FUSE_CUDA(cudaEventRecord(ev, st2));
    FUSE_CUDA(cudaStreamWaitEvent(st, ev, 0));
    // 3. fused keys, one sort
    count_launches(1);
    fused_key_kernel<<<grid_of(rows), 256, 0, st>>>(rd, rs, rows, tomb, w, keys);
    FUSE_CUDA(cudaGetLastError());
    if (rows > 1) FUSE_CUDA(launch_radix_sort_desc(keys, tmp, rows, sort_scratch, st));
    // 4. the leading entries, until the candidate set is complete
    int64_t m = std::min<int64_t>(rows, std::max<int64_t>(4096, 4 * (int64_t)K));
    for (;;) {
        FusedCand* d_out = static_cast<FusedCand*>(alloc((size_t)m * sizeof(FusedCand), st));
        if (!d_out) {
            cleanup();
            return PVS_ERR_OOM;
        }
        count_launches(1);
        top_entries_kernel<<<grid_of(m), 256, 0, st>>>(keys, m, rd, rs, d_out);
        FUSE_CUDA(cudaGetLastError());
        std::vector<FusedCand> h((size_t)m);
        int h_status[2] = {0, 0};
        FUSE_CUDA(cudaMemcpyAsync(h.data(), d_out, (size_t)m * sizeof(FusedCand),
                                  cudaMemcpyDeviceToHost, st));
        FUSE_CUDA(cudaMemcpyAsync(h_status, status, sizeof(h_status), cudaMemcpyDeviceToHost, st));
        FUSE_CUDA(cudaStreamSynchronize(st));
        if (h_status[0] != 0) result = (pvs_status)h_status[0];
        else if (h_status[1] != 0) result = (pvs_status)h_status[1];
        if (result != PVS_OK) break;
        int64_t live = 0;
        while (live < m && h[(size_t)live].id >= 0) ++live;
        if (live < K) {   // fewer than K items with a positive score: all of them
            out->assign(h.begin(), h.begin() + live);
            break;
        }
        // every item whose binary32 value reaches the one just below the K-th
        const uint32_t thr = h[(size_t)K - 1].fbits - 1u;
        int64_t cnt = K;
        while (cnt < live && h[(size_t)cnt].fbits >= thr) ++cnt;
        if (cnt < m || m == rows) {
            out->assign(h.begin(), h.begin() + cnt);
            break;
        }
        m = std::min<int64_t>(rows, 4 * m);   // the boundary group runs past the prefix
    }
    cleanup();
#undef FUSE_CUDA
    return result;
}

void free_staged_list(StagedList* s) {
    if (!s) return;
    int prev = -1;
    cudaGetDevice(&prev);
    if (s->index) cudaSetDevice(s->index->device);
    if (s->stream) {
        if (s->rank_of) cudaFreeAsync(s->rank_of, s->stream);
        if (s->list) cudaFreeAsync(s->list, s->stream);
        if (s->seen) cudaFreeAsync(s->seen, s->stream);
        if (s->status) cudaFreeAsync(s->status, s->stream);
        cudaStreamSynchronize(s->stream);
        cudaStreamDestroy(s->stream);
    }
    if (s->ready) cudaEventDestroy(s->ready);
    cudaGetLastError();
    if (prev >= 0) cudaSetDevice(prev);
    delete s;
}

pvs_status stage_sparse_list(pvs_cursor* c, const int64_t* sparse, int64_t ns,
                             StagedList** out) {
    *out = nullptr;
    if (!c || !c->index || ns < 0 || (ns > 0 && !sparse)) return PVS_ERR_INVALID;
    pvs_index* x = c->index;
    if (cudaSetDevice(x->device) != cudaSuccess) {
        cudaGetLastError();
        return PVS_ERR_CUDA;
    }
    StagedList* s = new (std::nothrow) StagedList();
    if (!s) return PVS_ERR_OOM;
    s->index = x;
    s->rows = c->snap->rows;
    const uint32_t* tomb = c->snap->d_tomb;
    const size_t rows = (size_t)std::max<int64_t>(s->rows, 1);
    auto failed = [&](cudaError_t e) {
        cudaGetLastError();
        free_staged_list(s);
        return e == cudaErrorMemoryAllocation ? PVS_ERR_OOM : PVS_ERR_CUDA;
    };
    cudaError_t e = cudaStreamCreateWithFlags(&s->stream, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&s->ready, cudaEventDisableTiming);
    // the ids on the device and their check (a bit per id: 1.1 MB at 8.8M
    // rows, held in L2); the finish then finds its few ids in one pass over
    // the list, so no table of every item's rank is written beside the
    // interval pass
    const size_t words = rows / 32 + 1;
    if (e == cudaSuccess)
        e = cudaMallocFromPoolAsync(reinterpret_cast<void**>(&s->list),
                                    (size_t)std::max<int64_t>(ns, 1) * 8, x->scratch_pool,
                                    s->stream);
    if (e == cudaSuccess)
        e = cudaMallocFromPoolAsync(reinterpret_cast<void**>(&s->seen), words * 4,
                                    x->scratch_pool, s->stream);
    if (e == cudaSuccess)
        e = cudaMallocFromPoolAsync(reinterpret_cast<void**>(&s->status), sizeof(int),
                                    x->scratch_pool, s->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(s->seen, 0, words * 4, s->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(s->status, 0, sizeof(int), s->stream);
    if (e == cudaSuccess && ns > 0)
        e = cudaMemcpyAsync(s->list, sparse, (size_t)ns * 8, cudaMemcpyHostToDevice, s->stream);
    if (e != cudaSuccess) return failed(e);
    s->tomb = tomb;
    s->n = ns;
    s->checked = false;   // check_staged_list queues the check
    *out = s;
    return PVS_OK;
}

pvs_status check_staged_list(StagedList* s) {
    if (!s || s->checked) return PVS_OK;
    s->checked = true;
    int prev = -1;
    cudaGetDevice(&prev);
    if (s->index && prev != s->index->device) cudaSetDevice(s->index->device);
    cudaError_t e = cudaSuccess;
    if (s->n > 0) {
        count_launches(1);
        list_check_kernel<<<grid_of(s->n), 256, 0, s->stream>>>(s->list, s->n, s->rows, s->tomb,
                                                                s->seen, s->status);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaEventRecord(s->ready, s->stream);
    if (s->index && prev >= 0 && prev != s->index->device) cudaSetDevice(prev);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return PVS_ERR_CUDA;
    }
    return PVS_OK;
}

pvs_status rank_queries(pvs_cursor* c, const int32_t* dense_ids, int32_t nd, bool exact,
                        const int64_t* sparse, int64_t ns, const int32_t* sparse_ids, int32_t nsq,
                        int64_t* dense_lo, int64_t* dense_hi, int64_t* sparse_rank,
                        bool* supported, const StagedList* staged) {
    if (supported) *supported = false;
    if (!c || !c->index || !supported || nd < 0 || nsq < 0 || nd > kRankQueryMax ||
        nsq > kRankQueryMax || ns < 0 || (nd > 0 && (!dense_ids || !dense_lo || !dense_hi)) ||
        (nsq > 0 && (!sparse_ids || !sparse_rank || (ns > 0 && !sparse && !staged))))
        return PVS_ERR_INVALID;
    if (c->state < 0) return PVS_ERR_FAILED;
    if (nd > 0 && (c->generator != PVS_GEN_INTERVALS || c->batch_ws || !c->scanned || !c->lo ||
                   c->ahead != 0))
        return PVS_OK;   // not supported: the caller finishes another way
    *supported = true;
    pvs_index* x = c->index;
    int prev = -1;
    cudaGetDevice(&prev);
    if (prev != x->device) cudaSetDevice(x->device);
    struct Restore {
        int dev;
        ~Restore() {
            if (dev >= 0) cudaSetDevice(dev);
        }
    } restore{prev != x->device ? prev : -1};

    const SnapData* sd = c->snap.get();
    const int64_t rows = sd->rows;
    for (int32_t i = 0; i < nd; ++i)
        if (dense_ids[i] < 0 || dense_ids[i] >= rows || !sd->is_visible(dense_ids[i]))
            return PVS_ERR_INVALID;
    for (int32_t i = 0; i < nsq; ++i)
        if (sparse_ids[i] < 0 || sparse_ids[i] >= rows) return PVS_ERR_INVALID;
    const uint32_t* tomb = sd->d_tomb;
    cudaStream_t st = c->stream;
    // the second stream, its event and the pinned staging stay with the
    // cursor (created at its first rank query, freed with its buffers)
    if (!c->rq_stream || !c->rq_event || !c->rq_pinned) {
        if ((!c->rq_stream &&
             cudaStreamCreateWithFlags(&c->rq_stream, cudaStreamNonBlocking) != cudaSuccess) ||
            (!c->rq_event &&
             cudaEventCreateWithFlags(&c->rq_event, cudaEventDisableTiming) != cudaSuccess) ||
            (!c->rq_pinned && cudaMallocHost(&c->rq_pinned, kRankQueryPinned) != cudaSuccess)) {
            cudaGetLastError();
            return PVS_ERR_CUDA;
        }
    }
    cudaStream_t st2 = c->rq_stream;
    cudaEvent_t ev = c->rq_event;
    std::vector<void*> held;
    auto alloc = [&](size_t bytes, cudaStream_t s) -> void* {
        void* p = nullptr;
        if (cudaMallocFromPoolAsync(&p, std::max<size_t>(bytes, 16), x->scratch_pool, s) !=
            cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        held.push_back(p);
        return p;
    };
    // st frees the scratch after whatever st2 still has queued, and ends
    // every call joined (the next call's st2 work follows this call's st)
    auto cleanup = [&]() {
        if (cudaEventRecord(ev, st2) == cudaSuccess) cudaStreamWaitEvent(st, ev, 0);
        for (void* p : held) cudaFreeAsync(p, st);
        if (cudaEventRecord(ev, st) == cudaSuccess) cudaStreamWaitEvent(st2, ev, 0);
        cudaGetLastError();
    };
#define RQ_CUDA(expr)                                              \
    do {                                                           \
        cudaError_t e_ = (expr);                                   \
        if (e_ != cudaSuccess) {                                   \
            cudaGetLastError();                                    \
            cleanup();                                             \
            return e_ == cudaErrorMemoryAllocation ? PVS_ERR_OOM   \
                                                   : PVS_ERR_CUDA; \
        }                                                          \
    } while (0)
    // host staging: the queried ids in, the counts and ranks out (pinned,
    // so the copies are asynchronous; every use ends at this call's wait)
    const size_t id_bytes = (size_t)std::max(nd, 1) * 8 + (size_t)std::max(nsq, 1) * 4;
    int64_t* h_dids = static_cast<int64_t*>(c->rq_pinned);
    int32_t* h_sids = reinterpret_cast<int32_t*>(h_dids + std::max(nd, 1));
    unsigned long long* h_hist =
        reinterpret_cast<unsigned long long*>(static_cast<char*>(c->rq_pinned) + id_bytes);
    unsigned long long* h_maybe = h_hist + nd + 1;
    uint64_t* h_keys = reinterpret_cast<uint64_t*>(h_maybe + nd + 1);
    int32_t* h_srank = reinterpret_cast<int32_t*>(h_keys + std::max(nd, 1));
    int* h_status = reinterpret_cast<int*>(h_srank + std::max(nsq, 1));
    for (int32_t i = 0; i < nd; ++i) h_dids[i] = dense_ids[i];
    for (int32_t i = 0; i < nsq; ++i) h_sids[i] = sparse_ids[i];
    h_status[0] = h_status[1] = 0;

    int* status = static_cast<int*>(alloc(2 * sizeof(int), st));
    if (!status) {
        cleanup();
        return PVS_ERR_OOM;
    }
    RQ_CUDA(cudaMemsetAsync(status, 0, 2 * sizeof(int), st));
    RQ_CUDA(cudaEventRecord(ev, st));   // st2 uses the status word too
    RQ_CUDA(cudaStreamWaitEvent(st2, ev, 0));
    // dense: the items' scores and sorted keys, then one pass over the bounds
    if (nd > 0) {
        int64_t* d_dids = static_cast<int64_t*>(alloc((size_t)nd * 8, st));
        float* d_score = static_cast<float*>(alloc((size_t)nd * 4, st));
        uint64_t* d_keys = static_cast<uint64_t*>(alloc((size_t)nd * 8, st));
        unsigned long long* d_hist =
            static_cast<unsigned long long*>(alloc((size_t)(nd + 1) * 16, st));
        unsigned long long* d_maybe = d_hist + nd + 1;
        if (!d_dids || !d_score || !d_keys || !d_hist) {
            cleanup();
            return PVS_ERR_OOM;
        }
        RQ_CUDA(cudaMemcpyAsync(d_dids, h_dids, (size_t)nd * 8, cudaMemcpyHostToDevice, st));
        RQ_CUDA(cudaMemsetAsync(d_hist, 0, (size_t)(nd + 1) * 16, st));
        RQ_CUDA(launch_score_ids(d_dids, nd, c->qraw, x->raw, x->m_raw, d_score, c->ctr, st));
        count_launches(1);
        query_keys_kernel<<<1, kRankQueryMax, 0, st>>>(d_dids, d_score, nd, d_keys, status);
        RQ_CUDA(cudaGetLastError());
        // the residual codes place most rows of an exact count without their fp32 row
        const bool resid = exact && x->m_pad <= kResidMaxPad;
        if (resid) {
            const pvs_status rs = ensure_resid(x, st, status);
            if (rs != PVS_OK) {
                cleanup();
                return rs;
            }
        }
        static const int grid = [] {
            int g = 0;
            if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&g, rank_count_kernel,
                                                              kCountWarps * 32, 0) != cudaSuccess) {
                cudaGetLastError();
                g = 1;
            }
            return g;
        }();
        int64_t blocks = (int64_t)std::max(grid, 1) * std::max(x->num_sms, 1);
        blocks = std::min<int64_t>(blocks,
                                   std::max<int64_t>(1, (rows + kCountTile - 1) / kCountTile));
        count_launches(1);
        // |zq_j| <= Q keeps sum |zq_j z_j| <= m_pad Q 127 below 2^31
        const int qrange = (int)std::min<int64_t>(16383, ((int64_t(1) << 31) - 1) /
                                                             (127 * (int64_t)x->m_pad));
        // the query codes' 4 m_pad bytes beside 33 KB of static shared memory
        // pass the default 48 KB once m_pad exceeds 3,840
        if (resid) RQ_CUDA(raise_smem_limit((const void*)rank_count_kernel, (size_t)x->m_pad * 4));
        rank_count_kernel<<<(unsigned)blocks, kCountWarps * 32,
                            resid ? (size_t)x->m_pad * 4 : 0, st>>>(
            c->lo, c->hi, rows, tomb, c->qraw, x->raw, x->m_raw, d_keys, nd, exact ? 1 : 0,
            resid ? x->codes : nullptr, resid ? x->resid : nullptr, x->rparam, x->m_pad, qrange,
            c->qs, d_hist, d_maybe, status, c->ctr);
        RQ_CUDA(cudaGetLastError());
        RQ_CUDA(cudaMemcpyAsync(h_hist, d_hist, (size_t)(nd + 1) * 16, cudaMemcpyDeviceToHost,
                                st));
        RQ_CUDA(cudaMemcpyAsync(h_keys, d_keys, (size_t)nd * 8, cudaMemcpyDeviceToHost, st));
    }
    // sparse (second stream; a copy from pageable memory may hold this thread
    // until it is done, so the dense work is queued first): a PBM ranking's
    // table read at the queried ids, or one pass over a host list (staged
    // ahead, or copied and checked here) that finds the queried ids, sorted
    // and without repeats
    int32_t* d_srank = nullptr;
    std::vector<int32_t> uniq, slot_of;   // distinct queried ids ascending; each query's slot
    if (nsq > 0 && staged && staged->rows != rows) {
        cleanup();
        return PVS_ERR_INVALID;
    }
    if (nsq > 0) {
        const bool table = staged && staged->rank_of;
        int nfind = nsq;
        if (!table) {
            uniq.assign(sparse_ids, sparse_ids + nsq);
            std::sort(uniq.begin(), uniq.end());
            uniq.erase(std::unique(uniq.begin(), uniq.end()), uniq.end());
            slot_of.resize((size_t)nsq);
            for (int32_t i = 0; i < nsq; ++i)
                slot_of[(size_t)i] = (int32_t)(std::lower_bound(uniq.begin(), uniq.end(),
                                                                sparse_ids[i]) -
                                               uniq.begin());
            nfind = (int)uniq.size();
            std::copy(uniq.begin(), uniq.end(), h_sids);
        }
        int32_t* d_sids = static_cast<int32_t*>(alloc((size_t)nfind * 4, st2));
        d_srank = static_cast<int32_t*>(alloc((size_t)nfind * 4, st2));
        int64_t* d_list = staged ? staged->list : nullptr;
        if (!staged) {   // the host list, copied and checked by this call
            const size_t words = (size_t)std::max<int64_t>(rows, 1) / 32 + 1;
            d_list = static_cast<int64_t*>(alloc((size_t)std::max<int64_t>(ns, 1) * 8, st2));
            uint32_t* seen = static_cast<uint32_t*>(alloc(words * 4, st2));
            if (!d_list || !seen) {
                cleanup();
                return PVS_ERR_OOM;
            }
            RQ_CUDA(cudaMemsetAsync(seen, 0, words * 4, st2));
            if (ns > 0) {
                RQ_CUDA(cudaMemcpyAsync(d_list, sparse, (size_t)ns * 8, cudaMemcpyHostToDevice,
                                        st2));
                count_launches(1);
                list_check_kernel<<<grid_of(ns), 256, 0, st2>>>(d_list, ns, rows, tomb, seen,
                                                                status + 1);
                RQ_CUDA(cudaGetLastError());
            }
        }
        if (!d_sids || !d_srank || (!table && ns > 0 && !d_list)) {
            cleanup();
            return PVS_ERR_OOM;
        }
        RQ_CUDA(cudaMemcpyAsync(d_sids, h_sids, (size_t)nfind * 4, cudaMemcpyHostToDevice, st2));
        if (staged) {   // staged ahead: its verdict becomes this call's
            RQ_CUDA(cudaStreamWaitEvent(st2, staged->ready, 0));
            RQ_CUDA(cudaMemcpyAsync(status + 1, staged->status, sizeof(int),
                                    cudaMemcpyDeviceToDevice, st2));
        }
        if (table) {
            count_launches(1);
            gather_ranks_kernel<<<(nsq + 255) / 256, 256, 0, st2>>>(staged->rank_of, d_sids, nsq,
                                                                    d_srank);
        } else {
            const int64_t n_list = staged ? std::max<int64_t>(ns, 0) : ns;
            RQ_CUDA(cudaMemsetAsync(d_srank, 0, (size_t)nfind * 4, st2));
            count_launches(1);
            list_find_kernel<<<grid_of(n_list), 256, 0, st2>>>(d_list, n_list, d_sids, nfind,
                                                               d_srank);
        }
        RQ_CUDA(cudaGetLastError());
        RQ_CUDA(cudaMemcpyAsync(h_srank, d_srank, (size_t)nfind * 4, cudaMemcpyDeviceToHost, st2));
    }
    RQ_CUDA(cudaEventRecord(ev, st2));
    RQ_CUDA(cudaStreamWaitEvent(st, ev, 0));
    RQ_CUDA(cudaMemcpyAsync(h_status, status, 2 * sizeof(int), cudaMemcpyDeviceToHost, st));
    RQ_CUDA(cudaStreamSynchronize(st));
    pvs_status result = PVS_OK;
    if (h_status[0] != 0) result = (pvs_status)h_status[0];
    else if (h_status[1] != 0) result = (pvs_status)h_status[1];
    if (result == PVS_OK) {
        // the item with the j-th smallest key: 1 + rows surely above it, plus
        // the rows that may be above it
        unsigned long long above = 0, may = 0;
        struct Ranks {
            int32_t id;
            int64_t lo, hi;
            bool operator<(const Ranks& o) const { return id < o.id; }
        };
        std::vector<Ranks> by_id((size_t)nd);
        for (int32_t j = nd - 1; j >= 0; --j) {
            above += h_hist[j + 1];
            by_id[(size_t)j].id = (int32_t)rank_key_id(h_keys[j]);
            by_id[(size_t)j].lo = (int64_t)above + 1;
        }
        for (int32_t j = 0; j < nd; ++j) {
            may += h_maybe[j];   // prefix sum of the differences (mod 2^64)
            by_id[(size_t)j].hi = by_id[(size_t)j].lo + (int64_t)may;
        }
        std::sort(by_id.begin(), by_id.end());
        for (int32_t i = 0; i < nd; ++i) {
            const auto it = std::lower_bound(by_id.begin(), by_id.end(), Ranks{dense_ids[i], 0, 0});
            if (it == by_id.end() || it->id != dense_ids[i]) {
                result = PVS_ERR_INVALID;   // a repeated item
                break;
            }
            dense_lo[i] = it->lo;
            dense_hi[i] = it->hi;
        }
        for (int32_t i = 0; i < nsq; ++i)
            sparse_rank[i] = slot_of.empty() ? h_srank[i] : h_srank[slot_of[(size_t)i]];
    }
    cleanup();
#undef RQ_CUDA
    return result;
}

}  // namespace pvs
