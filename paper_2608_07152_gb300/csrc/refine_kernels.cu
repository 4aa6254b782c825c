// Authoritative float32 scores of PVS candidates (Sec. 2.3.1: raw vectors are
// read only for candidates the intervals do not order; App. A.1: a score
// outside its interval fails the request).
//
// The authoritative score is RN_f32 of the exact inner product sum_j q_j v_j.
// One warp scores one candidate:
//   * every product of two float32 values is exact in binary64; lanes
//     accumulate S = sum p_j and A = sum |p_j| in binary64 and reduce them;
//   * |S - exact| <= (m - 1) u A / (1 - (m - 1) u) with u = 2^-53 for any
//     summation order; with beta = 4 m u A the whole interval
//     [RD(S - beta), RU(S + beta)] rounds to one float32 value in all but
//     rare cases, and that value is the answer;
//   * otherwise the warp sums the products exactly in a fixed-point
//     accumulator (20 signed 32-bit digits in int64 slots, weight 2^-352 for
//     the lowest bit) and rounds the exact sum to nearest-even.
#include "kernels.h"
#include "pvs_common.cuh"

namespace pvs {

constexpr int kAccDigits = 20;
constexpr int kAccBase = 352;   // bit 0 of the accumulator has weight 2^-352

// Add one exact binary64 product into the per-lane fixed-point accumulator.
__device__ inline void acc_add(long long* acc, double p) {
    if (p == 0.0) return;
    const unsigned long long bits = (unsigned long long)__double_as_longlong(p);
    const int bexp = (int)((bits >> 52) & 0x7ff);           // normal: |p| >= 2^-298
    const unsigned long long mant = (bits & 0xfffffffffffffull) | (1ull << 52);
    const int pos = bexp - 1075 + kAccBase;                 // weight of mant's bit 0
    const int d = pos >> 5, o = pos & 31;
    unsigned long long w0, rest;
    if (o == 0) {
        w0 = mant & 0xffffffffull;
        rest = mant >> 32;
    } else {
        w0 = (mant & ((1ull << (32 - o)) - 1ull)) << o;
        rest = mant >> (32 - o);
    }
    const unsigned long long w1 = rest & 0xffffffffull, w2 = rest >> 32;
    if (bits >> 63) {
        acc[d] -= (long long)w0;
        acc[d + 1] -= (long long)w1;
        acc[d + 2] -= (long long)w2;
    } else {
        acc[d] += (long long)w0;
        acc[d + 1] += (long long)w1;
        acc[d + 2] += (long long)w2;
    }
}

// Round the exact value held in normalised digits (magnitude, sign) to the
// nearest float32, ties to even.
__device__ inline float acc_round(const unsigned int* mag, bool negative) {
    int top = -1;
    for (int k = kAccDigits - 1; k >= 0; --k)
        if (mag[k]) {
            top = 32 * k + 31 - __clz(mag[k]);
            break;
        }
    if (top < 0) return 0.0f;
    auto bit = [&](int i) -> unsigned int {
        return i < 0 ? 0u : (mag[i >> 5] >> (i & 31)) & 1u;
    };
    const int sub_lsb = -149 + kAccBase;     // bit index of 2^-149
    int lsb = top - 23;
    if (lsb < sub_lsb) lsb = sub_lsb;
    unsigned long long M = 0;
    for (int i = top; i >= lsb; --i) M = (M << 1) | bit(i);
    const unsigned int rbit = bit(lsb - 1);
    bool sticky = false;
    for (int i = lsb - 2; i >= 0 && !sticky; --i) sticky = bit(i) != 0;
    if (rbit && (sticky || (M & 1ull))) ++M;
    // M <= 2^24; value = M * 2^(lsb - kAccBase), exact in binary64
    double v = (double)M * pow2d(lsb - kAccBase);
    float f = __double2float_rn(v);   // exact when representable; inf on overflow
    return negative ? -f : f;
}

// One warp: exact RN_f32(sum q_j v_j) over m_raw (multiple of 4) entries.
__device__ inline float exact_dot_warp(const float* __restrict__ q, const float* __restrict__ v,
                                       int m_raw, bool* used_fallback) {
    const int lane = threadIdx.x & 31;
    const float4* q4 = reinterpret_cast<const float4*>(q);
    const float4* v4 = reinterpret_cast<const float4*>(v);
    const int n4 = m_raw >> 2;
    double S = 0.0, A = 0.0;
    for (int j = lane; j < n4; j += kWarp) {
        const float4 a = __ldg(q4 + j), b = __ldg(v4 + j);
        const double p0 = __dmul_rn((double)a.x, (double)b.x);
        const double p1 = __dmul_rn((double)a.y, (double)b.y);
        const double p2 = __dmul_rn((double)a.z, (double)b.z);
        const double p3 = __dmul_rn((double)a.w, (double)b.w);
        S = __dadd_rn(S, __dadd_rn(__dadd_rn(p0, p1), __dadd_rn(p2, p3)));
        A = __dadd_rn(A, __dadd_rn(__dadd_rn(fabs(p0), fabs(p1)), __dadd_rn(fabs(p2), fabs(p3))));
    }
    S = warp_sum(S);
    A = warp_sum(A);
    const double beta = __dmul_ru(A, 4.0 * (double)m_raw * 0x1p-53);
    const float flo = __double2float_rn(__dsub_rd(S, beta));
    const float fhi = __double2float_rn(__dadd_ru(S, beta));
    if (flo == fhi) {
        *used_fallback = false;
        return flo == 0.0f ? 0.0f : flo;
    }
    // exact fallback
    *used_fallback = true;
    long long acc[kAccDigits];
#pragma unroll
    for (int k = 0; k < kAccDigits; ++k) acc[k] = 0;
    for (int j = lane; j < n4; j += kWarp) {
        const float4 a = __ldg(q4 + j), b = __ldg(v4 + j);
        acc_add(acc, __dmul_rn((double)a.x, (double)b.x));
        acc_add(acc, __dmul_rn((double)a.y, (double)b.y));
        acc_add(acc, __dmul_rn((double)a.z, (double)b.z));
        acc_add(acc, __dmul_rn((double)a.w, (double)b.w));
    }
#pragma unroll
    for (int k = 0; k < kAccDigits; ++k) acc[k] = warp_sum(acc[k]);
    // normalise: carry-propagate signed digits into 32-bit digits
    unsigned int mag[kAccDigits];
    long long carry = 0;
#pragma unroll
    for (int k = 0; k < kAccDigits; ++k) {
        const long long x = acc[k] + carry;
        mag[k] = (unsigned int)(x & 0xffffffffll);
        carry = x >> 32;   // arithmetic shift: floor division
    }
    const bool negative = carry < 0;
    if (negative) {  // two's complement negate over all digits
        unsigned long long c = 1;
#pragma unroll
        for (int k = 0; k < kAccDigits; ++k) {
            const unsigned long long x = (unsigned long long)(~mag[k]) + c;
            mag[k] = (unsigned int)x;
            c = x >> 32;
        }
    }
    return acc_round(mag, negative);
}

__global__ void __launch_bounds__(256) refine_kernel(
    const int32_t* __restrict__ cand, const unsigned int* cand_len, const int32_t* __restrict__ w_id,
    float* w_lo, float* w_hi, float* lo, float* hi, const float* __restrict__ qraw,
    const float* __restrict__ raw, int m_raw, int* status, DevCounters* ctr) {
    const int lane = threadIdx.x & 31;
    const int64_t n = *cand_len;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    unsigned long long refined = 0, fallbacks = 0;
    for (int64_t i = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); i < n;
         i += warps) {
        const int32_t w = cand[i];
        const float l = w_lo[w], h = w_hi[w];
        if (!(l < h)) continue;    // resolved: lo == hi is the exact score
        const int32_t id = w_id[w];
        bool fb;
        const float s = exact_dot_warp(qraw, raw + (int64_t)id * m_raw, m_raw, &fb);
        if (lane == 0) {
            ++refined;
            fallbacks += fb;
            if (!isfinite(s)) set_status(status, PVS_ERR_OVERFLOW);
            else if (s < l || s > h) set_status(status, PVS_ERR_INTERVAL);
            w_lo[w] = s;
            w_hi[w] = s;
            lo[id] = s;
            hi[id] = s;
        }
    }
    if (lane == 0 && refined) {
        atomicAdd(&ctr->refined, refined);
        if (fallbacks) atomicAdd(&ctr->exact_fallbacks, fallbacks);
    }
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
    const float s = exact_dot_warp(qraw, raw + ids[i] * m_raw, m_raw, &fb);
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
