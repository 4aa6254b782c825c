// Exact authoritative float32 score of one vector, computed by one warp
// (arXiv 2608.07152 Sec. 2.3.1 authoritative scores; App. A.1).
//
// The score is RN_f32 of the exact inner product sum_j q_j v_j.  Three
// layers, each deciding only when its error bound proves the rounding:
//   1. exact_dot_warp_eft (the common path, float32 pipe): error-free
//      transformations of every product and partial sum with a bounded
//      error sum, decided in float32 (see below);
//   2. exact_dot_warp_impl, binary64: every product of two float32 values is
//      exact in binary64; lanes accumulate S = sum p_j and A = sum |p_j|;
//      |S - exact| <= (m - 1) u A / (1 - (m - 1) u) with u = 2^-53 for any
//      summation order, and with beta = 4 m u A the interval
//      [RD(S - beta), RU(S + beta)] rounding to one float32 value decides;
//   3. otherwise the warp sums the products exactly in a fixed-point
//      accumulator (20 signed 32-bit digits in int64 slots, weight 2^-352 for
//      the lowest bit) and rounds the exact sum to nearest-even.
// A result that rounds to zero is +0.
#pragma once

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
    // products of finite float32 values always land in range; anything else
    // (callers check finiteness first) is ignored rather than written out of bounds
    if (bexp == 0 || bexp == 0x7ff || pos < 0 || d + 2 >= kAccDigits) return;
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
    return (negative && f != 0.0f) ? -f : f;   // a result that rounds to zero is +0
}

// Products q_j * v_j of one lane, visited in a fixed order: float4 loads for
// 16-byte aligned rows whose length is a multiple of 4 (the index layout),
// scalar loads otherwise.
template <bool kVec4, typename F>
__device__ inline void for_lane_products(const float* __restrict__ q, const float* __restrict__ v,
                                         int m, F&& f) {
    const int lane = threadIdx.x & 31;
    if constexpr (kVec4) {
        const float4* q4 = reinterpret_cast<const float4*>(q);
        const float4* v4 = reinterpret_cast<const float4*>(v);
        for (int j = lane; j < (m >> 2); j += kWarp) {
            const float4 a = __ldg(q4 + j), b = __ldg(v4 + j);
            f(__dmul_rn((double)a.x, (double)b.x), __dmul_rn((double)a.y, (double)b.y),
              __dmul_rn((double)a.z, (double)b.z), __dmul_rn((double)a.w, (double)b.w));
        }
    } else {
        for (int j = lane; j < m; j += kWarp)
            f(__dmul_rn((double)__ldg(q + j), (double)__ldg(v + j)), 0.0, 0.0, 0.0);
    }
}

// One warp: exact RN_f32(sum q_j v_j) over m finite entries.
template <bool kVec4>
__device__ inline float exact_dot_warp_impl(const float* __restrict__ q,
                                            const float* __restrict__ v, int m,
                                            bool* used_fallback) {
    double S = 0.0, A = 0.0;
    for_lane_products<kVec4>(q, v, m, [&](double p0, double p1, double p2, double p3) {
        S = __dadd_rn(S, __dadd_rn(__dadd_rn(p0, p1), __dadd_rn(p2, p3)));
        A = __dadd_rn(A, __dadd_rn(__dadd_rn(fabs(p0), fabs(p1)), __dadd_rn(fabs(p2), fabs(p3))));
    });
    S = warp_sum(S);
    A = warp_sum(A);
    const double beta = __dmul_ru(A, 4.0 * (double)m * 0x1p-53);
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
    for_lane_products<kVec4>(q, v, m, [&](double p0, double p1, double p2, double p3) {
        acc_add(acc, p0);
        acc_add(acc, p1);
        acc_add(acc, p2);
        acc_add(acc, p3);
    });
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

// Index rows: 16-byte aligned, m_raw a multiple of 4 (zero padded).
__device__ inline float exact_dot_warp(const float* __restrict__ q, const float* __restrict__ v,
                                       int m_raw, bool* used_fallback) {
    return exact_dot_warp_impl<true>(q, v, m_raw, used_fallback);
}

// Fast form on the float32 pipe (binary64 throughput is a small fraction of
// float32 throughput on this part).  Error-free transformations (Knuth's
// TwoSum; TwoProduct with one fused multiply-add, as in Ogita, Rump and Oishi,
// "Accurate sum and dot product", 2005) split every product and every partial
// sum of the main accumulator s into its rounded value and exact error; the
// errors are summed in float32 into c.  Bookkeeping that makes the result
// rigorous for any summation order:
//   * exact = s + (sum of all error terms) + d, where |d| <= m 2^-150 covers
//     the only inexact step, a TwoProduct error term that underflows;
//   * every float32 addition of the error sum satisfies x + y = fl(x + y)(1 + e)
//     with |e| <= 2^-24, so |c - sum of error terms| <= 2^-24 sum |fl(node)|
//     over the additions that built c; a holds that sum rounded upward.
// The decision is taken in float32 too (below); rows it cannot settle go to
// the binary64 / exact path.
// Out of line so that the rare ambiguous case does not cost the fast loop
// registers.
static __device__ __noinline__ float exact_dot_warp_slow(const float* __restrict__ q,
                                                  const float* __restrict__ v, int m_raw,
                                                  bool* used_fallback) {
    return exact_dot_warp_impl<true>(q, v, m_raw, used_fallback);
}

__device__ inline void two_sum_f(float a, float b, float& s, float& e) {
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

struct EftAcc {
    float s = 0.0f, c = 0.0f, a1 = 0.0f, a2 = 0.0f;
    __device__ inline void add_product(float x, float y) {
        const float p = __fmul_rn(x, y);
        const float ep = __fmaf_rn(x, y, -p);
        float es;
        two_sum_f(s, p, s, es);
        const float t = __fadd_rn(ep, es);
        c = __fadd_rn(c, t);
        a1 = __fadd_ru(a1, fabsf(t));
        a2 = __fadd_ru(a2, fabsf(c));
    }
    // Merge another lane's accumulator (commutative: every lane of a butterfly
    // ends with the same bits).
    __device__ inline void merge(float s2, float c2, float a12, float a22) {
        float es;
        two_sum_f(s, s2, s, es);
        const float cc = __fadd_rn(c, c2);
        const float c3 = __fadd_rn(cc, es);
        a1 = __fadd_ru(__fadd_ru(a1, a12), fabsf(cc));
        a2 = __fadd_ru(__fadd_ru(a2, a22), fabsf(c3));
        c = c3;
    }
};

// Butterfly merge of the lanes' accumulators, then the float32 decision:
// r = RN(s + c) with its exact error e2 (TwoSum), so exact = r + e2 + d with
// |d| <= 2^-24 a + m 2^-149 (the error-sum and underflow bounds, rounded up).
// Within half the gap around r on either side (a quarter of an ulp below a
// power of two) the nearest float32 is r.  Returns false when that does not
// settle the row (then the binary64 / exact path must).
__device__ inline bool eft_finish(EftAcc acc, int m_raw, float* out) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float s2 = __shfl_xor_sync(0xffffffffu, acc.s, off);
        const float c2 = __shfl_xor_sync(0xffffffffu, acc.c, off);
        const float a12 = __shfl_xor_sync(0xffffffffu, acc.a1, off);
        const float a22 = __shfl_xor_sync(0xffffffffu, acc.a2, off);
        acc.merge(s2, c2, a12, a22);
    }
    float r, e2;
    two_sum_f(acc.s, acc.c, r, e2);
    const float ar = fabsf(r);
    if (!(ar >= 0x1p-100f && ar <= 0x1p+126f && isfinite(acc.c))) return false;
    const float a = __fadd_ru(acc.a1, acc.a2);
    const float bound = __fadd_ru(fabsf(e2), __fadd_ru(__fmul_ru(a, 0x1p-24f),
                                                       __fmul_ru((float)m_raw, 0x1p-149f)));
    const unsigned int bits = __float_as_uint(ar);
    const float ulp = __uint_as_float(bits & 0x7f800000u) * 0x1p-23f;
    const float half_gap = (bits & 0x007fffffu) ? ulp * 0.5f : ulp * 0.25f;
    if (!(bound < half_gap)) return false;
    *out = r;
    return true;
}

// Index rows: 16-byte aligned, m_raw a multiple of 4 (zero padded).  q_fast
// holds the same values as q and may point to shared memory (it is read with
// generic loads); q (global) serves the out-of-line exact path.  Up to
// kBatch float4 of the row are in flight per lane: a row of up to
// 4 * 32 * kBatch values costs one round trip to memory.
template <int kBatch = 8>
__device__ inline float exact_dot_warp_eft(const float* q_fast, const float* __restrict__ q,
                                           const float* __restrict__ v, int m_raw,
                                           bool* used_fallback) {
    const int lane = threadIdx.x & 31;
    const float4* q4 = reinterpret_cast<const float4*>(q_fast);
    const float4* v4 = reinterpret_cast<const float4*>(v);
    // two independent accumulators (components x, z and y, w) halve the
    // dependency chains; they merge like two lanes of the butterfly
    EftAcc acc, acc2;
    const int n4 = m_raw >> 2;
#pragma unroll 1
    for (int j0 = lane; j0 < n4; j0 += kWarp * kBatch) {
        float4 y[kBatch];
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
            const int j = j0 + kWarp * b;
            y[b] = j < n4 ? __ldg(v4 + j) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        }
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
            const int j = j0 + kWarp * b;
            if (j < n4) {
                const float4 x = q4[j];
                acc.add_product(x.x, y[b].x);
                acc2.add_product(x.y, y[b].y);
                acc.add_product(x.z, y[b].z);
                acc2.add_product(x.w, y[b].w);
            }
        }
    }
    acc.merge(acc2.s, acc2.c, acc2.a1, acc2.a2);
    float r;
    if (eft_finish(acc, m_raw, &r)) {
        *used_fallback = false;
        return r;
    }
    return exact_dot_warp_slow(q, v, m_raw, used_fallback);
}

// The same score with the row already in shared memory (v_sh, generic loads);
// v (global) is the same row for the exact path.
__device__ inline float exact_dot_warp_eft_smem(const float* q_fast, const float* __restrict__ q,
                                                const float* v_sh, const float* __restrict__ v,
                                                int m_raw, bool* used_fallback) {
    const int lane = threadIdx.x & 31;
    const float4* q4 = reinterpret_cast<const float4*>(q_fast);
    const float4* v4 = reinterpret_cast<const float4*>(v_sh);
    EftAcc acc, acc2;   // two dependency chains, merged as in the butterfly
    const int n4 = m_raw >> 2;
    for (int j = lane; j < n4; j += kWarp) {
        const float4 x = q4[j], y = v4[j];
        acc.add_product(x.x, y.x);
        acc2.add_product(x.y, y.y);
        acc.add_product(x.z, y.z);
        acc2.add_product(x.w, y.w);
    }
    acc.merge(acc2.s, acc2.c, acc2.a1, acc2.a2);
    float r;
    if (eft_finish(acc, m_raw, &r)) {
        *used_fallback = false;
        return r;
    }
    return exact_dot_warp_slow(q, v, m_raw, used_fallback);
}

// Any row of m float32 values.
__device__ inline float exact_dot_warp_any(const float* __restrict__ q,
                                           const float* __restrict__ v, int m,
                                           bool* used_fallback) {
    return exact_dot_warp_impl<false>(q, v, m, used_fallback);
}

}  // namespace pvs
