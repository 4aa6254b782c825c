// Device-side helpers shared by the PVS kernels: ordered keys, status words,
// bounded waits, warp reductions, and the per-vector quantizer of Sec. 2.3.1.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <map>
#include <mutex>
#include <utility>

#include "../../include/pvs.h"
#include "kernels.h"

namespace pvs {

constexpr int kWarp = 32;

// ---------------------------------------------------------------------------
// Ordered 32-bit keys of float32 values: key(a) < key(b) iff a < b, with -0
// mapped onto +0.  Removed / emitted entries carry the float -inf.
// ---------------------------------------------------------------------------
__host__ __device__ inline uint32_t fkey(float f) {
    uint32_t u;
#ifdef __CUDA_ARCH__
    u = __float_as_uint(f);
#else
    __builtin_memcpy(&u, &f, 4);
#endif
    if (u == 0x80000000u) u = 0u;  // -0 -> +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__host__ __device__ inline float fkey_inv(uint32_t k) {
    uint32_t u = (k & 0x80000000u) ? (k & 0x7fffffffu) : ~k;
    float f;
#ifdef __CUDA_ARCH__
    f = __uint_as_float(u);
#else
    __builtin_memcpy(&f, &u, 4);
#endif
    return f;
}

// 64-bit rank key: larger key = earlier rank.  (score descending, id ascending)
__host__ __device__ inline uint64_t rank_key(float s, uint32_t id) {
    return ((uint64_t)fkey(s) << 32) | (uint64_t)(0xffffffffu - id);
}
__host__ __device__ inline uint32_t rank_key_id(uint64_t k) {
    return 0xffffffffu - (uint32_t)(k & 0xffffffffu);
}
__host__ __device__ inline float rank_key_score(uint64_t k) {
    return fkey_inv((uint32_t)(k >> 32));
}

// Interval of Sec. 2.3.1 / App. A.1 from the exact Int8 dot product, in the
// operation order the oracle states (RN centre, RU/RD bounds).
__device__ __forceinline__ void interval_epilogue(int dot, const QueryScalars& q, float sv,
                                                  float vn, float en, float& lo, float& hi) {
    float fdot = __int2float_rn(dot);
    float ss = __fmul_rn(q.s, sv);
    float c = __fmul_rn(ss, fdot);
    float e1 = __fmul_ru(q.enorm, vn);
    float e2 = __fmul_ru(q.qhat, en);
    float E = __fadd_ru(e1, e2);
    float g1 = __fadd_ru(fabsf(c), E);
    float g2 = __fmul_ru(q.qnorm, vn);
    float g3 = __fadd_ru(g1, g2);
    float G = __fmul_ru(g3, q.gamma);
    float r = __fadd_ru(E, G);
    lo = __fsub_rd(c, r);
    hi = __fadd_ru(c, r);
}

__device__ __forceinline__ bool tombstoned(const uint32_t* tomb, int64_t row) {
    return tomb != nullptr && ((__ldg(tomb + (row >> 5)) >> (row & 31)) & 1u);
}

// First error wins.
__device__ inline void set_status(int* status, int code) {
    atomicCAS(status, 0, code);
}

__device__ inline unsigned long long globaltimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

template <typename T>
__device__ inline T warp_sum(T v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ inline float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ inline double warp_max(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmax(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// 2^k as a double for -1022 <= k <= 1023 (exact).
__device__ inline double pow2d(int k) {
    return __longlong_as_double((long long)(1023 + k) << 52);
}

// ---------------------------------------------------------------------------
// Norm bound of Sec. 2.3.1 / App. A.1 norms, computed cooperatively by one
// warp over values x_j each exactly representable in binary64:
//   M = max|x_j| = f 2^e (f in [0.5,1)); t_j = ceil(RU(x_j^2) 2^(48-2e));
//   T = sum t_j (exact integer); bound = RU32(RU_sqrt(RU64(T) 2^(2e-48))).
// Every lane passes its own partial (maxabs over its values and the integer
// sum it accumulated against the shared exponent) through two phases; see
// quantize_row_warp for the call pattern.
// ---------------------------------------------------------------------------
__device__ inline int norm_exponent(double M) {
    int e;
    frexp(M, &e);
    return e;
}

__device__ inline long long norm_term(double x, int e) {
    double sq = __dmul_ru(x, x);
    double scaled = sq * pow2d(48 - 2 * e);   // exact power-of-two scaling
    return (long long)ceil(scaled);
}

__device__ inline float norm_finish(long long T, int e) {
    if (T == 0) return 0.0f;
    double t = __ll2double_ru(T);
    double sumsq = t * pow2d(2 * e - 48);     // exact
    double root = __dsqrt_ru(sumsq);
    return __double2float_ru(root);
}

// ---------------------------------------------------------------------------
// One warp quantizes one row of m float32 values (Sec. 2.3.1):
//   s = RN(maxabs / 127) (zero vector: 1; underflow: smallest subnormal),
//   z_j = clip(round_half_away(RN(v_j / s)), -127, 127),
//   vnorm = norm_bound(v), enorm = norm_bound(v - s z).
// Codes go to z[0..m_pad) (zero padded).  Returns a PVS status (0, or
// PVS_ERR_NONFINITE / PVS_ERR_OVERFLOW) identical in every lane.
// ---------------------------------------------------------------------------
struct RowQuant {
    float s, vnorm, enorm;
    int status;
};

// fixed_s > 0: one scale for the whole corpus (scalar-quantization
// intervals) in place of the row's own; a code that would leave [-127, 127]
// sets PVS_ERR_INVALID (the row is outside the scale's range).
__device__ inline RowQuant quantize_row_warp(const float* __restrict__ v, int m, int m_pad,
                                             int8_t* __restrict__ z, float fixed_s = 0.0f) {
    const int lane = threadIdx.x & 31;
    float maxabs = 0.0f;
    bool finite = true;
    for (int j = lane; j < m; j += kWarp) {
        float x = v[j];
        finite &= isfinite(x);
        maxabs = fmaxf(maxabs, fabsf(x));
    }
    finite = __all_sync(0xffffffffu, finite);
    maxabs = warp_max(maxabs);
    RowQuant r;
    r.status = 0;
    if (!finite) {
        r.status = PVS_ERR_NONFINITE;
        r.s = r.vnorm = r.enorm = 0.0f;
        return r;
    }
    float s;
    if (fixed_s > 0.0f) {
        s = fixed_s;
    } else if (maxabs == 0.0f) {
        s = 1.0f;
    } else {
        s = __fdiv_rn(maxabs, 127.0f);
        if (s == 0.0f) s = __uint_as_float(1u);  // 2^-149
    }
    // codes and residual maximum
    double emax = 0.0;
    bool out_of_range = false;
    for (int j = lane; j < m_pad; j += kWarp) {
        int c = 0;
        if (j < m && maxabs != 0.0f) {
            float t = __fdiv_rn(v[j], s);
            float rt = roundf(t);                      // half away from zero
            out_of_range |= fabsf(rt) > 127.0f;
            rt = fminf(fmaxf(rt, -127.0f), 127.0f);
            c = (int)rt;
            double e = __dsub_rn((double)v[j], __dmul_rn((double)s, (double)c));  // exact
            emax = fmax(emax, fabs(e));
        }
        z[j] = (int8_t)c;
    }
    __syncwarp();
    emax = warp_max(emax);
    out_of_range = __any_sync(0xffffffffu, out_of_range) && fixed_s > 0.0f;
    // norm of v
    long long Tv = 0, Te = 0;
    int ev = maxabs > 0.0f ? norm_exponent((double)maxabs) : 0;
    int ee = emax > 0.0 ? norm_exponent(emax) : 0;
    for (int j = lane; j < m; j += kWarp) {
        double x = (double)v[j];
        if (maxabs > 0.0f) Tv += norm_term(x, ev);
        if (emax > 0.0) {
            int c = z[j];
            double e = __dsub_rn(x, __dmul_rn((double)s, (double)c));
            Te += norm_term(e, ee);
        }
    }
    Tv = warp_sum(Tv);
    Te = warp_sum(Te);
    r.s = s;
    r.vnorm = norm_finish(Tv, ev);
    r.enorm = norm_finish(Te, ee);
    if (isinf(r.vnorm) || isinf(r.enorm)) r.status = PVS_ERR_OVERFLOW;
    if (out_of_range) r.status = PVS_ERR_INVALID;
    return r;
}

// Raise, never lower, a kernel's dynamic shared-memory limit on the current
// device.  The limit belongs to the function, not to a launch: host threads
// that launch one kernel with different sizes would otherwise undo each
// other's setting between one thread's set and its launch.
inline cudaError_t raise_smem_limit(const void* fn, size_t bytes) {
    static std::mutex mu;
    static std::map<std::pair<int, const void*>, size_t> limits;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    size_t& cur = limits[std::make_pair(dev, fn)];
    if (bytes <= cur) return cudaSuccess;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) cur = bytes;
    return e;
}

}  // namespace pvs
