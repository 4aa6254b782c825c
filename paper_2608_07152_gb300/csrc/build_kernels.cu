// PVS index build and query encoding (Sec. 2.3.1; norms for App. A.1).
//
// One warp quantizes one vector: float32 loads, warp max of |v_j|, IEEE
// division for the scale and the codes, and the order-independent integer
// accumulation of the norm bounds (quantize_row_warp).  The raw float32 row
// is copied next to the codes for authoritative scoring.
#include "kernels.h"
#include "pvs_common.cuh"

namespace pvs {

__global__ void __launch_bounds__(256) build_kernel(const float* __restrict__ vecs, int64_t n,
                                                    int m, int m_pad, int m_raw,
                                                    int8_t* __restrict__ codes,
                                                    float* __restrict__ scale,
                                                    float* __restrict__ vnorm,
                                                    float* __restrict__ enorm,
                                                    float* __restrict__ raw, int* status,
                                                    const float* fixed_scale) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    const float fs = fixed_scale ? *fixed_scale : 0.0f;
    for (int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); row < n;
         row += warps) {
        const float* v = vecs + row * (int64_t)m;
        RowQuant r = quantize_row_warp(v, m, m_pad, codes + row * (int64_t)m_pad, fs);
        float* dst = raw + row * (int64_t)m_raw;
        for (int j = lane; j < m_raw; j += kWarp) dst[j] = j < m ? v[j] : 0.0f;
        if (lane == 0) {
            scale[row] = r.s;
            vnorm[row] = r.vnorm;
            enorm[row] = r.enorm;
            if (r.status) set_status(status, r.status);
        }
    }
}

cudaError_t launch_build(const float* vecs, int64_t n, int m, int m_pad, int m_raw,
                         int8_t* codes, float* scale, float* vnorm, float* enorm, float* raw,
                         int* status, cudaStream_t st, const float* fixed_scale) {
    if (n <= 0) return cudaSuccess;
    int64_t blocks = (n + 7) / 8;
    if (blocks > 152 * 64) blocks = 152 * 64;
    count_launches(1);
    build_kernel<<<(unsigned)blocks, 256, 0, st>>>(vecs, n, m, m_pad, m_raw, codes, scale, vnorm,
                                                   enorm, raw, status, fixed_scale);
    return cudaGetLastError();
}

// Largest |v_j| over count floats, as float bits (nonnegative floats order
// like their bits; a NaN entry wins and makes the scale NaN, and the build
// then reports the non-finite row).
__global__ void maxabs_kernel(const float* __restrict__ v, int64_t count, unsigned int* out) {
    unsigned int m = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count; i += stride)
        m = max(m, __float_as_uint(fabsf(v[i])));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
    if ((threadIdx.x & 31) == 0 && m) atomicMax(out, m);
}

// s = RN(maxabs / 127), 1 for an all-zero corpus, 2^-149 if the quotient underflows.
__global__ void scale_from_maxabs_kernel(const unsigned int* maxabs_bits, float* s) {
    const float mx = __uint_as_float(*maxabs_bits);
    float v = 1.0f;
    if (mx != 0.0f) {
        v = __fdiv_rn(mx, 127.0f);
        if (v == 0.0f) v = __uint_as_float(1u);
    }
    *s = v;
}

cudaError_t launch_maxabs(const float* v, int64_t count, unsigned int* out, cudaStream_t st) {
    if (count <= 0) return cudaSuccess;
    int64_t blocks = (count + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    count_launches(1);
    maxabs_kernel<<<(unsigned)blocks, 256, 0, st>>>(v, count, out);
    return cudaGetLastError();
}

cudaError_t launch_scale_from_maxabs(const unsigned int* maxabs_bits, float* s, cudaStream_t st) {
    count_launches(1);
    scale_from_maxabs_kernel<<<1, 1, 0, st>>>(maxabs_bits, s);
    return cudaGetLastError();
}

// Queries: one block of kEncThreads per query, the quantizer of
// quantize_row_warp spread over its warps (maxima and exact integer sums do
// not depend on the order, so the results are bit-identical), plus the
// query-side scalars of App. A.1: ||s_q z_q|| rounded up and
// gamma_m = RU(a / RD(1 - a)), a = (8m + 64) 2^-23.
// q and qraw may be the same buffer (a host query staged in qraw): the raw
// copy, after every read of the first pass, rewrites the values it read.
constexpr int kEncThreads = 256;
constexpr int kEncWarps = kEncThreads / kWarp;

__global__ void __launch_bounds__(kEncThreads) encode_kernel(const float* q, int nq, int m,
                                                            int m_pad, int m_raw,
                                                            int8_t* __restrict__ zq, float* qraw,
                                                            QueryScalars* __restrict__ qs) {
    __shared__ float s_f[kEncWarps];
    __shared__ double s_d[kEncWarps];
    __shared__ long long s_a[kEncWarps], s_b[kEncWarps];
    __shared__ int s_i[kEncWarps];
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int qi = blockIdx.x;
    if (qi >= nq) return;
    const float* v = q + (int64_t)qi * m;
    int8_t* z = zq + (int64_t)qi * m_pad;
    auto block_max_f = [&](float x) {
        x = warp_max(x);
        if (lane == 0) s_f[warp] = x;
        __syncthreads();
        float r = s_f[0];
        for (int w = 1; w < kEncWarps; ++w) r = fmaxf(r, s_f[w]);
        __syncthreads();
        return r;
    };
    auto block_max_d = [&](double x) {
        x = warp_max(x);
        if (lane == 0) s_d[warp] = x;
        __syncthreads();
        double r = s_d[0];
        for (int w = 1; w < kEncWarps; ++w) r = fmax(r, s_d[w]);
        __syncthreads();
        return r;
    };
    auto block_sum2 = [&](long long& x, long long& y) {
        x = warp_sum(x);
        y = warp_sum(y);
        if (lane == 0) {
            s_a[warp] = x;
            s_b[warp] = y;
        }
        __syncthreads();
        x = 0;
        y = 0;
        for (int w = 0; w < kEncWarps; ++w) {
            x += s_a[w];
            y += s_b[w];
        }
        __syncthreads();
    };
    // finiteness and max |q_j|
    float maxabs = 0.0f;
    bool finite = true;
    for (int j = t; j < m; j += kEncThreads) {
        const float x = v[j];
        finite &= isfinite(x);
        maxabs = fmaxf(maxabs, fabsf(x));
    }
    finite = __all_sync(0xffffffffu, finite);
    if (lane == 0) s_i[warp] = finite;
    maxabs = block_max_f(maxabs);   // (its barrier publishes s_i)
    for (int w = 0; w < kEncWarps; ++w) finite &= s_i[w] != 0;
    for (int j = t; j < m_raw; j += kEncThreads) qraw[(int64_t)qi * m_raw + j] = j < m ? v[j] : 0.0f;
    QueryScalars out{};
    out.status = 0;
    if (finite) {
        float s;
        if (maxabs == 0.0f) {
            s = 1.0f;
        } else {
            s = __fdiv_rn(maxabs, 127.0f);
            if (s == 0.0f) s = __uint_as_float(1u);  // 2^-149
        }
        // codes and residual maximum (each thread later reads only its own codes)
        double emax = 0.0;
        for (int j = t; j < m_pad; j += kEncThreads) {
            int c = 0;
            if (j < m && maxabs != 0.0f) {
                const float tq = __fdiv_rn(v[j], s);
                float rt = roundf(tq);                     // half away from zero
                rt = fminf(fmaxf(rt, -127.0f), 127.0f);
                c = (int)rt;
                const double e = __dsub_rn((double)v[j], __dmul_rn((double)s, (double)c));  // exact
                emax = fmax(emax, fabs(e));
            }
            z[j] = (int8_t)c;
        }
        emax = block_max_d(emax);
        // norm bounds of q and of its residual
        long long Tv = 0, Te = 0;
        const int ev = maxabs > 0.0f ? norm_exponent((double)maxabs) : 0;
        const int ee = emax > 0.0 ? norm_exponent(emax) : 0;
        for (int j = t; j < m; j += kEncThreads) {
            const double x = (double)v[j];
            if (maxabs > 0.0f) Tv += norm_term(x, ev);
            if (emax > 0.0) {
                const int c = z[j];
                Te += norm_term(__dsub_rn(x, __dmul_rn((double)s, (double)c)), ee);
            }
        }
        block_sum2(Tv, Te);
        out.s = s;
        out.qnorm = norm_finish(Tv, ev);
        out.enorm = norm_finish(Te, ee);
        if (isinf(out.qnorm) || isinf(out.enorm)) out.status = PVS_ERR_OVERFLOW;
        // ||q_hat||: the values s z_j are exact in binary64
        double M = 0.0;
        for (int j = t; j < m; j += kEncThreads) M = fmax(M, fabs(__dmul_rn((double)s, (double)z[j])));
        M = block_max_d(M);
        long long T = 0, unused = 0;
        const int e = M > 0.0 ? norm_exponent(M) : 0;
        if (M > 0.0)
            for (int j = t; j < m; j += kEncThreads) T += norm_term(__dmul_rn((double)s, (double)z[j]), e);
        block_sum2(T, unused);
        out.qhat = norm_finish(T, e);
        if (out.status == 0 && isinf(out.qhat)) out.status = PVS_ERR_OVERFLOW;
    } else {
        out.status = PVS_ERR_NONFINITE;
    }
    if (t == 0) {
        const float a = (float)((8.0 * (double)m + 64.0) * 0x1p-23);   // exact
        out.gamma = __fdiv_ru(a, __fsub_rd(1.0f, a));
        qs[qi] = out;
    }
}

cudaError_t launch_encode_query(const float* q, int m, int m_pad, int m_raw, int8_t* zq,
                                float* qraw, QueryScalars* qs, cudaStream_t st) {
    count_launches(1);
    encode_kernel<<<1, kEncThreads, 0, st>>>(q, 1, m, m_pad, m_raw, zq, qraw, qs);
    return cudaGetLastError();
}

cudaError_t launch_encode_queries(const float* q, int nq, int m, int m_pad, int m_raw,
                                  int8_t* zq, float* qraw, QueryScalars* qs, cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    count_launches(1);
    encode_kernel<<<nq, kEncThreads, 0, st>>>(q, nq, m, m_pad, m_raw, zq, qraw, qs);
    return cudaGetLastError();
}

}  // namespace pvs
