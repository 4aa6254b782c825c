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
                                                    float* __restrict__ raw, int* status) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); row < n;
         row += warps) {
        const float* v = vecs + row * (int64_t)m;
        RowQuant r = quantize_row_warp(v, m, m_pad, codes + row * (int64_t)m_pad);
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
                         int* status, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    int64_t blocks = (n + 7) / 8;
    if (blocks > 152 * 64) blocks = 152 * 64;
    count_launches(1);
    build_kernel<<<(unsigned)blocks, 256, 0, st>>>(vecs, n, m, m_pad, m_raw, codes, scale, vnorm,
                                                   enorm, raw, status);
    return cudaGetLastError();
}

// Query encoding: the same quantizer, plus ||s_q z_q|| rounded up and
// gamma_m = RU(a / RD(1 - a)), a = (8m + 64) 2^-23 (App. A.1).
// q and qraw may be the same buffer (a host query staged in qraw): the raw
// copy then rewrites the values it read.
__global__ void encode_kernel(const float* q, int nq, int m, int m_pad, int m_raw,
                              int8_t* __restrict__ zq, float* qraw,
                              QueryScalars* __restrict__ qs) {
    const int lane = threadIdx.x & 31;
    const int qi = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (qi >= nq) return;
    const float* v = q + (int64_t)qi * m;
    int8_t* z = zq + (int64_t)qi * m_pad;
    RowQuant r = quantize_row_warp(v, m, m_pad, z);
    float* dst = qraw + (int64_t)qi * m_raw;
    for (int j = lane; j < m_raw; j += kWarp) dst[j] = j < m ? v[j] : 0.0f;
    __syncwarp();
    // ||q_hat||: values s_q z_j are exact in binary64
    float qhat = 0.0f;
    if (r.status == 0) {
        double M = 0.0;
        for (int j = lane; j < m; j += kWarp)
            M = fmax(M, fabs(__dmul_rn((double)r.s, (double)z[j])));
        M = warp_max(M);
        long long T = 0;
        int e = M > 0.0 ? norm_exponent(M) : 0;
        if (M > 0.0)
            for (int j = lane; j < m; j += kWarp)
                T += norm_term(__dmul_rn((double)r.s, (double)z[j]), e);
        T = warp_sum(T);
        qhat = norm_finish(T, e);
        if (isinf(qhat)) r.status = PVS_ERR_OVERFLOW;
    }
    if (lane == 0) {
        float a = (float)((8.0 * (double)m + 64.0) * 0x1p-23);   // exact
        float den = __fsub_rd(1.0f, a);
        QueryScalars out;
        out.s = r.s;
        out.qnorm = r.vnorm;
        out.qhat = qhat;
        out.enorm = r.enorm;
        out.gamma = __fdiv_ru(a, den);
        out.status = r.status;
        qs[qi] = out;
    }
}

cudaError_t launch_encode_query(const float* q, int m, int m_pad, int m_raw, int8_t* zq,
                                float* qraw, QueryScalars* qs, cudaStream_t st) {
    count_launches(1);
    encode_kernel<<<1, 32, 0, st>>>(q, 1, m, m_pad, m_raw, zq, qraw, qs);
    return cudaGetLastError();
}

cudaError_t launch_encode_queries(const float* q, int nq, int m, int m_pad, int m_raw,
                                  int8_t* zq, float* qraw, QueryScalars* qs, cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    count_launches(1);
    // one warp per block: the queries spread over every SM (their norm bounds
    // use binary64, whose per-SM rate is low on this part)
    encode_kernel<<<nq, 32, 0, st>>>(q, nq, m, m_pad, m_raw, zq, qraw, qs);
    return cudaGetLastError();
}

}  // namespace pvs
