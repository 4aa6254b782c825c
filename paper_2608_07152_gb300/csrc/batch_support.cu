// Small kernels around the batched interval pass: corpus maxima of the norm
// bounds, the per-query upper bound rmax_q of the interval half-width (the
// cheap pre-filter of the filter pass), copying batch-encoded queries into the
// cursors' own buffers, carrying a working set's state (resolved scores,
// delivered items) into freshly computed full bounds when a cursor rescans,
// and gathering the status words and counters of many cursors so that a
// batch is checked with one copy and one synchronisation.
#include "kernels.h"
#include "pvs_common.cuh"

namespace pvs {

// out[0] = max vnorm, out[1] = max enorm over rows [0, rows); out zeroed by
// the caller.  Non-negative floats order like their bit patterns.
__global__ void norm_max_kernel(const float* __restrict__ vnorm, const float* __restrict__ enorm,
                                int64_t rows, unsigned int* out) {
    float mv = 0.0f, me = 0.0f;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < rows; i += stride) {
        mv = fmaxf(mv, vnorm[i]);
        me = fmaxf(me, enorm[i]);
    }
    mv = warp_max(mv);
    me = warp_max(me);
    if ((threadIdx.x & 31) == 0) {
        atomicMax(&out[0], __float_as_uint(mv));
        atomicMax(&out[1], __float_as_uint(me));
    }
}

cudaError_t launch_norm_max(const float* vnorm, const float* enorm, int64_t rows,
                            unsigned int* out, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(out, 0, 2 * sizeof(unsigned int), st);
    if (e != cudaSuccess || rows <= 0) return e;
    int64_t blocks = (rows + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    count_launches(1);
    norm_max_kernel<<<(unsigned)blocks, 256, 0, st>>>(vnorm, enorm, rows, out);
    return cudaGetLastError();
}

// rmax_q >= RU(E + G) for every row: each factor of the interval formula is
// replaced by its corpus maximum (vnorm, enorm) and |c| by an upper bound of
// |q_hat . v_hat| <= ||q_hat|| (||v|| + ||e_v||), times (1 + 2^-21) for the two
// roundings of the centre; all operations round up and are monotone.
__global__ void rmax_kernel(const QueryScalars* qs, int nq, const unsigned int* maxes,
                            float* rmax) {
    const int q = blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= nq) return;
    const QueryScalars s = qs[q];
    const float vmax = __uint_as_float(maxes[0]), emax = __uint_as_float(maxes[1]);
    const float E = __fadd_ru(__fmul_ru(s.enorm, vmax), __fmul_ru(s.qhat, emax));
    const float cmax = __fmul_ru(__fmul_ru(s.qhat, __fadd_ru(vmax, emax)), 1.0f + 0x1p-21f);
    const float G = __fmul_ru(__fadd_ru(__fadd_ru(cmax, E), __fmul_ru(s.qnorm, vmax)), s.gamma);
    rmax[q] = __fadd_ru(E, G);
}

cudaError_t launch_rmax(const QueryScalars* qs, int nq, const unsigned int* maxes, float* rmax,
                        cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    count_launches(1);
    rmax_kernel<<<(nq + 127) / 128, 128, 0, st>>>(qs, nq, maxes, rmax);
    return cudaGetLastError();
}

// Block q copies query q's encoding from the batch buffers to its cursor.
__global__ void copy_query_kernel(const int8_t* __restrict__ zq_b, const float* __restrict__ qraw_b,
                                  const QueryScalars* __restrict__ qs_b, const QueryDst* dst,
                                  int m_pad, int m_raw) {
    const int q = blockIdx.x;
    const QueryDst d = dst[q];
    for (int j = threadIdx.x; j < m_pad; j += blockDim.x) d.zq[j] = zq_b[(int64_t)q * m_pad + j];
    for (int j = threadIdx.x; j < m_raw; j += blockDim.x) d.qraw[j] = qraw_b[(int64_t)q * m_raw + j];
    if (threadIdx.x == 0) {
        *d.qs = qs_b[q];
        *d.ctr = DevCounters{};
        *d.status = 0;
    }
}

cudaError_t launch_copy_queries(const int8_t* zq_b, const float* qraw_b, const QueryScalars* qs_b,
                                const QueryDst* dst, int nq, int m_pad, int m_raw,
                                cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    count_launches(1);
    copy_query_kernel<<<nq, 256, 0, st>>>(zq_b, qraw_b, qs_b, dst, m_pad, m_raw);
    return cudaGetLastError();
}

// Working-set state into fresh full bounds: delivered items become -inf,
// scored items carry their exact score.
__global__ void scatter_ws_kernel(const int32_t* __restrict__ w_id, const float* __restrict__ w_lo,
                                  const float* __restrict__ w_hi, const unsigned int* w_len,
                                  float* lo, float* hi) {
    const int64_t n = *w_len;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        const float l = w_lo[i], h = w_hi[i];
        const int32_t id = w_id[i];
        if (l == -INFINITY) {
            lo[id] = -INFINITY;
            hi[id] = -INFINITY;
        } else if (l == h) {
            lo[id] = l;
            hi[id] = h;
        }
    }
}

cudaError_t launch_scatter_ws(const int32_t* w_id, const float* w_lo, const float* w_hi,
                              const unsigned int* w_len, float* lo, float* hi, int grid,
                              cudaStream_t st) {
    count_launches(1);
    scatter_ws_kernel<<<grid, 256, 0, st>>>(w_id, w_lo, w_hi, w_len, lo, hi);
    return cudaGetLastError();
}

__global__ void gather_state_kernel(const CursorRef* __restrict__ refs, int n, int* status_out,
                                    DevCounters* ctr_out) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    status_out[i] = *refs[i].status;
    if (ctr_out) ctr_out[i] = *refs[i].ctr;
}

cudaError_t launch_gather_state(const CursorRef* refs, int n, int* status_out,
                                DevCounters* ctr_out, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    count_launches(1);
    gather_state_kernel<<<(n + 255) / 256, 256, 0, st>>>(refs, n, status_out, ctr_out);
    return cudaGetLastError();
}

}  // namespace pvs
