// pvs_rank_exact_noalloc: exact top-n ranking of a caller-held set of vectors
// that performs no device memory allocation.
//
// It is the score-key-sort part of a pull (exact scores -> 64-bit rank keys
// -> descending sort -> emit), run over vectors the caller already holds on
// the device, with the rank keys kept in one file-scope static device array
// instead of memory obtained from cudaMalloc.  Some callers cannot allocate
// device memory at the point where they need a ranking: services whose
// device memory is owned by their own pool or budget, where an allocation
// outside the pool either fails or breaks its accounting, and
// latency-critical callers, for whom cudaMalloc can take milliseconds and
// cudaFree waits for the whole device to go idle.
//
// The scratch array: PVS_NOALLOC_MAX_VECTORS 64-bit keys plus one status word
// (64 KiB + 256 B).  Every GPU that loads this library holds it until the
// process exits.  Every call on a device uses the same array and leaves its
// keys behind; the status word is cleared at the start of each call, and no
// key is read that the same call did not write.  Calls whose device work
// overlaps (for example on two streams at once) race on the array.
//
// Host code must not use the array's name as a device address: the symbol is
// a host-side stand-in.  The device address is fetched once per device with
// cudaGetSymbolAddress, during the first call made with that device current.
// That first call should therefore come before any stream capture begins.
#include <mutex>

#include "exact_dot.cuh"
#include "kernels.h"
#include "pvs_common.cuh"

namespace pvs {

constexpr int kNoAllocMax = PVS_NOALLOC_MAX_VECTORS;
constexpr int kNoAllocStatusSlot = kNoAllocMax;            // key slots, then the status
constexpr int kNoAllocSlots = kNoAllocMax + 32;           // 256 B of status padding

static __device__ __align__(256) unsigned long long g_noalloc_scratch[kNoAllocSlots];

// One warp per vector: finite check, exact score, rank key into scratch.
__global__ void __launch_bounds__(256) noalloc_score_kernel(const float* __restrict__ q,
                                                            const float* __restrict__ vecs,
                                                            int n, int dim,
                                                            unsigned long long* scratch) {
    const int lane = threadIdx.x & 31;
    const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (i >= n) return;
    const float* v = vecs + (int64_t)i * dim;
    bool finite = true;
    for (int j = lane; j < dim; j += kWarp) finite &= isfinite(q[j]) && isfinite(v[j]);
    finite = __all_sync(0xffffffffu, finite);
    int* status = reinterpret_cast<int*>(scratch + kNoAllocStatusSlot);
    if (!finite) {
        if (lane == 0) {
            set_status(status, PVS_ERR_NONFINITE);
            scratch[i] = 0ull;
        }
        return;
    }
    bool fb;
    const float s = exact_dot_warp_any(q, v, dim, &fb);
    if (lane == 0) {
        if (!isfinite(s)) set_status(status, PVS_ERR_OVERFLOW);
        scratch[i] = rank_key(s, (uint32_t)i);
    }
}

// One CTA: bitonic sort of the n keys (descending), then the first `top` out.
__global__ void __launch_bounds__(1024) noalloc_sort_emit_kernel(
    const unsigned long long* __restrict__ scratch, int n, int pow2, int top, int64_t* out_ids,
    float* out_scores) {
    extern __shared__ unsigned long long sk[];
    for (int i = threadIdx.x; i < pow2; i += blockDim.x) sk[i] = i < n ? scratch[i] : 0ull;
    __syncthreads();
    for (int size = 2; size <= pow2; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = threadIdx.x; i < pow2 / 2; i += blockDim.x) {
                const int a = 2 * i - (i & (stride - 1));
                const int b = a + stride;
                const bool desc = (a & size) == 0;
                const unsigned long long x = sk[a], y = sk[b];
                if ((x < y) == desc) {
                    sk[a] = y;
                    sk[b] = x;
                }
            }
            __syncthreads();
        }
    }
    for (int i = threadIdx.x; i < top; i += blockDim.x) {
        out_ids[i] = rank_key_id(sk[i]);
        out_scores[i] = rank_key_score(sk[i]);
    }
}

namespace {

constexpr int kMaxDevices = 256;
std::mutex g_setup_mutex;
unsigned long long* g_scratch_addr[kMaxDevices] = {nullptr};

// Device address of the scratch array for the current device (set up once).
cudaError_t scratch_address(unsigned long long** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(noalloc_sort_emit_kernel,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kNoAllocMax * (int)sizeof(unsigned long long));
        if (e != cudaSuccess) return e;
        g_scratch_addr[dev] = static_cast<unsigned long long*>(p);
    }
    *out = g_scratch_addr[dev];
    return cudaSuccess;
}

bool on_device(const void* p) {
    cudaPointerAttributes a;
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

}  // namespace
}  // namespace pvs

extern "C" pvs_status pvs_rank_exact_noalloc(const float* query, const float* vecs, int32_t n,
                                             int32_t dim, int32_t top, int64_t* out_ids,
                                             float* out_scores, void* cuda_stream) {
    using namespace pvs;
    if (n < 0 || n > kNoAllocMax || dim < 1 || dim > kMaxDim || top < 0 || top > n)
        return PVS_ERR_INVALID;
    if (!query || !on_device(query)) return PVS_ERR_INVALID;
    if (n > 0 && (!vecs || !on_device(vecs))) return PVS_ERR_INVALID;
    if (top > 0 && (!out_ids || !out_scores || !on_device(out_ids) || !on_device(out_scores)))
        return PVS_ERR_INVALID;
    unsigned long long* scratch = nullptr;
    cudaError_t e = scratch_address(&scratch);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return PVS_ERR_CUDA;
    }
    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    e = cudaMemsetAsync(scratch + kNoAllocStatusSlot, 0, sizeof(unsigned long long), st);
    if (e == cudaSuccess && n > 0) {
        count_launches(1);
        noalloc_score_kernel<<<(n + 7) / 8, 256, 0, st>>>(query, vecs, n, dim, scratch);
        e = cudaGetLastError();
    }
    if (e == cudaSuccess && top > 0) {
        int pow2 = 1;
        while (pow2 < n) pow2 <<= 1;
        count_launches(1);
        noalloc_sort_emit_kernel<<<1, 1024, pow2 * sizeof(unsigned long long), st>>>(
            scratch, n, pow2, top, out_ids, out_scores);
        e = cudaGetLastError();
    }
    unsigned long long status = 0;
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(&status, scratch + kNoAllocStatusSlot, sizeof(status),
                            cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return PVS_ERR_CUDA;
    }
    return (pvs_status)(int)(status & 0xffffffffull);
}
