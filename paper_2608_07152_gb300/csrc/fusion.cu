// Complete-list weighted RRF on the device: the fallback of EAHR's adaptive
// policy when both ranked lists must be read deep (arXiv 2608.07152, Sec. 2.1
// defines T*_K over the complete lists; Sec. 2.2's last paragraph notes that
// when early determination is impossible, fusing the complete lists gives
// the same result).
//
// Steps, one request, on the dense cursor's stream:
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
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

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

}  // namespace pvs
