// PVS pull without a host round trip (Sec. 2.3.1 incremental ranking,
// Sec. 2.1 exact prefix): three launches turn the cursor's working set into
// the next n exact ranks.
//   1. tau = n-th largest lower bound among live working-set entries: radix
//      select over ordered float keys, 11/11/10-bit digits, shared-memory
//      histograms updated once per distinct digit per warp (match.any);
//   2. candidates = live entries with hi >= tau (a superset of every item that
//      can hold one of the next n ranks), compacted with warp ballots;
//   3. every unresolved candidate (lo < hi) is scored exactly, one warp each
//      on every SM (refine_kernel: the binary64 arithmetic is slow per SM on
//      this part, so it is spread over the whole GPU), checked against its
//      interval (App. A.1) and marked resolved (lo = hi = score) in the
//      working set and the full bounds;
//   4. the candidates' rank keys (score desc, id asc) are sorted in shared
//      memory (bitonic, up to kPullSortCap); a larger candidate set first
//      selects its n largest keys with a 64-bit radix select;
//   5. the first n keys are written out and marked emitted (-inf).
// Steps 1-2 and 4-5 each run in one CTA of 512 threads (<= 64 registers each)
// with ~25 KB of shared memory, so they fit on an SM beside another cursor's
// interval-pass CTA.
#include "exact_dot.cuh"
#include "kernels.h"
#include "pvs_common.cuh"

namespace pvs {

constexpr int kPullThreads = 512;   // 32K registers: fits beside an interval-pass CTA
constexpr int kPullWarps = kPullThreads / 32;
constexpr int kPullSortCap = 2048;
constexpr int kHistBins = 2048;

struct PullShared {
    unsigned int hist[kHistBins];
    unsigned long long sk[kPullSortCap];
    unsigned int warp_tot[kPullWarps];
    unsigned long long prefix;
    unsigned long long k;
    unsigned int count;
    int ok;
};

// Block-wide: digit d with count(digits > d) < k <= count(digits >= d);
// updates sh.prefix / sh.k.  Thread t owns bins [kBinsPerThread t, +kBinsPerThread).
constexpr int kBinsPerThread = kHistBins / kPullThreads;
__device__ inline void block_pick_digit(PullShared& sh, int shift) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int b0 = kBinsPerThread * t;
    unsigned int x = 0;
#pragma unroll
    for (int b = 0; b < kBinsPerThread; ++b) x += sh.hist[b0 + b];
    const unsigned int own = x;
    // inclusive suffix scan within the warp (lanes >= lane)
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned int v = __shfl_down_sync(0xffffffffu, x, o);
        if (lane + o < 32) x += v;
    }
    if (lane == 0) sh.warp_tot[warp] = x;
    __syncthreads();
    unsigned int above_warps = 0;
    for (int w = warp + 1; w < kPullWarps; ++w) above_warps += sh.warp_tot[w];
    const unsigned long long incl = (unsigned long long)x + above_warps;   // bins >= b0
    const unsigned long long above = incl - own;                          // bins past mine
    const unsigned long long k = sh.k;
    __syncthreads();
    if (above < k && k <= incl) {
        unsigned long long acc = above;
        for (int b = kBinsPerThread - 1; b >= 0; --b) {
            const unsigned int h = sh.hist[b0 + b];
            if (acc + h >= k) {
                sh.prefix |= (unsigned long long)(b0 + b) << shift;
                sh.k = k - acc;
                break;
            }
            acc += h;
        }
        sh.ok = 1;
    }
    __syncthreads();
}

// Histogram of digit (key >> shift) & dmask over keys that match the prefix
// above `shift + bits`.  Keys come from a functor: valid(i) / key(i).
template <typename KeyT, typename Src>
__device__ inline void block_histogram(PullShared& sh, unsigned int len, int shift, int bits,
                                       KeyT prefix, Src src) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    for (int i = t; i < kHistBins; i += kPullThreads) sh.hist[i] = 0;
    __syncthreads();
    const int top = shift + bits;
    const KeyT hmask = top >= (int)(8 * sizeof(KeyT)) ? (KeyT)0 : ~(KeyT)0 << top;
    const unsigned int dmask = (1u << bits) - 1u;
    for (unsigned int i0 = warp * 32; i0 < len; i0 += kPullThreads) {
        const unsigned int i = i0 + lane;
        KeyT key = 0;
        bool valid = i < len && src.valid(i);
        if (valid) {
            key = src.key(i);
            valid = (key & hmask) == (prefix & hmask);
        }
        const unsigned int d = valid ? (unsigned int)((key >> shift) & dmask) : (0x10000u + lane);
        const unsigned int peers = __match_any_sync(0xffffffffu, d);
        if (valid && lane == __ffs(peers) - 1) atomicAdd(&sh.hist[d], (unsigned int)__popc(peers));
    }
    __syncthreads();
}

struct LoKeys {
    const float* w_lo;
    __device__ bool valid(unsigned int i) const { return w_lo[i] != -INFINITY; }
    __device__ uint32_t key(unsigned int i) const { return fkey(w_lo[i]); }
};

struct CandKeys {
    const unsigned long long* keys;
    __device__ bool valid(unsigned int) const { return true; }
    __device__ unsigned long long key(unsigned int i) const { return keys[i]; }
};

__device__ inline void bitonic_desc_smem(unsigned long long* sk, int pow2) {
    for (int size = 2; size <= pow2; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = threadIdx.x; i < pow2 / 2; i += kPullThreads) {
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
}

// Steps 1-2 (one CTA): tau and the candidate list; the count goes to
// ctr->cand for the refinement and emission launches.
__global__ void __launch_bounds__(kPullThreads, 2) pull_select_kernel(PullArgs a) {
    __shared__ PullShared sh;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const unsigned int len = *a.w_len;
    const int n = a.n;
    if (t == 0) {
        sh.prefix = 0;
        sh.k = (unsigned long long)n;
        sh.count = 0;
    }
    __syncthreads();
    const LoKeys lok{a.w_lo};
    const int shifts32[3] = {21, 10, 0}, bits32[3] = {11, 11, 10};
    for (int p = 0; p < 3; ++p) {
        block_histogram<uint32_t>(sh, len, shifts32[p], bits32[p], (uint32_t)sh.prefix, lok);
        if (t == 0) sh.ok = 0;
        __syncthreads();
        block_pick_digit(sh, shifts32[p]);
        if (!sh.ok) {  // fewer than n live entries: the working set was too small
            if (t == 0) {
                set_status(a.status, PVS_ERR_INVALID);
                a.ctr->cand = 0;
            }
            return;
        }
    }
    const uint32_t tau = (uint32_t)sh.prefix;
    for (unsigned int i0 = warp * 32; i0 < len; i0 += kPullThreads) {
        const unsigned int i = i0 + lane;
        const bool f = i < len && a.w_lo[i] != -INFINITY && fkey(a.w_hi[i]) >= tau;
        const unsigned int bal = __ballot_sync(0xffffffffu, f);
        unsigned int base = 0;
        if (lane == 0 && bal) base = atomicAdd(&sh.count, (unsigned int)__popc(bal));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (f) a.cand[base + __popc(bal & ((1u << lane) - 1u))] = (int32_t)i;
    }
    __syncthreads();
    if (t == 0) {
        a.ctr->cand = sh.count;
        a.ctr->cand_total += sh.count;
    }
}

// Steps 4-5 (one CTA): order the candidates (all scored by now) and emit the
// first n.
__global__ void __launch_bounds__(kPullThreads, 2) pull_emit_kernel(PullArgs a) {
    __shared__ PullShared sh;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const unsigned int c = a.ctr->cand;
    const int n = a.n;
    if (c < (unsigned int)n) {      // only after a failure recorded by the select step
        if (t == 0) set_status(a.status, PVS_ERR_INVALID);
        return;
    }
    int m;   // keys in sh.sk to sort
    if (c <= (unsigned int)kPullSortCap) {
        for (unsigned int j = t; j < c; j += kPullThreads) {
            const int32_t w = a.cand[j];
            sh.sk[j] = rank_key(a.w_lo[w], (uint32_t)w);
        }
        m = (int)c;
    } else {
        for (unsigned int j = t; j < c; j += kPullThreads) {
            const int32_t w = a.cand[j];
            a.keys[j] = rank_key(a.w_lo[w], (uint32_t)w);
        }
        if (t == 0) {
            sh.prefix = 0;
            sh.k = (unsigned long long)n;
        }
        __syncthreads();
        const CandKeys ck{a.keys};
        const int shifts64[6] = {53, 42, 31, 20, 9, 0}, bits64[6] = {11, 11, 11, 11, 11, 9};
        for (int p = 0; p < 6; ++p) {
            block_histogram<unsigned long long>(sh, c, shifts64[p], bits64[p], sh.prefix, ck);
            block_pick_digit(sh, shifts64[p]);
        }
        const unsigned long long kth = sh.prefix;   // keys are unique: exactly n keys >= kth
        if (t == 0) sh.count = 0;
        __syncthreads();
        for (unsigned int i0 = warp * 32; i0 < c; i0 += kPullThreads) {
            const unsigned int i = i0 + lane;
            const unsigned long long kv = i < c ? a.keys[i] : 0ull;
            const bool f = i < c && kv >= kth;
            const unsigned int bal = __ballot_sync(0xffffffffu, f);
            unsigned int base = 0;
            if (lane == 0 && bal) base = atomicAdd(&sh.count, (unsigned int)__popc(bal));
            base = __shfl_sync(0xffffffffu, base, 0);
            const unsigned int pos = base + __popc(bal & ((1u << lane) - 1u));
            if (f && pos < (unsigned int)kPullSortCap) sh.sk[pos] = kv;
        }
        __syncthreads();
        m = n;
    }
    int pow2 = 1;
    while (pow2 < m) pow2 <<= 1;
    for (int j = m + t; j < pow2; j += kPullThreads) sh.sk[j] = 0ull;
    __syncthreads();
    bitonic_desc_smem(sh.sk, pow2);
    for (int r = t; r < n; r += kPullThreads) {
        const unsigned long long k = sh.sk[r];
        const uint32_t w = rank_key_id(k);
        const int32_t id = a.w_id[w];
        a.out_ids[r] = id;
        a.out_scores[r] = rank_key_score(k);
        a.w_lo[w] = -INFINITY;
        a.w_hi[w] = -INFINITY;
        a.lo[id] = -INFINITY;
        a.hi[id] = -INFINITY;
    }
}

cudaError_t launch_pull_fused(const PullArgs& a, int refine_grid, cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    if (a.n > kPullFusedMax) return cudaErrorInvalidValue;
    count_launches(1);
    pull_select_kernel<<<1, kPullThreads, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // step 3: exact scores of the unresolved candidates on every SM
    e = launch_refine(a.cand, &a.ctr->cand, a.w_id, a.w_lo, a.w_hi, a.lo, a.hi, a.qraw, a.raw,
                      a.m_raw, a.status, a.ctr, refine_grid, st);
    if (e != cudaSuccess) return e;
    count_launches(1);
    pull_emit_kernel<<<1, kPullThreads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace pvs
