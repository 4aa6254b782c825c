// PVS pulls without a host round trip (Sec. 2.3.1 incremental ranking,
// Sec. 2.1 exact prefix): the cursor's working set becomes the next n exact
// ranks in these steps:
//   1. tau = n-th largest lower bound among live working-set entries;
//   2. candidates = live entries with hi >= tau (a superset of every item that
//      can hold one of the next n ranks);
//   3. every unresolved candidate (lo < hi) is scored exactly
//      (exact_dot.cuh), checked against its interval (App. A.1) and marked
//      resolved (lo = hi = score) in the working set and the full bounds;
//   4. the candidates are ordered by rank key (score desc, id asc);
//   5. the first n are written out and marked emitted (-inf).
// Two forms:
//   * three launches (the first pull of a fresh working set, which refines
//     most of it, and every batched first pull): one CTA selects by radix
//     select over ordered float keys (11/11/10-bit digits, shared-memory
//     histograms, match.any aggregation), refinement runs on every SM
//     (refine_kernels.cu), one CTA orders and emits;
//   * one cluster launch (every later pull): each CTA of the cluster selects
//     from the cursor's frontier or the whole working set, the CTAs split the
//     refinement, and CTA 0 emits after a cluster barrier.
// Every CTA has 512 threads (<= 64 registers) and ~25 KB of shared memory, so
// it fits on an SM beside another cursor's interval-pass CTA.
#include "exact_dot.cuh"
#include <vector>

#include "kernels.h"
#include "pipeline.cuh"
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
    unsigned int cand_n;
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
    constexpr int kUnroll = 4;   // loads in flight per thread before the histogram updates
    for (unsigned int i0 = warp * 32; i0 < len; i0 += kPullThreads * kUnroll) {
        KeyT key[kUnroll];
        bool valid[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const unsigned int i = i0 + u * kPullThreads + lane;
            valid[u] = i < len && src.valid(i);
            key[u] = valid[u] ? src.key(i) : (KeyT)0;
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const bool v = valid[u] && (key[u] & hmask) == (prefix & hmask);
            const unsigned int d = v ? (unsigned int)((key[u] >> shift) & dmask) : (0x10000u + lane);
            const unsigned int peers = __match_any_sync(0xffffffffu, d);
            if (v && lane == __ffs(peers) - 1) atomicAdd(&sh.hist[d], (unsigned int)__popc(peers));
        }
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
__device__ inline void pull_select_body(const PullArgs& a, PullShared& sh) {
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
#pragma unroll 4
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

__global__ void __launch_bounds__(kPullThreads, 2) pull_select_kernel(PullArgs a) {
    __shared__ PullShared sh;
    pull_select_body(a, sh);
}

// One CTA per cursor.
__global__ void __launch_bounds__(kPullThreads, 2)
    pull_select_batch_kernel(const __grid_constant__ PullArgsPack p) {
    __shared__ PullShared sh;
    pull_select_body(p.a[blockIdx.x], sh);
}

// Sort the m keys in sh.sk (descending) and emit the first n: ids, scores,
// and -inf bounds for the delivered rows.
__device__ inline void emit_sorted(const PullArgs& a, PullShared& sh, int m) {
    const int t = threadIdx.x;
    const int n = a.n;
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
        if (a.lo) {
            a.lo[id] = -INFINITY;
            a.hi[id] = -INFINITY;
        }
    }
}

// More than kPullSortCap candidates (a list in global memory; the selection
// uses sh.hist): keys to a.keys, radix selection of the n-th largest key,
// the n largest into sh.sk.  Out of line: rare, and register-hungry.
static __device__ __noinline__ void emit_many(const PullArgs& a, PullShared& sh,
                                              const int32_t* cand, unsigned int c) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int n = a.n;
    for (unsigned int j = t; j < c; j += kPullThreads) {
        const int32_t w = cand[j];
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
    emit_sorted(a, sh, n);
}

// Steps 4-5 (one CTA): order the candidates (all scored by now) and emit the
// first n.
__device__ inline void pull_emit_list(const PullArgs& a, PullShared& sh, const int32_t* cand,
                                      unsigned int c) {
    const int t = threadIdx.x;
    if (c < (unsigned int)a.n) {      // only after a failure recorded by the select step
        if (t == 0) set_status(a.status, PVS_ERR_INVALID);
        return;
    }
    if (c > (unsigned int)kPullSortCap) {
        emit_many(a, sh, cand, c);
        return;
    }
    if (c <= (unsigned int)kPullThreads) {
        // one candidate per thread: its rank is the number of larger keys (keys
        // are unique), and its id is loaded with its score
        unsigned long long key = 0;
        int32_t w = 0, id = 0;
        if (t < (int)c) {
            w = cand[t];
            const float sc = a.w_lo[w];
            id = a.w_id[w];
            key = rank_key(sc, (uint32_t)w);
            sh.sk[t] = key;
        }
        __syncthreads();
        if (t < (int)c) {
            unsigned int r = 0;
            for (unsigned int f = 0; f < c; ++f) r += sh.sk[f] > key;
            if (r < (unsigned int)a.n) {
                a.out_ids[r] = id;
                a.out_scores[r] = rank_key_score(key);
                a.w_lo[w] = -INFINITY;
                a.w_hi[w] = -INFINITY;
                if (a.lo) {
                    a.lo[id] = -INFINITY;
                    a.hi[id] = -INFINITY;
                }
            }
        }
        return;
    }
    for (unsigned int j = t; j < c; j += kPullThreads) {
        const int32_t w = cand[j];
        sh.sk[j] = rank_key(a.w_lo[w], (uint32_t)w);
    }
    emit_sorted(a, sh, (int)c);
}

// The status word as it stands after a pull, into the caller's pinned host
// word (host-buffer pulls then need no separate copy).
// Publishes the status word to pinned host memory last: the host may poll it
// instead of synchronising, so the block's output writes are made visible to
// the host first.
__device__ inline void mirror_status(const PullArgs& a) {
    __syncthreads();
    if (threadIdx.x == 0 && a.status_mirror) {
        __threadfence_system();
        *reinterpret_cast<volatile int*>(a.status_mirror) = *reinterpret_cast<volatile int*>(a.status);
    }
}

__device__ inline void pull_emit_body(const PullArgs& a, PullShared& sh) {
    if (threadIdx.x == 0) a.ctr->front_k = 0;   // rows leave without the frontier's count
    pull_emit_list(a, sh, a.cand, a.ctr->cand);
    mirror_status(a);
}

__global__ void __launch_bounds__(kPullThreads, 2) pull_emit_kernel(PullArgs a) {
    __shared__ PullShared sh;
    pull_emit_body(a, sh);
}

__global__ void __launch_bounds__(kPullThreads, 2)
    pull_emit_batch_kernel(const __grid_constant__ PullArgsPack p) {
    __shared__ PullShared sh;
    pull_emit_body(p.a[blockIdx.x], sh);
}

// ---- one launch per pull: a cluster of CTAs per cursor -------------------------
// Every CTA of the cluster derives tau and the candidate list itself (the same
// set; its order may differ), refines the candidates it owns (working-set
// index modulo the cluster's warps), and after a cluster barrier with
// release / acquire semantics CTA 0 orders the candidates and emits.
//   tau: every thread takes the largest live lower bound of its share; in
//   every warp the j-th largest of these, j = ceil(n / warps), bounds the
//   answer from below, and so does t0, their minimum (each warp holds j values
//   >= t0).  One more pass gathers the live rows with hi >= t0 (every row with
//   lo >= t0 among them); tau is the n-th largest lower bound of the gathered
//   rows and the candidates are those with hi >= tau.  If more rows than
//   kPullSortCap reach t0, CTA 0 runs the radix selection instead.
constexpr int kPullCluster = 8;        // single cursor: the whole pull in one cluster of 8
constexpr int kPullClusterBatch = 2;   // batched pulls: many cursors at once, 2 CTAs each


// Rows whose lower bound may reach the frontier bound: kFrontMult times the
// ranks of the pull that builds it (the frontier then serves later pulls).
constexpr int kFrontMult = 6;
// The gather keeps working-set indices only (in the bytes of sh.sk): twice the
// rows of (key, index) pairs in the same shared memory.
constexpr int kGatherCap = kPullSortCap * 2;
static_assert(kFrontCap == kGatherCap, "the frontier is the gathered set");

struct FastSelect {
    int mode;            // 1: list in sh.hist (sh.cand_n entries); 0: radix fallback; -1: < n live
    bool from_front;     // the rows came from the carried frontier
    bool new_front;      // a whole-set gather at a wide bound: it can become the frontier
    uint32_t t0;         // the bound of the gather
    unsigned int g;      // rows gathered (hi >= t0)
    unsigned int l;      // of them with lo >= t0
    unsigned int mult;   // the gather's bound was for mult * n rows (1: the tight bound)
};

// Gather, with one shared-memory atomic per row that reaches t0 (few do),
// the working-set indices of the live rows with hi >= t0 into the bytes of
// sh.sk (count sh.count, capacity kGatherCap) and the lo keys of those with
// lo >= t0 into sh.hist (count sh.cand_n, capacity kPullSortCap).
// Rows: the frontier's len entries, or working-set indices 0 .. len-1.
__device__ inline void gather_rows(const PullArgs& a, PullShared& sh, bool from_front,
                                   unsigned int len, uint32_t t0) {
    const int t = threadIdx.x;
    auto take = [&](float l, float h, unsigned int i) {
        if (l == -INFINITY) return;
        const uint32_t hk = fkey(h);
        if (hk < t0) return;
        const unsigned int pos = atomicAdd(&sh.count, 1u);
        if (pos < (unsigned int)kGatherCap) reinterpret_cast<uint32_t*>(sh.sk)[pos] = i;
        const uint32_t lk = fkey(l);
        if (lk >= t0) {
            const unsigned int q = atomicAdd(&sh.cand_n, 1u);
            if (q < (unsigned int)kPullSortCap) sh.hist[q] = lk;
        }
    };
    if (from_front) {
        for (unsigned int e = t; e < len; e += kPullThreads) {
            const int32_t w = a.front[e];
            take(a.w_lo[w], a.w_hi[w], (unsigned int)w);
        }
    } else {
        const unsigned int len4 = len >> 2;   // working-set arrays are 16-byte aligned
        const float4* lo4 = reinterpret_cast<const float4*>(a.w_lo);
        const float4* hi4 = reinterpret_cast<const float4*>(a.w_hi);
#pragma unroll 4
        for (unsigned int i = t; i < len4; i += kPullThreads) {
            const float4 l = lo4[i], h = hi4[i];
            take(l.x, h.x, 4 * i);
            take(l.y, h.y, 4 * i + 1);
            take(l.z, h.z, 4 * i + 2);
            take(l.w, h.w, 4 * i + 3);
        }
        for (unsigned int i = 4 * len4 + t; i < len; i += kPullThreads) take(a.w_lo[i], a.w_hi[i], i);
    }
    __syncthreads();
}

// Selection for the one-launch pull; every CTA of the cluster reaches the
// same outcome.  Rows come from the frontier when it still holds at least n
// rows with lo >= its bound, else from the whole working set (then t0 comes
// from the per-thread maxima, for kFrontMult * n ranks).  Gathered: (hi key,
// index) of the rows with hi >= t0 in sh.sk; lo keys of those with lo >= t0
// in sh.hist, among which tau is the n-th largest.
__device__ inline FastSelect pull_select_fast(const PullArgs& a, PullShared& sh) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int n = a.n;
    FastSelect r{1, false, false, 0u, 0u, 0u, 1u};
    const unsigned int fk = a.ctr->front_k;
    r.from_front = a.front != nullptr && fk >= (unsigned int)n;
    r.new_front = !r.from_front && a.front != nullptr;
    unsigned int len;
    // whole-set pass: bounds for mult * n rows, widest first; the cursor's hint
    // (front_hint) starts deep cursors, whose wide gathers overflow, lower
    const unsigned int hint = a.ctr->front_hint == 3u ? 3u : (unsigned int)kFrontMult;
    uint32_t t0_mid = 0, t0_tight = 0;
    if (r.from_front) {
        len = a.ctr->front_n;
        r.t0 = a.ctr->front_bound;
        if (t == 0) {
            sh.count = 0;
            sh.cand_n = 0;
            sh.ok = 0;
        }
        __syncthreads();
    } else {
        len = *a.w_len;
        uint32_t mx = 0;   // 0: no live row (every live key is larger)
        auto live_key = [](float l) -> uint32_t { return l == -INFINITY ? 0u : fkey(l); };
        const unsigned int len4 = len >> 2;   // working-set arrays are 16-byte aligned
        // a small set goes one row per thread so that every warp holds rows
        const bool vec = len4 >= (unsigned int)kPullThreads;
        if (vec) {
            const float4* lo4 = reinterpret_cast<const float4*>(a.w_lo);
#pragma unroll 4
            for (unsigned int i = t; i < len4; i += kPullThreads) {
                const float4 l = lo4[i];
                mx = max(mx, max(max(live_key(l.x), live_key(l.y)), max(live_key(l.z), live_key(l.w))));
            }
            for (unsigned int i = 4 * len4 + t; i < len; i += kPullThreads)
                mx = max(mx, live_key(a.w_lo[i]));
        } else {
            for (unsigned int i = t; i < len; i += kPullThreads) mx = max(mx, live_key(a.w_lo[i]));
        }
        const int busy_warps =
            max(1, min(kPullWarps, (int)((min(len, (unsigned int)kPullThreads) + 31) / 32)));
        // Every warp lists its j2 largest thread maxima (values of distinct
        // rows); the R-th largest of the listed values bounds the R-th largest
        // live lower bound from below.  R = n (over each warp's first j1
        // values; the warps that hold rows list at least n) gives the tight
        // bound; R = kFrontMult n, at most their j2 values each, the wide one.
        // Threads without live rows list zeros (a bound of 0 gathers every row).
        const int j1 = min(32, (n + busy_warps - 1) / busy_warps);
        const int j2 = r.new_front
                           ? max(j1, min(32, ((int)hint * n + busy_warps - 1) / busy_warps))
                           : j1;
        const unsigned int r2 = min(hint * (unsigned int)n, (unsigned int)(busy_warps * j2));
        const unsigned int rm = min(3u * (unsigned int)n, r2);
        for (int it = 0; it < j2; ++it) {
            const uint32_t top = __reduce_max_sync(0xffffffffu, mx);
            const unsigned int holders = __ballot_sync(0xffffffffu, mx == top);
            if (lane == __ffs(holders) - 1) mx = 0;
            if (lane == 0) sh.hist[warp * j2 + it] = top;
        }
        if (t == 0) {
            sh.count = 0;
            sh.cand_n = 0;
            sh.ok = 0;
            sh.warp_tot[0] = 0;   // wide bound
            sh.warp_tot[1] = 0;   // tight bound
            sh.warp_tot[2] = 0;   // middle bound (3 n rows)
        }
        __syncthreads();
        const int nv = kPullWarps * j2;
        for (int e = t; e < nv; e += kPullThreads) {
            const uint32_t v = sh.hist[e];
            unsigned int gt = 0, ge = 0, gt1 = 0, ge1 = 0;
            for (int f = 0; f < nv; ++f) {
                const uint32_t u = sh.hist[f];
                const bool first = (f % j2) < j1;
                gt += u > v;
                ge += u >= v;
                gt1 += first && u > v;
                ge1 += first && u >= v;
            }
            if (gt < r2 && r2 <= ge) sh.warp_tot[0] = v;                       // same value from every writer
            if (gt < rm && rm <= ge) sh.warp_tot[2] = v;
            if ((e % j2) < j1 && gt1 < (unsigned int)n && (unsigned int)n <= ge1) sh.warp_tot[1] = v;
        }
        __syncthreads();
        r.t0 = sh.warp_tot[0];
        r.mult = r.new_front ? hint : 1u;
        t0_mid = sh.warp_tot[2];
        t0_tight = sh.warp_tot[1];
        __syncthreads();   // sh.hist is the gather's buffer
    }
    for (;;) {
        gather_rows(a, sh, r.from_front, len, r.t0);
        r.g = sh.count;
        r.l = sh.cand_n;
        if (r.g <= (unsigned int)kGatherCap && r.l <= (unsigned int)kPullSortCap) break;
        // too many rows reach this bound: gather again at the next tighter one
        // (3 n rows, still a frontier; then n rows, none)
        uint32_t next = 0;
        if (!r.from_front && r.mult > 3u && t0_mid > r.t0) {
            next = t0_mid;
            r.mult = 3u;
        } else if (!r.from_front && r.mult > 1u && t0_tight > r.t0) {
            next = t0_tight;
            r.mult = 1u;
            r.new_front = false;
        } else {
            r.mode = 0;
            return r;
        }
        r.t0 = next;
        __syncthreads();
        if (t == 0) {
            sh.count = 0;
            sh.cand_n = 0;
        }
        __syncthreads();
    }
    // tau: the lower-bound key v with #{> v} < n <= #{>= v} among the l rows
    // with lo >= t0 (the n-th largest is one of them when l >= n).  Counting
    // is quadratic in l; for a long list a bound t_sub <= the n-th largest
    // (the n-th largest of the warps' listed top thread maxima, listed past
    // the keys) leaves only the entries >= t_sub to count.
    uint32_t t_sub = 0;
    const int jn = (n + kPullWarps - 1) / kPullWarps;
    if (r.l > 256 && r.l + (unsigned int)(kPullWarps * jn) <= (unsigned int)kPullSortCap) {
        uint32_t mx = 0;
        for (unsigned int e = t; e < r.l; e += kPullThreads) mx = max(mx, sh.hist[e]);
        uint32_t* listed = sh.hist + r.l;
        for (int it = 0; it < jn; ++it) {
            const uint32_t top = __reduce_max_sync(0xffffffffu, mx);
            const unsigned int holders = __ballot_sync(0xffffffffu, mx == top);
            if (lane == __ffs(holders) - 1) mx = 0;
            if (lane == 0) listed[warp * jn + it] = top;
        }
        if (t == 0) sh.warp_tot[2] = 0;
        __syncthreads();
        const int nv = kPullWarps * jn;
        for (int e = t; e < nv; e += kPullThreads) {
            const uint32_t v = listed[e];
            unsigned int gt = 0, ge = 0;
            for (int f = 0; f < nv; ++f) {
                gt += listed[f] > v;
                ge += listed[f] >= v;
            }
            if (gt < (unsigned int)n && (unsigned int)n <= ge) sh.warp_tot[2] = v;
        }
        __syncthreads();
        t_sub = sh.warp_tot[2];
    }
    for (unsigned int e = t; e < r.l; e += kPullThreads) {
        const uint32_t le = sh.hist[e];
        if (le < t_sub) continue;   // below the n-th largest
        unsigned int gt = 0, ge = 0;
        for (unsigned int f = 0; f < r.l; ++f) {
            const uint32_t lf = sh.hist[f];
            gt += lf > le;
            ge += lf >= le;
        }
        if (gt < (unsigned int)n && (unsigned int)n <= ge) {
            sh.prefix = le;   // every writer writes the same value
            sh.ok = 1;
        }
    }
    __syncthreads();
    if (!sh.ok) {
        r.mode = -1;
        return r;
    }
    const uint32_t tau = (uint32_t)sh.prefix;
    if (t == 0) sh.cand_n = 0;
    __syncthreads();
    // candidates: gathered rows with hi >= tau (no score has been written yet:
    // the cluster's first barrier comes after the selection)
    int32_t* list = reinterpret_cast<int32_t*>(sh.hist);   // the lower bounds are done with
    const uint32_t* gidx = reinterpret_cast<const uint32_t*>(sh.sk);
    for (unsigned int e = t; e < r.g; e += kPullThreads) {
        const uint32_t w = gidx[e];
        if (fkey(a.w_hi[w]) >= tau) {
            const unsigned int pos = atomicAdd(&sh.cand_n, 1u);
            if (pos < (unsigned int)kPullSortCap) list[pos] = (int32_t)w;
        }
    }
    __syncthreads();
    if (sh.cand_n > (unsigned int)kPullSortCap) r.mode = 0;   // (the same in every CTA)
    return r;
}

// Exact scores of the candidates this warp owns (index modulo the cluster's warps).
__device__ inline void cluster_refine(const PullArgs& a, const int32_t* cand, unsigned int c,
                                      unsigned int gwarp, unsigned int cluster_warps) {
    const int lane = threadIdx.x & 31;
    unsigned long long refined = 0, fallbacks = 0;
    for (unsigned int j0 = 0; j0 < c; j0 += 32) {
        const unsigned int j = j0 + lane;
        int32_t w = 0, id = 0;
        float l = 0.0f, h = 0.0f;
        bool own = false;
        if (j < c) {
            w = cand[j];
            if ((unsigned int)w % cluster_warps == gwarp) {
                l = a.w_lo[w];
                h = a.w_hi[w];
                id = a.w_id[w];
                own = l < h;   // lo == hi: already the exact score
            }
        }
        unsigned int mine = __ballot_sync(0xffffffffu, own);
        // start every owned row on its way into L1 (one 128-byte line per lane
        // per step) before scoring the first
        const int lines = (a.m_raw * (int)sizeof(float) + 127) >> 7;
        for (unsigned int pm = mine; pm; pm &= pm - 1) {
            const int32_t idp = __shfl_sync(0xffffffffu, id, __ffs(pm) - 1);
            const char* row = reinterpret_cast<const char*>(a.raw + (int64_t)idp * a.m_raw);
            for (int ln = lane; ln < lines; ln += 32)
                asm volatile("prefetch.global.L1 [%0];" ::"l"(row + (ln << 7)));
        }
        while (mine) {
            const int b = __ffs(mine) - 1;
            mine &= mine - 1;
            const int32_t wb = __shfl_sync(0xffffffffu, w, b);
            const int32_t idb = __shfl_sync(0xffffffffu, id, b);
            const float lb = __shfl_sync(0xffffffffu, l, b);
            const float hb = __shfl_sync(0xffffffffu, h, b);
            bool fb;
            const float s = exact_dot_warp_eft<2>(a.qraw, a.qraw, a.raw + (int64_t)idb * a.m_raw,
                                                  a.m_raw, &fb);
            if (lane == 0) {
                ++refined;
                fallbacks += fb;
                if (!isfinite(s)) set_status(a.status, PVS_ERR_OVERFLOW);
                else if (s < lb || s > hb) set_status(a.status, PVS_ERR_INTERVAL);
                a.w_lo[wb] = s;
                a.w_hi[wb] = s;
                if (a.lo) {
                    a.lo[idb] = s;
                    a.hi[idb] = s;
                }
            }
        }
    }
    if (lane == 0 && refined) {
        atomicAdd(&a.ctr->refined, refined);
        if (fallbacks) atomicAdd(&a.ctr->exact_fallbacks, fallbacks);
    }
}

static __device__ __noinline__ void pull_select_radix(const PullArgs& a, PullShared& sh) {
    pull_select_body(a, sh);
}

template <int kCtas>
__device__ inline void pull_cluster_body(const PullArgs& a, PullShared& sh) {
    const uint32_t rank = cluster_ctarank();
    const FastSelect fs = pull_select_fast(a, sh);
    const int mode = fs.mode;
    // Every CTA has read the working set before any CTA writes a score into
    // it.  In the fast path that ordering is all this barrier carries; after
    // the radix fallback it also publishes CTA 0's list (the outcome is the
    // same in every CTA).
    if (mode == 0) {
        if (rank == 0) pull_select_radix(a, sh);   // list and count in global memory
        cluster_barrier();
    } else {
        cluster_barrier_relaxed();
    }
    const int32_t* cand = mode == 1 ? reinterpret_cast<const int32_t*>(sh.hist) : a.cand;
    const unsigned int c = mode == 1 ? sh.cand_n : (mode == 0 ? a.ctr->cand : 0u);
    cluster_refine(a, cand, c, rank * kPullWarps + (threadIdx.x >> 5), kCtas * kPullWarps);
    cluster_barrier();   // every exact score is visible to CTA 0
    if (rank != 0) return;
    if (mode == -1) {    // fewer than n live rows: the working set was too small
        if (threadIdx.x == 0) {
            set_status(a.status, PVS_ERR_INVALID);
            a.ctr->cand = 0;
        }
        mirror_status(a);
        return;
    }
    if (mode == 1 && threadIdx.x == 0) {
        a.ctr->cand = c;
        a.ctr->cand_total += c;
    }
    // the frontier for the next pulls (every CTA has read the old one by now):
    // a whole-set gather becomes the frontier; a frontier pull uses up n of
    // its rows with lo >= bound (rows only leave that set by being emitted)
    if (threadIdx.x == 0) {   // (without a frontier buffer: any old frontier is void)
        if (mode == 1 && fs.from_front) {
            a.ctr->front_k -= (unsigned int)a.n;
        } else if (mode == 1 && fs.new_front) {
            a.ctr->front_n = fs.g;
            a.ctr->front_bound = fs.t0;
            a.ctr->front_k = fs.l >= (unsigned int)a.n ? fs.l - (unsigned int)a.n : 0u;
        } else {
            a.ctr->front_k = 0;
        }
        // where to start the next whole-set gather: the wide bound again while
        // its gathers fit with room to spare, else the middle one
        if (mode == 1 && !fs.from_front)
            a.ctr->front_hint = (fs.mult == (unsigned int)kFrontMult ||
                                 (fs.mult == 3u && fs.g < (unsigned int)kGatherCap / 4))
                                    ? (unsigned int)kFrontMult : 3u;
    }
    if (mode == 1 && fs.new_front)
        for (unsigned int e = threadIdx.x; e < fs.g; e += kPullThreads)
            a.front[e] = (int32_t)reinterpret_cast<const uint32_t*>(sh.sk)[e];
    __syncthreads();   // sh.sk is the emission's sort buffer
    pull_emit_list(a, sh, cand, c);
    mirror_status(a);
}

__global__ void __cluster_dims__(kPullCluster, 1, 1) __launch_bounds__(kPullThreads, 2)
    pull_cluster_kernel(PullArgs a) {
    __shared__ PullShared sh;
    pull_cluster_body<kPullCluster>(a, sh);
}

// One cluster per cursor.
__global__ void __cluster_dims__(kPullClusterBatch, 1, 1) __launch_bounds__(kPullThreads, 2)
    pull_cluster_batch_kernel(const __grid_constant__ PullArgsPack p) {
    __shared__ PullShared sh;
    pull_cluster_body<kPullClusterBatch>(p.a[blockIdx.x / kPullClusterBatch], sh);
}

cudaError_t launch_pull_cluster(const PullArgs& a, cudaStream_t st) {
    if (a.n <= 0) return cudaSuccess;
    if (a.n > kPullFusedMax) return cudaErrorInvalidValue;
    count_launches(1);
    pull_cluster_kernel<<<kPullCluster, kPullThreads, 0, st>>>(a);
    return cudaGetLastError();
}

constexpr int kCopiesPerLaunch = 64;
struct RankCopyPack {
    RankCopy e[kCopiesPerLaunch];
};

__global__ void copy_ranks_kernel(const __grid_constant__ RankCopyPack p) {
    const RankCopy& e = p.e[blockIdx.x];
    for (int i = threadIdx.x; i < e.count; i += blockDim.x) {
        e.dst_ids[i] = e.src_ids[i];
        e.dst_scores[i] = e.src_scores[i];
    }
}

cudaError_t launch_copy_ranks(const RankCopy* host, int n, cudaStream_t st) {
    for (int first = 0; first < n; first += kCopiesPerLaunch) {
        const int count = n - first < kCopiesPerLaunch ? n - first : kCopiesPerLaunch;
        RankCopyPack p;
        for (int i = 0; i < count; ++i) p.e[i] = host[first + i];
        count_launches(1);
        copy_ranks_kernel<<<count, 128, 0, st>>>(p);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// Packs of up to kPullPack cursors' arguments (the last one partial).
static std::vector<PullArgsPack> pull_packs(const PullArgs* host, int n) {
    std::vector<PullArgsPack> packs((size_t)((n + kPullPack - 1) / kPullPack));
    for (int i = 0; i < n; ++i) packs[(size_t)(i / kPullPack)].a[i % kPullPack] = host[i];
    return packs;
}
static int pack_count(int n, size_t k) {
    const int rest = n - (int)k * kPullPack;
    return rest < kPullPack ? rest : kPullPack;
}

cudaError_t launch_pull_cluster_batch(const PullArgs* host_args, int ncursors, cudaStream_t st) {
    if (ncursors <= 0) return cudaSuccess;
    const std::vector<PullArgsPack> packs = pull_packs(host_args, ncursors);
    for (size_t k = 0; k < packs.size(); ++k) {
        count_launches(1);
        pull_cluster_batch_kernel<<<pack_count(ncursors, k) * kPullClusterBatch, kPullThreads, 0,
                                    st>>>(packs[k]);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
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

// ---- batched open: per-query thresholds and ordered working sets --------------

struct RowKeys {   // live lower bounds of one query's dump row
    const float* lo;
    __device__ bool valid(unsigned int i) const { return lo[i] != -INFINITY; }
    __device__ uint32_t key(unsigned int i) const { return fkey(lo[i]); }
};

// One CTA per query: tau[q] = k-th largest live lower bound among the sampled
// rows (dump row q), or -inf if fewer than k are live.
//   1. every thread takes the maximum key of its share of the row (float4
//      loads, several in flight); the k-th largest of these maxima, t0, is a
//      lower bound of the answer: k threads each hold a value >= t0;
//   2. the values >= t0 (usually a few times k) are gathered into shared
//      memory and sorted; the k-th of them is the answer.
// When k exceeds the thread count, fewer than k threads saw a live value, or
// more than kPullSortCap values reach t0, a three-pass radix select decides.
__device__ inline void tau_radix(PullShared& sh, const RowKeys& src, unsigned int nsample,
                                 unsigned int k, float* out) {
    const int t = threadIdx.x;
    if (t == 0) {
        sh.prefix = 0;
        sh.k = k;
    }
    __syncthreads();
    const int shifts32[3] = {21, 10, 0}, bits32[3] = {11, 11, 10};
    for (int p = 0; p < 3; ++p) {
        block_histogram<uint32_t>(sh, nsample, shifts32[p], bits32[p], (uint32_t)sh.prefix, src);
        if (t == 0) sh.ok = 0;
        __syncthreads();
        block_pick_digit(sh, shifts32[p]);
        if (!sh.ok) {
            if (t == 0) *out = -INFINITY;
            return;
        }
    }
    if (t == 0) *out = fkey_inv((uint32_t)sh.prefix);
}

__global__ void __launch_bounds__(kPullThreads, 2) batch_tau_kernel(const float* dump_lo,
                                                                    int64_t ld,
                                                                    unsigned int nsample,
                                                                    unsigned int k, float* tau) {
    __shared__ PullShared sh;
    const int q = blockIdx.x, t = threadIdx.x;
    const float* row = dump_lo + (int64_t)q * ld;
    const RowKeys src{row};
    if (k == 0 || k > (unsigned int)kPullThreads) {
        tau_radix(sh, src, nsample, k, &tau[q]);
        return;
    }
    // 1. per-thread maxima (key 0: no live value; every live key is larger)
    const unsigned int n4 = nsample >> 2;
    const float4* row4 = reinterpret_cast<const float4*>(row);
    auto live_key = [](float v) -> uint32_t { return v == -INFINITY ? 0u : fkey(v); };
    uint32_t mx = 0;
#pragma unroll 4
    for (unsigned int i = t; i < n4; i += kPullThreads) {
        const float4 v = __ldg(row4 + i);
        mx = max(mx, max(max(live_key(v.x), live_key(v.y)), max(live_key(v.z), live_key(v.w))));
    }
    for (unsigned int i = 4 * n4 + t; i < nsample; i += kPullThreads) mx = max(mx, live_key(row[i]));
    sh.sk[t] = ((unsigned long long)mx << 32) | (unsigned int)t;
    __syncthreads();
    bitonic_desc_smem(sh.sk, kPullThreads);
    const uint32_t t0 = (uint32_t)(sh.sk[k - 1] >> 32);
    __syncthreads();
    if (t0 == 0) {   // fewer than k threads saw a live value
        tau_radix(sh, src, nsample, k, &tau[q]);
        return;
    }
    // 2. gather the values >= t0
    if (t == 0) sh.count = 0;
    __syncthreads();
    auto take = [&](float v) {
        const uint32_t key = live_key(v);
        if (key >= t0) {
            const unsigned int pos = atomicAdd(&sh.count, 1u);
            if (pos < (unsigned int)kPullSortCap) sh.sk[pos] = (unsigned long long)key << 32;
        }
    };
#pragma unroll 4
    for (unsigned int i = t; i < n4; i += kPullThreads) {
        const float4 v = __ldg(row4 + i);
        take(v.x), take(v.y), take(v.z), take(v.w);
    }
    for (unsigned int i = 4 * n4 + t; i < nsample; i += kPullThreads) take(row[i]);
    __syncthreads();
    const unsigned int cnt = sh.count;
    if (cnt > (unsigned int)kPullSortCap) {
        __syncthreads();
        tau_radix(sh, src, nsample, k, &tau[q]);
        return;
    }
    int pow2 = 1;
    while (pow2 < (int)cnt) pow2 <<= 1;
    for (int i = (int)cnt + t; i < pow2; i += kPullThreads) sh.sk[i] = 0ull;
    __syncthreads();
    bitonic_desc_smem(sh.sk, pow2);
    if (t == 0) tau[q] = fkey_inv((uint32_t)(sh.sk[k - 1] >> 32));
}

cudaError_t launch_batch_tau(const float* dump_lo, int64_t ld, unsigned int nsample, int nq,
                             unsigned int k, float* tau, cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    count_launches(1);
    batch_tau_kernel<<<nq, kPullThreads, 0, st>>>(dump_lo, ld, nsample, k, tau);
    return cudaGetLastError();
}

// One CTA per query: the unordered working set written by the filter pass
// (ids, bounds at [q * cap, ...)) is sorted by id into the cursor's own
// arrays, so that working-set index order is id order.
__global__ void __launch_bounds__(kPullThreads) ws_sort_kernel(const int32_t* w_id_b,
                                                               const float* w_lo_b,
                                                               const float* w_hi_b, int cap,
                                                               const unsigned int* w_len_b,
                                                               const WsDst* dst) {
    extern __shared__ unsigned long long keys[];
    const int q = blockIdx.x, t = threadIdx.x;
    const unsigned int len = w_len_b[q];
    const WsDst d = dst[q];
    if (len > (unsigned int)cap) {          // overflow: the cursor rescans instead
        if (t == 0) *d.w_len = 0;
        return;
    }
    int pow2 = 1;
    while (pow2 < (int)len) pow2 <<= 1;
    const int64_t base = (int64_t)q * cap;
    for (int i = t; i < pow2; i += kPullThreads)
        keys[i] = i < (int)len ? ((unsigned long long)(0xffffffffu - (uint32_t)w_id_b[base + i]) << 32) |
                                     (unsigned int)i
                               : 0ull;
    __syncthreads();
    bitonic_desc_smem(keys, pow2);
    for (int r = t; r < (int)len; r += kPullThreads) {
        const unsigned int pos = (unsigned int)(keys[r] & 0xffffffffull);
        d.w_id[r] = w_id_b[base + pos];
        d.w_lo[r] = w_lo_b[base + pos];
        d.w_hi[r] = w_hi_b[base + pos];
    }
    if (t == 0) *d.w_len = len;
}

cudaError_t launch_ws_sort(const int32_t* w_id_b, const float* w_lo_b, const float* w_hi_b,
                           int cap, const unsigned int* w_len_b, const WsDst* dst, int nq,
                           cudaStream_t st) {
    if (nq <= 0) return cudaSuccess;
    if (cap > kWsSortMax) return cudaErrorInvalidValue;
    int pow2 = 1;
    while (pow2 < cap) pow2 <<= 1;
    const size_t smem = (size_t)pow2 * sizeof(unsigned long long);
    cudaError_t e = raise_smem_limit((const void*)ws_sort_kernel, smem);
    if (e != cudaSuccess) return e;
    count_launches(1);
    ws_sort_kernel<<<nq, kPullThreads, smem, st>>>(w_id_b, w_lo_b, w_hi_b, cap, w_len_b, dst);
    return cudaGetLastError();
}

// Selection for every pack, then refinement for every pack, then emission.
cudaError_t launch_pull_batch(const PullArgs* host_args, int ncursors, int refine_blocks_per_cursor,
                              int m_raw, cudaStream_t st) {
    if (ncursors <= 0) return cudaSuccess;
    const std::vector<PullArgsPack> packs = pull_packs(host_args, ncursors);
    for (size_t k = 0; k < packs.size(); ++k) {
        count_launches(1);
        pull_select_batch_kernel<<<pack_count(ncursors, k), kPullThreads, 0, st>>>(packs[k]);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    for (size_t k = 0; k < packs.size(); ++k) {
        cudaError_t e = launch_refine_batch(packs[k], pack_count(ncursors, k),
                                            refine_blocks_per_cursor, m_raw, st);
        if (e != cudaSuccess) return e;
    }
    for (size_t k = 0; k < packs.size(); ++k) {
        count_launches(1);
        pull_emit_batch_kernel<<<pack_count(ncursors, k), kPullThreads, 0, st>>>(packs[k]);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace pvs
