// EAHR host driver (arXiv 2608.07152, Sec. 2.1 and 2.2): ordered Top-K of
// complete-list weighted RRF, read adaptively from two resumable exact
// ranked lists.
//
// Bounds (Sec. 2.2), all exact rationals:
//   u_i = g_i(d_i + 1) for an Open list, 0 for an Exhausted one;
//   L(x) = sum of the contributions already read; U(x) = L(x) + u_i for every
//   Open list i that has not returned x; B = u_0 + u_1.
// Certification: x+ = argmax over R = O \ A of (L, -id) is appended when its
// (L, id) beats (U(y), y) for every other y in R and L(x+) > B.
//
// With two lists every bound is a sum of at most two contributions
// a / (b r + c) with denominators below 2^32, so numerators stay below 2^49,
// denominators below 2^64, and comparisons are exact in 128-bit integers.
//
// Incremental structures: items read from both lists (their F is final)
// are kept best-first by (F desc, id asc), but only the K + 2 best of them:
// certification looks at the best two, and items leave this group only from
// the top, at most K times, so nothing further down can ever be looked at.
// Items read from one list only are ordered by their rank in that list
// (their L and U are monotone in it), so the best and second-best of each
// group are found without scanning O.
//
// Per-request state indexed by id (two rank arrays and a flag array over the
// id space: 80 MB at 8.8M ids) comes from a pool and goes back cleared: a
// request clears only the entries it wrote, so its cost follows its depth,
// not the id space (fresh zero pages cost a page fault per touched page).
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <limits>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include "../../include/merge.h"
#include "../../include/pbm.h"
#include "../../include/pvs.h"
#include "runtime.h"

// facts about merge cursors (merge.cu) and PBM cursors (pbm_capi.cu)
namespace pvs {
int64_t merge_id_space(const pvs_merge* m);
int64_t merge_length(const pvs_merge* m);
bool merge_fresh(const pvs_merge* m);
const SnapData* pbm_cursor_snapshot(const pbm_cursor* c);
}  // namespace pvs

namespace {

typedef unsigned __int128 u128;

struct Frac {
    uint64_t num = 0, den = 1;
};

inline int cmp(const Frac& a, const Frac& b) {
    const u128 l = (u128)a.num * b.den, r = (u128)b.num * a.den;
    return l < r ? -1 : (l > r ? 1 : 0);
}

inline Frac add(const Frac& a, const Frac& b) {
    if (a.num == 0) return b;
    if (b.num == 0) return a;
    Frac s;
    s.num = a.num * b.den + b.num * a.den;
    s.den = a.den * b.den;
    return s;
}

inline int bitlen(u128 x) {
    int n = 0;
    while (x) {
        ++n;
        x >>= 1;
    }
    return n;
}

// Correctly rounded (nearest, ties to even) binary64 value of num / den.
double frac_to_double(const Frac& f) {
    if (f.num == 0) return 0.0;
    const int s = 55 + bitlen(f.den) - bitlen(f.num);
    const u128 n = (u128)f.num << s;
    u128 q = n / f.den;
    const bool rem = (n % f.den) != 0;
    const int drop = bitlen(q) - 53;               // 2 or 3
    const u128 mask = ((u128)1 << drop) - 1;
    const u128 low = q & mask, half = (u128)1 << (drop - 1);
    u128 mant = q >> drop;
    if (low > half || (low == half && (rem || (mant & 1)))) ++mant;
    return std::ldexp((double)(uint64_t)mant, drop - s);
}

// g(r) = a / (b r + c)
struct Contrib {
    uint64_t a = 0, b = 1, c = 0;
    Frac at(int64_t r) const {
        Frac f;
        if (a == 0) return f;
        f.num = a;
        f.den = b * (uint64_t)r + c;
        return f;
    }
    // the same in binary64 (relative error within 2^-52)
    double at_d(int64_t r) const {
        return a == 0 ? 0.0 : (double)a / (double)(b * (uint64_t)r + c);
    }
};

struct Node {
    Frac F;
    int32_t id;
};
struct NodeCmp {
    bool operator()(const Node& x, const Node& y) const {
        const int c = cmp(x.F, y.F);
        if (c != 0) return c > 0;     // larger F first
        return x.id < y.id;           // then smaller id
    }
};

// The best `cap` items read from both lists, best first.
struct TopBoth {
    std::vector<Node> v;
    size_t cap = 2;
    bool empty() const { return v.empty(); }
    void insert(const Node& n) {
        if (v.size() == cap && !NodeCmp()(n, v.back())) return;   // not above the worst kept
        v.insert(std::upper_bound(v.begin(), v.end(), n, NodeCmp()), n);
        if (v.size() > cap) v.pop_back();
    }
    void pop_front() { v.erase(v.begin()); }
};

// The best `cap` nodes of a stream, whatever the order of arrival:
// candidates gather in a buffer that is cut back to the best `cap` whenever
// it fills; once `cap` are kept, anything not above the worst kept is
// dropped at once.
struct TopStream {
    static constexpr size_t kCut = 4096;
    size_t cap = 2;
    std::vector<Node> buf;
    bool full = false;
    Node worst;
    void push(const Node& n) {
        if (full && !NodeCmp()(n, worst)) return;
        buf.push_back(n);
        if (buf.size() >= kCut) cut();
    }
    void cut() {
        if (buf.size() > cap) {
            std::nth_element(buf.begin(), buf.begin() + (std::ptrdiff_t)(cap - 1), buf.end(),
                             NodeCmp());
            buf.resize(cap);
        }
        if (buf.size() == cap) {
            full = true;
            worst = *std::max_element(buf.begin(), buf.end(), NodeCmp());
        }
    }
};

// (a, x) beats (b, y): a > b, or a == b and x has the smaller id.
inline bool beats(const Frac& a, int32_t x, const Frac& b, int32_t y) {
    const int c = cmp(a, b);
    return c > 0 || (c == 0 && x < y);
}

// Zeroed id-indexed arrays, kept for reuse (at most kPoolMax of them and
// kPoolBytes in all; larger or surplus ones are freed).  The two lists'
// ranks of one id sit side by side (one cache line serves both lookups), and
// the certified-set flags are a bitset (1.1 MB at 8.8M ids, cache-resident).
// The two lists' read ids are stored here too (a valid list repeats no id,
// so cap entries hold it); their contents are always ids below cap.
struct Workspace {
    int32_t* ranks = nullptr;    // [cap][2]
    uint64_t* bits = nullptr;    // [(cap + 63) / 64]
    int32_t* read[2] = {nullptr, nullptr};   // [cap] each
    int64_t cap = 0;
    size_t bytes() const {
        return (size_t)cap * 4 * sizeof(int32_t) + (size_t)(cap + 63) / 8;
    }
    void release() {
        std::free(ranks);
        std::free(bits);
        std::free(read[0]);
        std::free(read[1]);
        ranks = nullptr;
        bits = nullptr;
        read[0] = read[1] = nullptr;
        cap = 0;
    }
};

// The ids read from one list, in rank order, in workspace storage.
struct IdList {
    int32_t* p = nullptr;
    size_t n = 0, cap = 0;
    size_t size() const { return n; }
    int32_t operator[](size_t i) const { return p[i]; }
    const int32_t* begin() const { return p; }
    const int32_t* end() const { return p + n; }
};

// memset of a large array over up to kMaxThreads threads (what a thread
// that cannot start would have cleared is cleared here).
void zero_parallel(void* dst, size_t bytes);

constexpr size_t kPoolMax = 16;
constexpr int64_t kParallelMin = int64_t(1) << 17;   // ranks per pull worth threads
constexpr unsigned kMaxThreads = 8;
constexpr int64_t kAheadMin = int64_t(1) << 17;   // dense pulls worth a helper thread
constexpr size_t kPoolBytes = size_t(1) << 30;

std::mutex g_pool_mutex;
std::vector<Workspace> g_pool;
size_t g_pool_bytes = 0;

// A zeroed workspace of at least `ids` entries: the smallest pooled one that
// fits, else a new one.
bool acquire(int64_t ids, Workspace* out) {
    {
        std::lock_guard<std::mutex> lock(g_pool_mutex);
        size_t best = g_pool.size();
        for (size_t k = 0; k < g_pool.size(); ++k)
            if (g_pool[k].cap >= ids && (best == g_pool.size() || g_pool[k].cap < g_pool[best].cap))
                best = k;
        if (best < g_pool.size()) {
            *out = g_pool[best];
            g_pool_bytes -= out->bytes();
            g_pool.erase(g_pool.begin() + (std::ptrdiff_t)best);
            return true;
        }
    }
    Workspace w;
    w.cap = ids;
    w.ranks = static_cast<int32_t*>(std::calloc((size_t)ids * 2, sizeof(int32_t)));
    w.bits = static_cast<uint64_t*>(std::calloc((size_t)(ids + 63) / 64, sizeof(uint64_t)));
    w.read[0] = static_cast<int32_t*>(std::calloc((size_t)ids, sizeof(int32_t)));
    w.read[1] = static_cast<int32_t*>(std::calloc((size_t)ids, sizeof(int32_t)));
    if (!w.ranks || !w.bits || !w.read[0] || !w.read[1]) {
        w.release();
        return false;
    }
    *out = w;
    return true;
}

// Return a workspace whose arrays are all zero again.
void give_back(Workspace w) {
    std::lock_guard<std::mutex> lock(g_pool_mutex);
    if (g_pool.size() < kPoolMax && g_pool_bytes + w.bytes() <= kPoolBytes) {
        g_pool_bytes += w.bytes();
        g_pool.push_back(w);
        return;
    }
    w.release();
}

void zero_parallel(void* dst, size_t bytes) {
    const unsigned T = std::min<unsigned>(kMaxThreads, std::thread::hardware_concurrency());
    if (bytes < (size_t(16) << 20) || T < 2) {
        std::memset(dst, 0, bytes);
        return;
    }
    uint8_t* b = static_cast<uint8_t*>(dst);
    auto part = [&](unsigned t) {
        const size_t lo = bytes * t / T, hi = bytes * (t + 1) / T;
        std::memset(b + lo, 0, hi - lo);
    };
    std::vector<std::thread> th;
    unsigned started = 1;
    try {
        th.reserve(T - 1);
        for (; started < T; ++started) th.emplace_back(part, started);
    } catch (...) {
    }
    part(0);
    for (unsigned t = started; t < T; ++t) part(t);
    for (auto& x : th) x.join();
}

// Smallest (at most 0) and largest (at least -1) id of a host list, long
// lists over up to kMaxThreads threads.
void id_range(const int64_t* l, int64_t len, int64_t* lo_out, int64_t* hi_out) {
    const unsigned T = len >= (int64_t(1) << 20)
                           ? std::min<unsigned>(kMaxThreads, std::thread::hardware_concurrency())
                           : 1u;
    std::vector<int64_t> lo((size_t)std::max(T, 1u), 0), hi((size_t)std::max(T, 1u), -1);
    auto part = [&](unsigned t) {
        const int64_t a = len * (int64_t)t / (int64_t)T, b = len * (int64_t)(t + 1) / (int64_t)T;
        int64_t x = 0, y = -1;
        for (int64_t k = a; k < b; ++k) {
            x = std::min(x, l[k]);
            y = std::max(y, l[k]);
        }
        lo[t] = x;
        hi[t] = y;
    };
    std::vector<std::thread> th;
    unsigned started = 1;
    if (T > 1) {
        try {
            th.reserve(T - 1);
            for (; started < T; ++started) th.emplace_back(part, started);
        } catch (...) {
        }
    }
    if (T >= 1) part(0);
    for (unsigned t = started; t < T; ++t) part(t);
    for (auto& x : th) x.join();
    *lo_out = *std::min_element(lo.begin(), lo.end());
    *hi_out = *std::max_element(hi.begin(), hi.end());
}

struct Source {
    // dense cursor, sparse PBM cursor, merge cursor or host list
    pvs_cursor* cursor = nullptr;
    pbm_cursor* sparse = nullptr;
    pvs_merge* merge = nullptr;
    const int64_t* list = nullptr;
    int64_t length = 0;
};

class Driver {
  public:
    Contrib g[2];
    Source src[2];
    bool active[2] = {true, true};   // positive weight
    int64_t depth[2] = {0, 0};
    bool exhausted[2] = {false, false};
    int32_t pulls[2] = {0, 0};
    int32_t checks = 0;
    IdList prefix[2];
    int32_t* ranks = nullptr;    // ranks[2 x + i]: rank of id x in list i (0: unread)
    uint64_t* bits = nullptr;    // bit x: x is certified (in A)
    int64_t id_space = 0;
    TopBoth both;
    size_t ptr[2] = {0, 0};
    int64_t both_read = 0;   // items read from both lists
    std::vector<int32_t> A;
    int K = 0;
    std::vector<int64_t> buf_ids;
    std::vector<float> buf_scores;
    const pvs::SnapData* snap = nullptr;

    Workspace ws;

    // A dense pull running on a helper thread while this one records the
    // other list and certifies (long pulls of a dense cursor only).  The
    // cursor is touched by that thread alone until it is joined; its ranks
    // stay in the cursor's pinned buffers until they are recorded.
    std::thread ahead;
    bool ahead_live = false;
    pvs_status ahead_status = PVS_OK;
    const int64_t* ahead_ids = nullptr;
    const float* ahead_scores = nullptr;
    int32_t ahead_got = 0;

    void start_ahead(int64_t n) {
        if (ahead_live || !src[0].cursor || !active[0] || exhausted[0]) return;
        n = std::min<int64_t>(n, std::numeric_limits<int32_t>::max());
        try {
            ahead = std::thread([this, n] {
                ahead_status = pvs::next_pinned(src[0].cursor, (int32_t)n, &ahead_ids,
                                                &ahead_scores, &ahead_got);
            });
            ahead_live = true;
        } catch (...) {   // no thread: the pull runs when it is needed
        }
    }
    void join_ahead() {
        if (ahead_live) ahead.join();
        ahead_live = false;
    }

    // The host sparse list scattered on the device by a helper thread while
    // the dense list is read (EAHR_POLICY_ADAPTIVE's finishes use it).
    std::thread stage;
    bool stage_live = false;
    pvs_status stage_status = PVS_OK;
    pvs::StagedList* staged = nullptr;

    // (a PBM source: its complete ranking, computed on the device)
    void start_stage() {
        if (stage_live || !src[0].cursor) return;
        const bool host_list = src[1].list && src[1].length > 0;
        if (!host_list && !src[1].sparse) return;
        try {
            stage = std::thread([this, host_list] {
                stage_status =
                    host_list ? pvs::stage_sparse_list(src[0].cursor, src[1].list, src[1].length,
                                                       &staged)
                              : pvs::pbm_stage_ranks(src[1].sparse, src[0].cursor->index, &staged);
            });
            stage_live = true;
        } catch (...) {   // no thread: a host list is copied by the finish itself
        }
    }
    void join_stage() {
        if (stage_live) stage.join();
        stage_live = false;
    }
    // The check of a staged host list, queued once the dense list's first
    // pull (and its interval pass) is done, so that it does not run beside
    // the pass.
    void check_stage() {
        join_stage();
        if (stage_status == PVS_OK && staged && !staged->checked)
            stage_status = pvs::check_staged_list(staged);
    }
    // The staged list once it is queued and checked (null when staging failed).
    const pvs::StagedList* staged_list() {
        check_stage();
        return stage_status == PVS_OK ? staged : nullptr;
    }

    int32_t rank(int i, int32_t x) const { return ranks[2 * (size_t)x + (size_t)i]; }
    bool inA(int32_t x) const { return (bits[(uint32_t)x >> 6] >> (x & 63)) & 1u; }

    // Every entry written is an id of prefix[i] (ranks) or of A (bits):
    // clear those, or whole arrays when that is cheaper, and pool them.
    ~Driver() {
        join_ahead();
        join_stage();
        pvs::free_staged_list(staged);
        if (!ws.ranks) return;
        if ((int64_t)(prefix[0].size() + prefix[1].size()) > ws.cap / 8) {
            zero_parallel(ranks, (size_t)ws.cap * 2 * sizeof(int32_t));
        } else {
            for (int i = 0; i < 2; ++i)
                for (int32_t x : prefix[i]) ranks[2 * (size_t)x + (size_t)i] = 0;
        }
        for (int32_t x : A) bits[(uint32_t)x >> 6] = 0;
        give_back(ws);
    }

    bool init(int64_t ids) {
        id_space = std::max<int64_t>(ids, 1);
        if (!acquire(id_space, &ws)) return false;
        ranks = ws.ranks;
        bits = ws.bits;
        for (int i = 0; i < 2; ++i) {
            prefix[i].p = ws.read[i];
            prefix[i].n = 0;
            prefix[i].cap = (size_t)ws.cap;
        }
        return true;
    }

    Frac u(int i) const {
        if (!active[i] || exhausted[i]) return Frac{};
        return g[i].at(depth[i] + 1);
    }

    Frac L(int32_t x) const {
        Frac f;
        const int32_t r0 = rank(0, x), r1 = rank(1, x);
        if (active[0] && r0) f = add(f, g[0].at(r0));
        if (active[1] && r1) f = add(f, g[1].at(r1));
        return f;
    }

    // L and U in binary64, within 2^-50 of the exact values (relative)
    double L_d(int32_t x) const {
        double f = 0.0;
        const int32_t r0 = rank(0, x), r1 = rank(1, x);
        if (active[0] && r0) f += g[0].at_d(r0);
        if (active[1] && r1) f += g[1].at_d(r1);
        return f;
    }
    double U_d(int32_t x) const {
        double f = L_d(x);
        for (int i = 0; i < 2; ++i)
            if (active[i] && !exhausted[i] && !rank(i, x)) f += u_d(i);
        return f;
    }
    double u_d(int i) const {
        if (!active[i] || exhausted[i]) return 0.0;
        return g[i].at_d(depth[i] + 1);
    }

    Frac U(int32_t x) const {
        Frac f = L(x);
        for (int i = 0; i < 2; ++i)
            if (active[i] && !exhausted[i] && !rank(i, x)) f = add(f, u(i));
        return f;
    }

    // Record ranks depth+1 .. depth+n of list i.  Ids from host lists are
    // checked as they are read: inside the id space, visible in the
    // snapshot (when there is one) and not repeated within the list.
    bool record(int i, const int64_t* ids, int64_t n) {
        if (n >= kParallelMin) {
            const int T = (int)std::min<unsigned>(kMaxThreads, std::thread::hardware_concurrency());
            if (T > 1) return record_parallel(i, ids, n, T);
        }
        const int j = 1 - i;
        const bool check = src[i].cursor == nullptr && src[i].sparse == nullptr &&
                           src[i].merge == nullptr;
        // ids arrive in rank order, scattered over the id space: fetch the
        // rank pair of the id kAhead positions on while this one is handled
        constexpr int64_t kAhead = 16;
        if (prefix[i].n + (size_t)n > prefix[i].cap) return false;   // an id repeats
        for (int64_t t = 0; t < n; ++t) {
            if (t + kAhead < n) {
                const int64_t y = ids[t + kAhead];
                if (y >= 0 && y < id_space) __builtin_prefetch(ranks + 2 * y, 1, 0);
            }
            const int64_t x64 = ids[t];
            if (check) {
                if (x64 < 0 || x64 >= id_space) return false;
                if (snap && !snap->is_visible(x64)) return false;
                if (rank(i, (int32_t)x64)) return false;
            }
            const int32_t x = (int32_t)x64;
            prefix[i].p[prefix[i].n++] = x;
            ranks[2 * (size_t)x + (size_t)i] = (int32_t)(depth[i] + t + 1);
            if (rank(j, x)) {
                ++both_read;
                if (!inA(x)) both.insert(Node{L(x), x});
            }
        }
        depth[i] += n;
        return true;
    }

    // record() over T threads, for long pulls: each thread takes a
    // contiguous part and, in one pass, writes the ranks (and the read ids)
    // and collects its part's best items read from both lists.  Which items
    // enter `both`, the K + 2 best, does not depend on the order of inserts.
    // A cursor's ids never repeat; a host list's are checked as they are
    // written: the rank slot is exchanged, and a slot that already held a
    // rank (from an earlier pull, or from another part of this one) means a
    // repeated id.  L of a doubly-read item comes from the rank just written
    // and the other list's rank (that list is not written here), so no slot
    // of list i is read while other parts may write it.
    bool record_parallel(int i, const int64_t* ids, int64_t n, int T) {
        const int j = 1 - i;
        const bool check = src[i].cursor == nullptr && src[i].sparse == nullptr &&
                           src[i].merge == nullptr;
        IdList& pre = prefix[i];
        const size_t base = pre.n;
        if (base + (size_t)n > pre.cap) return false;   // an id repeats
        // counted before the parts run: cleanup then covers whatever a part
        // wrote before it stopped (stale entries are ids below cap)
        pre.n = base + (size_t)n;
        const int64_t d0 = depth[i];
        std::vector<uint8_t> bad((size_t)T, 0);
        std::vector<std::vector<Node>> tops((size_t)T);
        std::vector<int64_t> doubly((size_t)T, 0);
        auto part = [&](int t) {
            const int64_t lo = n * t / T, hi = n * (t + 1) / T;
            // thread-local until the end: neighbouring threads' counters and
            // vectors would share cache lines
            TopStream top;
            top.cap = both.cap;
            top.buf.reserve(TopStream::kCut);
            int64_t count = 0;
            for (int64_t k = lo; k < hi; ++k) {
                if (k + 16 < hi) {
                    const int64_t y = ids[k + 16];
                    if (y >= 0 && y < id_space) __builtin_prefetch(ranks + 2 * y, 1, 0);
                }
                const int64_t x64 = ids[k];
                const int32_t r = (int32_t)(d0 + k + 1);
                if (check) {
                    if (x64 < 0 || x64 >= id_space || (snap && !snap->is_visible(x64))) {
                        bad[(size_t)t] = 1;
                        break;
                    }
                    pre.p[base + (size_t)k] = (int32_t)x64;   // recorded before the write
                    if (__atomic_exchange_n(ranks + 2 * x64 + i, r, __ATOMIC_RELAXED) != 0) {
                        bad[(size_t)t] = 1;
                        break;
                    }
                } else {
                    ranks[2 * (size_t)x64 + (size_t)i] = r;
                    pre.p[base + (size_t)k] = (int32_t)x64;
                }
                const int32_t x = (int32_t)x64;
                const int32_t rj = rank(j, x);
                if (rj) {
                    ++count;
                    if (!inA(x)) {
                        Frac f;
                        if (active[i]) f = add(f, g[i].at(r));
                        if (active[j]) f = add(f, g[j].at(rj));
                        top.push(Node{f, x});
                    }
                }
            }
            top.cut();
            doubly[(size_t)t] = count;
            tops[(size_t)t] = std::move(top.buf);
        };
        // parts whose thread could not be started run here, after part 0
        std::vector<std::thread> th;
        int started = 1;
        try {
            th.reserve((size_t)T - 1);
            for (; started < T; ++started) th.emplace_back(part, started);
        } catch (...) {
        }
        part(0);
        for (int t = started; t < T; ++t) part(t);
        for (auto& x : th) x.join();
        for (uint8_t b : bad)
            if (b) return false;
        for (const std::vector<Node>& top : tops)
            for (const Node& nd : top) both.insert(nd);
        for (int64_t c : doubly) both_read += c;
        depth[i] += n;
        return true;
    }

    // First item of list i, at or after position `from` of its prefix, that
    // is read from list i only and not fixed; -1 if none.
    int32_t only_from(int i, size_t from, int32_t skip) const {
        if (single(i) == 0) return -1;
        const int j = 1 - i;
        const IdList& pre = prefix[i];
        for (size_t p = from; p < pre.size(); ++p) {
            if (p + 16 < pre.size()) __builtin_prefetch(ranks + 2 * (size_t)pre[p + 16], 0, 0);
            const int32_t x = pre[p];
            if (inA(x) || x == skip) continue;
            if (active[j] && rank(j, x)) continue;
            return x;
        }
        return -1;
    }

    void advance_ptr(int i) {
        if (single(i) == 0) {   // every item of list i was read from both lists
            ptr[i] = prefix[i].size();
            return;
        }
        const int j = 1 - i;
        const IdList& pre = prefix[i];
        while (ptr[i] < pre.size()) {
            if (ptr[i] + 16 < pre.size())
                __builtin_prefetch(ranks + 2 * (size_t)pre[ptr[i] + 16], 0, 0);
            const int32_t x = pre[ptr[i]];
            if (inA(x) || (active[j] && rank(j, x))) {
                ++ptr[i];
                continue;
            }
            break;
        }
    }

    // Items read from list i only (certified or not).
    int64_t single(int i) const { return depth[i] - both_read; }

    // Sec. 2.2 certification; returns true when the result is complete.
    bool certify() {
        ++checks;
        const Frac B = add(u(0), u(1));
        while ((int)A.size() < K) {
            advance_ptr(0);
            advance_ptr(1);
            // candidates for x+
            int32_t cand[3] = {-1, -1, -1};
            if (!both.empty()) cand[0] = both.v[0].id;
            if (active[0]) cand[1] = only_from(0, ptr[0], -1);
            if (active[1]) cand[2] = only_from(1, ptr[1], -1);
            int32_t xp = -1;
            Frac Lx;
            for (int t = 0; t < 3; ++t) {
                if (cand[t] < 0) continue;
                const Frac l = L(cand[t]);
                if (xp < 0 || beats(l, cand[t], Lx, xp)) {
                    xp = cand[t];
                    Lx = l;
                }
            }
            if (xp < 0) return B.num == 0;   // R empty
            // strongest other item by (U, id)
            int32_t others[3] = {-1, -1, -1};
            if (!both.empty()) {
                size_t k = both.v[0].id == xp ? 1 : 0;
                if (k < both.v.size()) others[0] = both.v[k].id;
            }
            if (active[0]) others[1] = only_from(0, ptr[0], xp);
            if (active[1]) others[2] = only_from(1, ptr[1], xp);
            bool ok = cmp(Lx, B) > 0;
            for (int t = 0; t < 3 && ok; ++t)
                if (others[t] >= 0) ok = beats(Lx, xp, U(others[t]), others[t]);
            if (!ok) {
                // complete when nothing left can have a positive score
                if (B.num != 0) return false;
                return Lx.num == 0;
            }
            A.push_back(xp);
            bits[(uint32_t)xp >> 6] |= 1ull << (xp & 63);
            // read from both lists: then it was the best of that group
            if (active[0] && active[1] && rank(0, xp) && rank(1, xp)) both.pop_front();
        }
        return true;
    }

    // Pull up to n ranks from list i.  A producer's list length is only an
    // upper bound until it reports Exhausted (a sparse support U_s is known
    // only then); from then on it is the depth read.
    pvs_status pull(int i, int64_t n) {
        if (exhausted[i] || !active[i]) return PVS_OK;
        pulls[i]++;
        if (n > (int64_t)std::numeric_limits<int32_t>::max()) n = std::numeric_limits<int32_t>::max();
        if (src[i].cursor) {   // read where the pull left them (pinned), without a copy
            const int64_t* ids = nullptr;
            const float* scores = nullptr;
            int32_t got = 0;
            pvs_status s;
            if (ahead_live) {   // the pull started earlier: its ranks are the next ones
                join_ahead();
                s = ahead_status;
                ids = ahead_ids;
                scores = ahead_scores;
                got = ahead_got;
            } else {
                s = pvs::next_pinned(src[i].cursor, (int32_t)n, &ids, &scores, &got);
            }
            if (s < 0) return s;
            if (!record(i, ids, got)) return PVS_ERR_INVALID;
            if (s == PVS_EXHAUSTED) exhausted[i] = true;
        } else if (src[i].sparse || src[i].merge) {
            buf_ids.resize((size_t)n);
            buf_scores.resize((size_t)n);
            int32_t got = 0;
            pvs_status s =
                src[i].sparse
                    ? pbm_next(src[i].sparse, (int32_t)n, buf_ids.data(), buf_scores.data(), &got)
                    : pvs_merge_next(src[i].merge, (int32_t)n, buf_ids.data(), buf_scores.data(),
                                     &got);
            if (s < 0) return s;
            if (!record(i, buf_ids.data(), got)) return PVS_ERR_INVALID;
            if (s == PVS_EXHAUSTED) exhausted[i] = true;
        } else {
            const int64_t take = std::min<int64_t>(n, src[i].length - depth[i]);
            if (!record(i, src[i].list + depth[i], take)) return PVS_ERR_INVALID;
            if (depth[i] == src[i].length) exhausted[i] = true;
        }
        if (depth[i] >= src[i].length) exhausted[i] = true;
        if (exhausted[i]) src[i].length = depth[i];
        return PVS_OK;
    }
};

// Whether two snapshots (null: every row of `rows` visible) have one visible set.
bool same_visible(const pvs::SnapData* a, const pvs::SnapData* b, int64_t rows) {
    if (a == b) return true;
    const bool a_all = !a || a->visible == a->rows;
    const bool b_all = !b || b->visible == b->rows;
    if ((a && a->rows != rows) || (b && b->rows != rows)) return false;
    if (a_all || b_all) return a_all && b_all;
    return a->h_tomb == b->h_tomb;
}

bool contrib_from(const eahr_params* p, int i, int64_t max_rank, Contrib* out) {
    const int64_t wn = p->w_num[i], wd = p->w_den[i];
    if (wn < 0 || wn >= (1 << 16) || wd < 1 || wd >= (1 << 16)) return false;
    Contrib c;
    c.a = (uint64_t)wn;
    c.b = (uint64_t)wd;
    if (p->form == EAHR_RANK_SCALED)
        c.c = (uint64_t)(p->k - 1) * (uint64_t)wn;     // 1/(r q/p + k - 1) = p/(q r + (k-1) p)
    else
        c.c = (uint64_t)wd * (uint64_t)p->k;           // (p/q)/(k + r) = p/(q r + q k)
    if (c.a == 0) c.c = 0;
    // denominators must stay below 2^32 up to rank max_rank + 1
    const u128 dmax = (u128)c.b * (u128)(max_rank + 1) + c.c;
    if (dmax >= ((u128)1 << 32) || (c.a != 0 && c.b * 1 + c.c == 0)) return false;
    *out = c;
    return true;
}

pvs_status run_driver(Driver& d, const eahr_params* p, int64_t* out_ids, double* out_F,
                      int32_t* n_out, eahr_stats* st);

// The driver behind every entry point: allocation failures (prefixes of
// millions of ranks) become PVS_ERR_OOM instead of leaving the C ABI.
pvs_status run(Driver& d, const eahr_params* p, int64_t* out_ids, double* out_F, int32_t* n_out,
               eahr_stats* st) {
    try {
        return run_driver(d, p, out_ids, out_F, n_out, st);
    } catch (const std::bad_alloc&) {
        return PVS_ERR_OOM;
    }
}

// EAHR_POLICY_ADAPTIVE's finish (Sec. 2.2, last paragraph): complete-list
// fusion of the dense cursor's query and the host sparse list on the device,
// then T*_K from the candidates it returns, ordered by exact rational F
// (ties: smaller id first), zero-score items never appended (Sec. 2.1).
// The switch: once the ranks read reach a sixteenth of both lists, but at
// least kCompleteMin and at most kCompleteMax (the device finish costs about
// one full scoring of the corpus, which reading deeper soon exceeds).
constexpr int64_t kCompleteMin = (int64_t)1 << 16;
constexpr int64_t kCompleteMax = (int64_t)1 << 18;

pvs_status finish_complete(Driver& d, const eahr_params* p, int64_t* out_ids, double* out_F,
                           int32_t* n_out, eahr_stats* st) {
    d.join_ahead();
    pvs::FuseWeights w;
    for (int i = 0; i < 2; ++i) {
        w.a[i] = d.active[i] ? (double)d.g[i].a : 0.0;
        w.b[i] = (double)d.g[i].b;
        w.c[i] = (double)d.g[i].c;
    }
    std::vector<pvs::FusedCand> cand;
    pvs_status s = pvs::fuse_complete(d.src[0].cursor, d.src[1].list, d.src[1].length, w, p->K,
                                      &cand);
    if (s != PVS_OK) return s;
    std::vector<Node> nodes;
    nodes.reserve(cand.size());
    for (const pvs::FusedCand& c : cand) {
        Frac F;
        if (d.active[0] && c.rd > 0) F = add(F, d.g[0].at(c.rd));
        if (d.active[1] && c.rs > 0) F = add(F, d.g[1].at(c.rs));
        if (F.num != 0) nodes.push_back(Node{F, c.id});
    }
    std::sort(nodes.begin(), nodes.end(), NodeCmp());
    const int32_t q = (int32_t)std::min<size_t>((size_t)p->K, nodes.size());
    for (int32_t t = 0; t < q; ++t) {
        out_ids[t] = nodes[(size_t)t].id;
        if (out_F) out_F[t] = frac_to_double(nodes[(size_t)t].F);
    }
    *n_out = q;
    if (st) {
        for (int i = 0; i < 2; ++i) {
            st->depth[i] = d.src[i].length;   // both lists used to the end
            st->length[i] = d.src[i].length;
            st->exhausted[i] = d.active[i] ? 1 : 0;
            st->pulls[i] = d.pulls[i];
        }
        st->checks = d.checks;
        st->complete = 1;
    }
    return PVS_OK;
}

// EAHR_POLICY_ADAPTIVE's cheaper finish: exact ranks for the few items that
// can still be in T*_K.  Let LB be the K-th largest L(x) over the items read
// so far.  An item y with U(y) < LB cannot be in T*_K, because K items have
// F >= L >= LB > F(y); neither can an unread item when B < LB.  The others
// (the candidates) get their missing ranks from the device: the dense rank
// by counting the rows above the item's exact score, the sparse one from the
// host list.  Their F is then exact, and T*_K is their best K by (F desc, id
// asc), zero scores excluded (Sec. 2.1).  Returns PVS_OK with *handled false
// when it does not apply (B >= LB, fewer than K items read, too many
// candidates: *retry stays true; a cursor without bounds of every row:
// *retry false); the driver then reads on.
constexpr int64_t kQueryAt = (int64_t)1 << 12;   // ranks read (both lists) before it is tried

// Certification (Sec. 2.2) over a closed candidate set whose F lies in
// [lo[t].F, hi[t].F]: repeatedly, the candidate first by (lower bound desc,
// id asc) is next when its (lower bound, id) beats the (upper bound, id) of
// every other candidate left.  Fills *order with up to K candidate indices,
// zero scores excluded (Sec. 2.1); false when the bounds leave the order
// open.
bool order_by_bounds(const std::vector<Node>& lo, const std::vector<Node>& hi, int K,
                     std::vector<int32_t>* order) {
    order->clear();
    const size_t n = lo.size();
    std::vector<int32_t> by_lo(n), by_hi(n);
    for (size_t t = 0; t < n; ++t) by_lo[t] = by_hi[t] = (int32_t)t;
    std::sort(by_lo.begin(), by_lo.end(),
              [&](int32_t a, int32_t b) { return NodeCmp()(lo[(size_t)a], lo[(size_t)b]); });
    std::sort(by_hi.begin(), by_hi.end(),
              [&](int32_t a, int32_t b) { return NodeCmp()(hi[(size_t)a], hi[(size_t)b]); });
    std::vector<uint8_t> taken(n, 0);
    size_t p_lo = 0, p_hi = 0;
    while ((int)order->size() < K) {
        while (p_lo < n && taken[(size_t)by_lo[p_lo]]) ++p_lo;
        if (p_lo == n) break;
        const int32_t x = by_lo[p_lo];
        while (p_hi < n && taken[(size_t)by_hi[p_hi]]) ++p_hi;
        // the strongest other candidate by (upper bound, id)
        size_t q = p_hi;
        if (q < n && by_hi[q] == x) {
            ++q;
            while (q < n && taken[(size_t)by_hi[q]]) ++q;
        }
        if (q < n && !beats(lo[(size_t)x].F, lo[(size_t)x].id, hi[(size_t)by_hi[q]].F,
                            hi[(size_t)by_hi[q]].id))
            return false;
        if (lo[(size_t)x].F.num == 0) {   // nothing left with a positive score
            if (hi[(size_t)x].F.num != 0) return false;
            break;
        }
        order->push_back(x);
        taken[(size_t)x] = 1;
    }
    return true;
}

pvs_status finish_rank_queries(Driver& d, const eahr_params* p, int64_t* out_ids, double* out_F,
                               int32_t* n_out, eahr_stats* st, bool* handled, bool* retry) {
    *handled = false;
    *retry = true;
    pvs_cursor* c = d.src[0].cursor;
    // ranks already pulled are recorded first: the helper thread's pull, and
    // any ranks the cursor computed ahead (served without device work), so
    // that every item still unread is also undelivered by the cursor
    if (d.ahead_live) {
        d.join_ahead();
        if (d.ahead_status < 0) return d.ahead_status;
        d.pulls[0]++;
        if (!d.record(0, d.ahead_ids, d.ahead_got)) return PVS_ERR_INVALID;
        if (d.ahead_status == PVS_EXHAUSTED || d.depth[0] >= d.src[0].length) {
            d.exhausted[0] = true;
            d.src[0].length = d.depth[0];
        }
        if (d.certify()) return PVS_OK;   // the extra ranks decided it: the caller reports
    }
    if (!d.exhausted[0] && c->ahead > 0) {
        pvs_status s = d.pull(0, c->ahead);
        if (s < 0) return s;
        if (d.certify()) return PVS_OK;
    }
    const int K = p->K;
    // the K-th largest L over the items read (each once): binary64 values
    // (within 2^-50, relative) find the items that can hold it, all those
    // within 10^-12 of the K-th largest value or above, and exact rationals
    // decide among them
    struct Approx {
        double v;
        int32_t id;
    };
    std::vector<Approx> known;
    known.reserve(d.prefix[0].size() + d.prefix[1].size());
    for (int32_t x : d.prefix[0]) known.push_back(Approx{d.L_d(x), x});
    for (int32_t x : d.prefix[1])
        if (!d.rank(0, x)) known.push_back(Approx{d.L_d(x), x});
    if ((int64_t)known.size() < K) return PVS_OK;
    std::nth_element(known.begin(), known.begin() + (K - 1), known.end(),
                     [](const Approx& a, const Approx& b) { return a.v > b.v; });
    const double near = known[(size_t)K - 1].v * (1.0 - 1e-12);
    std::vector<Node> top;
    for (const Approx& a : known)
        if (a.v >= near) top.push_back(Node{d.L(a.id), a.id});
    std::nth_element(top.begin(), top.begin() + (K - 1), top.end(), NodeCmp());
    const Frac LB = top[(size_t)K - 1].F;
    if (LB.num == 0 || cmp(add(d.u(0), d.u(1)), LB) >= 0) return PVS_OK;
    // candidates and the ranks they miss (U below LB by more than 10^-12 in
    // binary64 is below it exactly)
    const double LB_d = (double)LB.num / (double)LB.den;
    std::vector<int32_t> cand, need_d, need_s;
    for (const Approx& a : known) {
        if (d.U_d(a.id) < LB_d * (1.0 - 1e-12) || cmp(d.U(a.id), LB) < 0) continue;
        cand.push_back(a.id);
        for (int i = 0; i < 2; ++i) {
            if (!d.active[i] || d.exhausted[i] || d.rank(i, a.id)) continue;
            (i == 0 ? need_d : need_s).push_back(a.id);
        }
    }
    if ((int64_t)need_d.size() > pvs::kRankQueryMax || (int64_t)need_s.size() > pvs::kRankQueryMax)
        return PVS_OK;
    // first the dense rank intervals the rows' bounds give (no row scored)
    std::vector<int64_t> rd_lo(need_d.size()), rd_hi(need_d.size()), rs(need_s.size());
    const pvs::StagedList* staged = need_s.empty() ? nullptr : d.staged_list();
    if (!need_s.empty() && !staged && !d.src[1].list) {   // a PBM source that could not be staged
        *retry = false;
        return PVS_OK;
    }
    bool supported = false;
    pvs_status s = pvs::rank_queries(c, need_d.data(), (int32_t)need_d.size(), false,
                                     d.src[1].list, d.src[1].list ? d.src[1].length : 0,
                                     need_s.data(), (int32_t)need_s.size(), rd_lo.data(),
                                     rd_hi.data(), rs.data(), &supported, staged);
    if (s != PVS_OK) return s;
    if (!supported) {   // this cursor never supports it
        *retry = false;
        return PVS_OK;
    }
    // F of every candidate, an interval while a dense rank is one
    std::vector<size_t> at_d(cand.size(), SIZE_MAX), at_s(cand.size(), SIZE_MAX);
    {
        std::vector<std::pair<int32_t, size_t>> pos(cand.size());
        for (size_t t = 0; t < cand.size(); ++t) pos[t] = {cand[t], t};
        std::sort(pos.begin(), pos.end());
        auto slot = [&](int32_t x) {
            return std::lower_bound(pos.begin(), pos.end(), std::make_pair(x, (size_t)0))->second;
        };
        for (size_t t = 0; t < need_d.size(); ++t) at_d[slot(need_d[t])] = t;
        for (size_t t = 0; t < need_s.size(); ++t) at_s[slot(need_s[t])] = t;
    }
    std::vector<Node> lo(cand.size()), hi(cand.size());
    auto fill = [&]() {
        for (size_t t = 0; t < cand.size(); ++t) {
            const int32_t x = cand[t];
            Frac Fl, Fh;
            for (int i = 0; i < 2; ++i) {
                if (!d.active[i]) continue;
                int64_t r = d.rank(i, x), r_hi = r;
                if (!r && i == 0 && at_d[t] != SIZE_MAX) {
                    r = rd_lo[at_d[t]];
                    r_hi = rd_hi[at_d[t]];
                } else if (!r && i == 1 && at_s[t] != SIZE_MAX) {
                    r = r_hi = rs[at_s[t]];
                }
                if (r > 0) {
                    Fh = add(Fh, d.g[i].at(r));
                    Fl = add(Fl, d.g[i].at(r_hi));
                }
            }
            lo[t] = Node{Fl, x};
            hi[t] = Node{Fh, x};
        }
    };
    fill();
    std::vector<int32_t> order;
    bool scored = false;
    // While the intervals leave the order open, exact dense ranks for the
    // candidates whose F interval is wider than a point and overlaps another
    // one that can still reach the Top-K (only they can hold the order up);
    // the rows around each such candidate's score are scored.  A last round
    // makes every dense rank exact, which decides the order.
    for (int round = 0; !order_by_bounds(lo, hi, K, &order); ++round) {
        scored = true;
        std::vector<size_t> pick;   // indices into need_d
        if (round < 3) {
            std::vector<Node> lows(lo);
            std::nth_element(lows.begin(), lows.begin() + (std::ptrdiff_t)(K - 1), lows.end(),
                             NodeCmp());
            const Frac floor_k = lows[(size_t)K - 1].F;   // the K-th largest lower bound
            std::vector<size_t> rel;
            for (size_t t = 0; t < cand.size(); ++t)
                if (cmp(hi[t].F, floor_k) >= 0) rel.push_back(t);
            for (size_t t : rel) {
                if (at_d[t] == SIZE_MAX || cmp(lo[t].F, hi[t].F) == 0) continue;
                for (size_t u : rel)
                    if (u != t && cmp(lo[t].F, hi[u].F) <= 0 && cmp(lo[u].F, hi[t].F) <= 0) {
                        pick.push_back(at_d[t]);
                        break;
                    }
            }
        }
        if (pick.empty())   // the last round: every dense rank
            for (size_t j = 0; j < need_d.size(); ++j)
                if (rd_lo[j] != rd_hi[j]) pick.push_back(j);
        if (pick.empty()) break;   // cannot happen: point intervals decide
        std::vector<int32_t> ids(pick.size());
        std::vector<int64_t> plo(pick.size()), phi(pick.size());
        for (size_t j = 0; j < pick.size(); ++j) ids[j] = need_d[pick[j]];
        s = pvs::rank_queries(c, ids.data(), (int32_t)ids.size(), true, nullptr, 0, nullptr, 0,
                              plo.data(), phi.data(), nullptr, &supported);
        if (s != PVS_OK) return s;
        for (size_t j = 0; j < pick.size(); ++j) {
            rd_lo[pick[j]] = plo[j];
            rd_hi[pick[j]] = phi[j];
        }
        fill();
    }
    // F is reported where it is known exactly (a point interval), NaN where
    // only the position is certified (as for an item unread in an Open list)
    const int32_t q = (int32_t)order.size();
    for (int32_t t = 0; t < q; ++t) {
        const size_t u = (size_t)order[(size_t)t];
        out_ids[t] = lo[u].id;
        if (out_F)
            out_F[t] = cmp(lo[u].F, hi[u].F) == 0 ? frac_to_double(lo[u].F) : std::nan("");
    }
    *n_out = q;
    if (st) {
        for (int i = 0; i < 2; ++i) {
            st->depth[i] = d.depth[i];
            st->length[i] = d.src[i].length;
            st->exhausted[i] = d.exhausted[i] ? 1 : 0;
            st->pulls[i] = d.pulls[i];
        }
        st->checks = d.checks;
        st->complete = scored ? 3 : 2;
    }
    *handled = true;
    return PVS_OK;
}

pvs_status run_driver(Driver& d, const eahr_params* p, int64_t* out_ids, double* out_F,
                      int32_t* n_out, eahr_stats* st) {
    const bool adaptive = p->policy == EAHR_POLICY_ADAPTIVE && d.src[0].cursor &&
                          (d.src[1].list || d.src[1].sparse);
    if (adaptive) d.start_stage();
    // the adaptive policy reads its first kQueryAt ranks in one pull per list
    // (its finish is tried there; fewer, larger pulls cost fewer round trips)
    const int step0 = p->step > 0 ? p->step : (adaptive ? (int)(kQueryAt / 2) : 16);
    const int64_t complete_at = std::min(
        kCompleteMax, std::max<int64_t>(kCompleteMin, (d.src[0].length + d.src[1].length) / 16));
    int64_t query_at = kQueryAt;
    int64_t size[2] = {step0, step0};
    d.K = p->K;
    d.both.cap = (size_t)p->K + 2;
    for (int i = 0; i < 2; ++i)
        if (!d.active[i]) d.exhausted[i] = false;
    // lists with zero weight contribute nothing and are never read
    bool done = false;
    if (!d.active[0] && !d.active[1]) done = true;
    // frozen scheduler state (Sec. 3.5)
    int skipped[2] = {0, 0};
    int64_t next_check = 0;   // access at which the next sparse-cadence check falls due
    const int64_t dense_checks = 4 * (int64_t)p->K;   // every step checked until 4K ranks are read
    while (!done) {
        if (p->policy == EAHR_POLICY_FROZEN) {
            int pick = -1;
            for (int i = 0; i < 2; ++i) {
                if (!d.active[i] || d.exhausted[i]) continue;
                if (pick < 0) {
                    pick = i;
                    continue;
                }
                const int c = cmp(d.u(i), d.u(pick));
                if (c > 0 || (c == 0 && d.depth[i] < d.depth[pick])) pick = i;
            }
            if (pick >= 0) {
                const int other = 1 - pick;
                const bool other_open = d.active[other] && !d.exhausted[other];
                if (other_open && skipped[other] >= 16) pick = other;   // fairness
                const bool was[2] = {d.exhausted[0], d.exhausted[1]};
                pvs_status s = d.pull(pick, step0);
                if (s < 0) return s;
                skipped[pick] = 0;
                const int o = 1 - pick;
                if (d.active[o] && !d.exhausted[o]) ++skipped[o];
                const int64_t access = d.depth[0] + d.depth[1];
                const bool newly = (d.exhausted[0] && !was[0]) || (d.exhausted[1] && !was[1]);
                if (!(access <= dense_checks || newly || access >= next_check)) continue;
                next_check = access + std::min<int64_t>(1024, std::max<int64_t>(64, access / 8));
            }
        } else if (p->policy == EAHR_POLICY_EQUAL_DEPTH) {
            for (int i = 0; i < 2; ++i) {
                pvs_status s = d.pull(i, step0);
                if (s < 0) return s;
            }
        } else {
            // the list whose next unread rank can still contribute more
            int pick = -1;
            for (int i = 0; i < 2; ++i) {
                if (!d.active[i] || d.exhausted[i]) continue;
                if (pick < 0) {
                    pick = i;
                    continue;
                }
                const int c = cmp(d.u(i), d.u(pick));
                if (c > 0 || (c == 0 && d.depth[i] < d.depth[pick])) pick = i;
            }
            if (pick >= 0) {
                pvs_status s = d.pull(pick, size[pick]);
                if (s < 0) return s;
                size[pick] = std::min<int64_t>(2 * size[pick], (int64_t)1 << 24);
                if (adaptive && pick == 0) d.check_stage();
            }
            // long dense pulls: the next one starts now, beside certification
            // and the other list's pull (ranks read ahead change no result)
            if (size[0] >= kAheadMin) d.start_ahead(size[0]);
        }
        done = d.certify();
        if (!done && adaptive && d.depth[0] + d.depth[1] >= query_at) {
            bool handled = false, retry = true;
            pvs_status s = finish_rank_queries(d, p, out_ids, out_F, n_out, st, &handled, &retry);
            if (s < 0) return s;
            if (handled) return PVS_OK;
            done = d.certify();   // ranks the attempt recorded may have decided it
            // else again after as much reading, or never
            query_at = retry ? 2 * (d.depth[0] + d.depth[1]) : std::numeric_limits<int64_t>::max();
        }
        if (!done && adaptive && d.src[1].list && d.depth[0] + d.depth[1] >= complete_at)
            return finish_complete(d, p, out_ids, out_F, n_out, st);
        if (!done) {
            bool any_open = false;
            for (int i = 0; i < 2; ++i) any_open |= d.active[i] && !d.exhausted[i];
            if (!any_open) done = true;   // cannot happen: exhausted lists decide
        }
    }
    const int32_t q = (int32_t)d.A.size();
    for (int32_t t = 0; t < q; ++t) {
        const int32_t x = d.A[t];
        out_ids[t] = x;
        if (out_F) {
            bool determined = true;
            for (int i = 0; i < 2; ++i)
                if (d.active[i] && !d.exhausted[i] && !d.rank(i, x)) determined = false;
            out_F[t] = determined ? frac_to_double(d.L(x)) : std::nan("");
        }
    }
    *n_out = q;
    if (st) {
        for (int i = 0; i < 2; ++i) {
            st->depth[i] = d.depth[i];
            st->length[i] = d.src[i].length;
            st->exhausted[i] = d.exhausted[i] ? 1 : 0;
            st->pulls[i] = d.pulls[i];
        }
        st->checks = d.checks;
        st->complete = 0;
    }
    return PVS_OK;
}

bool params_ok(const eahr_params* p) {
    return p && p->K >= 1 && p->k >= 1 && (p->form == EAHR_RANK_SCALED || p->form == EAHR_NUMERATOR) &&
           (p->policy == EAHR_POLICY_GEOMETRIC || p->policy == EAHR_POLICY_EQUAL_DEPTH ||
            p->policy == EAHR_POLICY_FROZEN || p->policy == EAHR_POLICY_ADAPTIVE) &&
           p->step >= 0;
}

}  // namespace

extern "C" {

pvs_status eahr_topk(pvs_cursor* dense, const int64_t* sparse_ids, int64_t n_sparse,
                     const eahr_params* p, int64_t* out_ids, double* out_F, int32_t* n_out,
                     eahr_stats* st) {
    if (n_out) *n_out = 0;
    if (!dense || !params_ok(p) || !out_ids || !n_out || n_sparse < 0 ||
        (n_sparse > 0 && !sparse_ids))
        return PVS_ERR_INVALID;
    if (pvs::cursor_emitted(dense) != 0) return PVS_ERR_INVALID;
    const pvs::SnapData* snap = pvs::cursor_snapshot(dense);
    const int64_t id_space = snap->rows;
    if (n_sparse > snap->visible) return PVS_ERR_INVALID;
    Driver d;
    d.snap = snap;
    d.src[0].cursor = dense;
    d.src[0].length = pvs::cursor_visible(dense);
    d.src[1].list = sparse_ids;
    d.src[1].length = n_sparse;
    for (int i = 0; i < 2; ++i) {
        if (!contrib_from(p, i, d.src[i].length, &d.g[i])) return PVS_ERR_INVALID;
        d.active[i] = d.g[i].a != 0;
        if (d.src[i].length == 0) d.exhausted[i] = true;
    }
    if (!d.init(id_space)) return PVS_ERR_OOM;
    return run(d, p, out_ids, out_F, n_out, st);
}

pvs_status eahr_topk_lists(const int64_t* list0, int64_t n0, const int64_t* list1, int64_t n1,
                           const eahr_params* p, int64_t* out_ids, double* out_F, int32_t* n_out,
                           eahr_stats* st) {
    if (n_out) *n_out = 0;
    if (!params_ok(p) || !out_ids || !n_out || n0 < 0 || n1 < 0 || (n0 > 0 && !list0) ||
        (n1 > 0 && !list1))
        return PVS_ERR_INVALID;
    // one pass per list: the id space (largest id + 1) and no negative id
    int64_t id_space = 0, lowest = 0;
    for (int i = 0; i < 2; ++i) {
        int64_t hi = -1, lo = 0;
        id_range(i == 0 ? list0 : list1, i == 0 ? n0 : n1, &lo, &hi);
        id_space = std::max(id_space, hi + 1);
        lowest = std::min(lowest, lo);
    }
    if (lowest < 0) return PVS_ERR_INVALID;
    if (id_space > ((int64_t)1 << 31)) return PVS_ERR_INVALID;
    Driver d;
    d.src[0].list = list0;
    d.src[0].length = n0;
    d.src[1].list = list1;
    d.src[1].length = n1;
    for (int i = 0; i < 2; ++i) {
        if (!contrib_from(p, i, d.src[i].length, &d.g[i])) return PVS_ERR_INVALID;
        d.active[i] = d.g[i].a != 0;
        if (d.src[i].length == 0) d.exhausted[i] = true;
    }
    if (!d.init(id_space)) return PVS_ERR_OOM;
    return run(d, p, out_ids, out_F, n_out, st);
}

pvs_status eahr_topk_pbm(pvs_cursor* dense, pbm_cursor* sparse, const eahr_params* p,
                         int64_t* out_ids, double* out_F, int32_t* n_out, eahr_stats* st) {
    if (n_out) *n_out = 0;
    if (!dense || !sparse || !params_ok(p) || !out_ids || !n_out) return PVS_ERR_INVALID;
    if (pvs::cursor_emitted(dense) != 0) return PVS_ERR_INVALID;
    pbm_stats ps;
    if (pbm_cursor_stats(sparse, &ps) != PVS_OK || ps.emitted != 0 || ps.state < 0)
        return PVS_ERR_INVALID;
    const pvs::SnapData* snap = pvs::cursor_snapshot(dense);
    // both channels rank items of one visible set (Sec. 2.4)
    if (ps.items != snap->rows || !same_visible(snap, pvs::pbm_cursor_snapshot(sparse), snap->rows))
        return PVS_ERR_INVALID;
    Driver d;
    d.snap = snap;
    d.src[0].cursor = dense;
    d.src[0].length = pvs::cursor_visible(dense);
    d.src[1].sparse = sparse;
    d.src[1].length = ps.items;
    for (int i = 0; i < 2; ++i) {
        if (!contrib_from(p, i, d.src[i].length, &d.g[i])) return PVS_ERR_INVALID;
        d.active[i] = d.g[i].a != 0;
        if (d.src[i].length == 0) d.exhausted[i] = true;
    }
    if (!d.init(snap->rows)) return PVS_ERR_OOM;
    return run(d, p, out_ids, out_F, n_out, st);
}

pvs_status eahr_topk_merge(pvs_merge* dense, pvs_merge* sparse, const eahr_params* p,
                           int64_t* out_ids, double* out_F, int32_t* n_out, eahr_stats* st) {
    if (n_out) *n_out = 0;
    if (!dense || !sparse || dense == sparse || !params_ok(p) || !out_ids || !n_out)
        return PVS_ERR_INVALID;
    if (!pvs::merge_fresh(dense) || !pvs::merge_fresh(sparse)) return PVS_ERR_INVALID;
    const int64_t id_space = std::max(pvs::merge_id_space(dense), pvs::merge_id_space(sparse));
    Driver d;
    d.src[0].merge = dense;
    d.src[0].length = pvs::merge_length(dense);
    d.src[1].merge = sparse;
    d.src[1].length = pvs::merge_length(sparse);
    for (int i = 0; i < 2; ++i) {
        if (!contrib_from(p, i, d.src[i].length, &d.g[i])) return PVS_ERR_INVALID;
        d.active[i] = d.g[i].a != 0;
        if (d.src[i].length == 0) d.exhausted[i] = true;
    }
    if (!d.init(id_space)) return PVS_ERR_OOM;
    return run(d, p, out_ids, out_F, n_out, st);
}

}  // extern "C"
