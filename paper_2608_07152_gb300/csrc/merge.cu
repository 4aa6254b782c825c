// Hierarchical Segment / Shard merging (include/merge.h): arXiv 2608.07152
// Sec. 2.4, ranked-list contract of Sec. 2.1.
//
// Host code over device-backed children: a k-way merge of the children's
// exact rankings under the rank key (score descending, id ascending).  Each
// child keeps a buffer of ranks read but not yet delivered; before an item
// is delivered, every child that is not exhausted has a non-empty buffer, so
// the item precedes everything any child can still produce (each child's
// later ranks have smaller keys than its buffered ones).  Refill sizes start
// from the request size spread over the children and double per refill.
//
// Refills are host round trips to the children's devices.  When a child runs
// dry, every other child whose buffer is down to a quarter of its next
// refill is refilled with it, and a round of several refills runs on one
// host thread per child (each child is its own cursor with its own state),
// so the round trips of one round overlap.  What is read ahead stays in the
// buffers; the merged order does not depend on it.
#include <algorithm>
#include <cstring>
#include <new>
#include <thread>
#include <unordered_set>
#include <vector>

#include "../../include/merge.h"
#include "pvs_common.cuh"
#include "runtime.h"

namespace {

constexpr int32_t kMaxChildren = 1024;
constexpr int64_t kMaxChunk = int64_t(1) << 20;

struct Child {
    int32_t kind = PVS_CHILD_DENSE;
    void* cur = nullptr;
    int64_t off = 0;
    int64_t length = 0;      // list length (upper bound for merges)
    int64_t id_space = 0;    // request ids of this child lie below this
    std::vector<int64_t> ids;
    std::vector<float> scores;
    size_t head = 0;
    bool exhausted = false;
    int64_t chunk = 0;       // next refill size
    // result of the last refill (written by the thread that ran it)
    pvs_status status = PVS_OK;
    int64_t got = 0;
    uint64_t key = 0;        // rank key of the buffered head (while left() > 0)
    size_t left() const { return ids.size() - head; }
    void set_key() { key = pvs::rank_key(scores[head], (uint32_t)ids[head]); }
};

constexpr size_t kRefillThreads = 16;   // concurrent refills per round

}  // namespace

struct pvs_merge {
    std::vector<Child> ch;
    // winner tree over the children's head keys: node i holds the child with
    // the larger key of nodes 2i and 2i+1, leaf P + c child c (-1: none)
    std::vector<int32_t> tree;
    int32_t P = 1;
    int64_t id_space = 0, length = 0;
    std::vector<uint64_t> seen;   // delivered request ids (bitmap)
    uint64_t last_key = 0;
    bool any = false;
    int64_t emitted = 0, read = 0, dups = 0, child_pulls = 0;
    int state = PVS_OK;
};

namespace {

pvs_status fail(pvs_merge* m, pvs_status s) {
    if (s < 0 && m->state >= 0) m->state = s;
    return s;
}

// Facts about a fresh child: list length and id space (in its own ids).
pvs_status describe(const pvs_merge_child& c, int64_t* length, int64_t* id_space) {
    switch (c.kind) {
        case PVS_CHILD_DENSE: {
            pvs_cursor* p = static_cast<pvs_cursor*>(c.cursor);
            pvs_stats st;
            if (pvs_cursor_stats(p, &st) != PVS_OK || st.state < 0 || st.emitted != 0)
                return PVS_ERR_INVALID;
            *length = st.visible;
            *id_space = pvs::cursor_snapshot(p)->rows;
            return PVS_OK;
        }
        case PVS_CHILD_SPARSE: {
            pbm_stats st;
            if (pbm_cursor_stats(static_cast<pbm_cursor*>(c.cursor), &st) != PVS_OK ||
                st.state < 0 || st.emitted != 0)
                return PVS_ERR_INVALID;
            *length = st.items;
            *id_space = st.items;
            return PVS_OK;
        }
        case PVS_CHILD_MERGE: {
            pvs_merge* g = static_cast<pvs_merge*>(c.cursor);
            if (g->state < 0 || g->emitted != 0 || g->read != 0) return PVS_ERR_INVALID;
            *length = g->length;
            *id_space = g->id_space;
            return PVS_OK;
        }
        default:
            return PVS_ERR_INVALID;
    }
}

// Append up to n ranks of a child to its buffer (what was delivered is
// dropped first).  Touches only the child: rounds run children concurrently.
void refill(Child& c, int64_t n) {
    c.ids.erase(c.ids.begin(), c.ids.begin() + (std::ptrdiff_t)c.head);
    c.scores.erase(c.scores.begin(), c.scores.begin() + (std::ptrdiff_t)c.head);
    c.head = 0;
    const size_t old = c.ids.size();
    c.ids.resize(old + (size_t)n);
    c.scores.resize(old + (size_t)n);
    int32_t got = 0;
    pvs_status s;
    int64_t* ids = c.ids.data() + old;
    float* scores = c.scores.data() + old;
    switch (c.kind) {
        case PVS_CHILD_DENSE:
            s = pvs_next(static_cast<pvs_cursor*>(c.cur), (int32_t)n, ids, scores, &got);
            break;
        case PVS_CHILD_SPARSE:
            s = pbm_next(static_cast<pbm_cursor*>(c.cur), (int32_t)n, ids, scores, &got);
            break;
        default:
            s = pvs_merge_next(static_cast<pvs_merge*>(c.cur), (int32_t)n, ids, scores, &got);
            break;
    }
    if (s < 0) got = 0;
    c.ids.resize(old + (size_t)got);
    c.scores.resize(old + (size_t)got);
    for (size_t k = old; k < c.ids.size(); ++k) c.ids[k] += c.off;
    if (c.left()) c.set_key();
    c.status = s;
    c.got = got;
    if (s == PVS_EXHAUSTED) c.exhausted = true;
}

// One round: refill every child that is dry, and with them every child that
// is down to a quarter of its next refill.  Returns the first error.
pvs_status refill_round(pvs_merge* m, int32_t n) {
    const int64_t k = (int64_t)m->ch.size();
    std::vector<Child*> due;
    bool dry = false;
    for (Child& c : m->ch) {
        if (c.exhausted) continue;
        if (c.chunk == 0) c.chunk = std::max<int64_t>(16, 2 * ((n + k - 1) / k));
        if (c.left() == 0) dry = true;
    }
    if (!dry) return PVS_OK;
    for (Child& c : m->ch)
        if (!c.exhausted && (int64_t)c.left() * 4 <= c.chunk) due.push_back(&c);
    for (size_t b = 0; b < due.size(); b += kRefillThreads) {
        const size_t e = std::min(due.size(), b + kRefillThreads);
        // refills whose thread could not be started run here
        std::vector<std::thread> th;
        size_t started = b + 1;
        try {
            th.reserve(e - b);
            for (; started < e; ++started)
                th.emplace_back(refill, std::ref(*due[started]), due[started]->chunk);
        } catch (...) {
        }
        refill(*due[b], due[b]->chunk);
        for (size_t t = started; t < e; ++t) refill(*due[t], due[t]->chunk);
        for (auto& x : th) x.join();
    }
    pvs_status first = PVS_OK;
    for (Child* c : due) {
        ++m->child_pulls;
        m->read += c->got;
        c->chunk = std::min<int64_t>(c->chunk * 2, kMaxChunk);
        if (c->status < 0 && first == PVS_OK) first = c->status;
    }
    return first;
}

// Key of child c's buffered head; 0 when it has none (real rank keys are
// larger: a finite score's ordered key is at least 2^23).
uint64_t head_key(const pvs_merge* m, int32_t c) {
    if (c < 0) return 0;
    const Child& x = m->ch[(size_t)c];
    return x.left() ? x.key : 0;
}

int32_t winner(const pvs_merge* m, int32_t a, int32_t b) {
    return head_key(m, a) >= head_key(m, b) ? a : b;
}

void tree_build(pvs_merge* m) {
    const int32_t k = (int32_t)m->ch.size();
    for (int32_t c = 0; c < m->P; ++c) m->tree[(size_t)(m->P + c)] = c < k ? c : -1;
    for (int32_t i = m->P - 1; i >= 1; --i)
        m->tree[(size_t)i] = winner(m, m->tree[(size_t)(2 * i)], m->tree[(size_t)(2 * i + 1)]);
}

// Child c's head changed: replay its path to the root.
void tree_update(pvs_merge* m, int32_t c) {
    for (int32_t i = (m->P + c) >> 1; i >= 1; i >>= 1)
        m->tree[(size_t)i] = winner(m, m->tree[(size_t)(2 * i)], m->tree[(size_t)(2 * i + 1)]);
}

bool seen(const pvs_merge* m, int64_t id) {
    return (m->seen[(size_t)(id >> 6)] >> (id & 63)) & 1u;
}

}  // namespace

namespace {
pvs_status merge_next(pvs_merge* m, int32_t n, int64_t* ids, float* scores, int32_t* n_out);
}  // namespace

extern "C" {

pvs_status pvs_merge_open(const pvs_merge_child* children, int32_t count, pvs_merge** out) {
    if (!out) return PVS_ERR_INVALID;
    *out = nullptr;
    if (!children || count < 1 || count > kMaxChildren) return PVS_ERR_INVALID;
    std::unordered_set<void*> distinct;
    pvs_merge* m = new (std::nothrow) pvs_merge();
    if (!m) return PVS_ERR_OOM;
    m->ch.resize((size_t)count);
    for (int32_t i = 0; i < count; ++i) {
        const pvs_merge_child& c = children[i];
        if (!c.cursor || c.id_offset < 0 || !distinct.insert(c.cursor).second) {
            delete m;
            return PVS_ERR_INVALID;
        }
        int64_t length = 0, space = 0;
        if (describe(c, &length, &space) != PVS_OK) {
            delete m;
            return PVS_ERR_INVALID;
        }
        Child& d = m->ch[(size_t)i];
        d.kind = c.kind;
        d.cur = c.cursor;
        d.off = c.id_offset;
        d.length = length;
        d.id_space = c.id_offset + space;
        d.exhausted = length == 0;
        m->id_space = std::max(m->id_space, d.id_space);
        m->length += length;
    }
    if (m->id_space > ((int64_t)1 << 31)) {
        delete m;
        return PVS_ERR_INVALID;
    }
    m->seen.assign((size_t)((m->id_space + 63) / 64), 0ull);
    while (m->P < count) m->P *= 2;
    m->tree.assign((size_t)(2 * m->P), -1);
    *out = m;
    return PVS_OK;
}

// Buffer growth that fails fails the merge cursor (PVS_ERR_OOM) instead of
// leaving the C ABI.
pvs_status pvs_merge_next(pvs_merge* m, int32_t n, int64_t* ids, float* scores, int32_t* n_out) {
    try {
        return merge_next(m, n, ids, scores, n_out);
    } catch (const std::bad_alloc&) {
        if (n_out) *n_out = 0;
        return m ? fail(m, PVS_ERR_OOM) : PVS_ERR_OOM;
    }
}

}  // extern "C"

namespace {

pvs_status merge_next(pvs_merge* m, int32_t n, int64_t* ids, float* scores, int32_t* n_out) {
    if (n_out) *n_out = 0;
    if (!m) return PVS_ERR_INVALID;
    if (m->state < 0) return PVS_ERR_FAILED;
    if (n < 1 || !ids || !scores || !n_out) return PVS_ERR_INVALID;
    int32_t count = 0;
    // every child that can still produce has a buffered head before each
    // item: children left dry by an error-free earlier call are refilled
    // here, and a child that runs dry below right away
    pvs_status s = refill_round(m, n);
    if (s != PVS_OK) return fail(m, s);
    tree_build(m);
    while (count < n) {
        const int32_t b = m->tree[1];
        if (head_key(m, b) == 0) break;   // every child exhausted and delivered
        Child* best = &m->ch[(size_t)b];
        const uint64_t best_key = best->key;
        const int64_t id = best->ids[best->head];
        const float sc = best->scores[best->head];
        ++best->head;
        if (best->left()) {
            best->set_key();
            tree_update(m, b);
        } else if (!best->exhausted) {
            s = refill_round(m, n);   // may refill several children
            if (s != PVS_OK) return fail(m, s);
            tree_build(m);
        } else {
            tree_update(m, b);
        }
        if (m->any && best_key == m->last_key) {   // another copy with the same score
            ++m->dups;
            continue;
        }
        if (id < 0 || id >= m->id_space || seen(m, id))
            return fail(m, PVS_ERR_INVALID);   // a copy with another score: conflict
        m->seen[(size_t)(id >> 6)] |= 1ull << (id & 63);
        ids[count] = id;
        scores[count] = sc;
        ++count;
        m->last_key = best_key;
        m->any = true;
    }
    m->emitted += count;
    *n_out = count;
    bool done = true;
    for (const Child& c : m->ch) done = done && c.exhausted && c.head >= c.ids.size();
    if (done) {
        m->state = PVS_EXHAUSTED;
        return PVS_EXHAUSTED;
    }
    return PVS_OK;
}

}  // namespace

extern "C" {

pvs_status pvs_merge_stats_get(pvs_merge* m, pvs_merge_stats* out) {
    if (!m || !out) return PVS_ERR_INVALID;
    out->emitted = m->emitted;
    out->read = m->read;
    out->duplicates = m->dups;
    out->child_pulls = m->child_pulls;
    out->id_space = m->id_space;
    out->length = m->length;
    out->state = m->state;
    out->reserved = 0;
    return PVS_OK;
}

void pvs_merge_close(pvs_merge* m) { delete m; }

}  // extern "C"

// Facts the EAHR driver needs about a merge cursor.
namespace pvs {
int64_t merge_id_space(const pvs_merge* m) { return m->id_space; }
int64_t merge_length(const pvs_merge* m) { return m->length; }
bool merge_fresh(const pvs_merge* m) { return m->state >= 0 && m->emitted == 0 && m->read == 0; }
}  // namespace pvs
