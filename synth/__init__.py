"""Seeded synthetic workloads for the PVS / EAHR path (no method arithmetic).

The paper's corpora (MS MARCO passages, CORD-19 snapshots encoded with
bge-small) and its sparse BM25 rankings are not available here; these
generators stand in for them with the shapes and structure of the workloads:

* ``unit_normal``        i.i.d. standard normal rows, L2-normalised;
* ``mixture_centres`` / ``mixture_rows`` / ``mixture_queries``
                         a Gaussian mixture (centres ~ N(0, I), uniform
                         component choice, isotropic within-component noise),
                         L2-normalised;
* ``near_duplicate_rows`` copies of chosen rows plus N(0, sigma^2) noise,
                         L2-normalised;
* ``copula_ranking``     a complete ranking whose Kendall tau against the
                         ranking of given proxy scores is about ``tau``
                         (Gaussian copula, rho = sin(pi tau / 2));
* ``controlled_streams`` the rank relations of the controlled-stream study
                         (block-32 correlated, partial overlap, independent,
                         reversed, all tied);
* ``bm25_postings`` / ``sparse_queries`` / ``topical_queries``
                         a stand-in for BM25 impact postings: term draws from
                         a Zipf law (the most frequent ranks removed like
                         stopwords), term frequencies from repeated draws,
                         BM25 weights (k1 = 0.9, b = 0.4) from the corpus's own
                         document frequencies and lengths, as term-major CSR;
                         optionally a share of each item's tokens from a
                         block of terms of its topic (its mixture component,
                         see ``mixture_components``), so that sparse and
                         dense rankings agree in part; queries of a few
                         distinct terms of weight 1.

Every generator is deterministic in its seed; large matrices are produced in
row chunks, each with its own derived seed, so any chunk can be regenerated
alone.  Tensors come out on the requested torch device.
"""
from __future__ import annotations

import math

import numpy as np
import torch

CHUNK_ROWS = 1 << 18


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & ((1 << 63) - 1))
    return g


def _chunk_seed(seed: int, chunk: int) -> int:
    return (int(seed) * 1000003 + 7919 * int(chunk) + 17) & ((1 << 63) - 1)


def _normalise(x: torch.Tensor) -> torch.Tensor:
    return x / torch.linalg.vector_norm(x, dim=1, keepdim=True).clamp_min(1e-30)


def unit_normal(n: int, d: int, seed: int, device="cpu", first: int = 0) -> torch.Tensor:
    """Rows first .. first+n-1 of an i.i.d. N(0, 1) matrix, L2-normalised."""
    out = torch.empty((n, d), dtype=torch.float32, device=device)
    for r in range(0, n, CHUNK_ROWS):
        c = min(CHUNK_ROWS, n - r)
        out[r:r + c] = _rows_normal(first + r, c, d, seed, device)
    return out


def _rows_normal(row0: int, count: int, d: int, seed: int, device) -> torch.Tensor:
    # row0 is aligned to CHUNK_ROWS by every caller that regenerates chunks
    chunk = row0 // CHUNK_ROWS
    x = torch.randn((count, d), generator=_gen(_chunk_seed(seed, chunk), device),
                    device=device, dtype=torch.float32)
    return _normalise(x)


def mixture_centres(n_components: int, d: int, seed: int, device="cpu") -> torch.Tensor:
    return torch.randn((n_components, d), generator=_gen(_chunk_seed(seed, -1), device),
                       device=device, dtype=torch.float32)


def mixture_rows(n: int, centres: torch.Tensor, within_std: float, seed: int,
                 first: int = 0) -> torch.Tensor:
    """Rows first .. first+n-1 of a mixture: centre[c] + within_std * N(0, I),
    c uniform over the components, L2-normalised."""
    device = centres.device
    k, d = centres.shape
    out = torch.empty((n, d), dtype=torch.float32, device=device)
    for r in range(0, n, CHUNK_ROWS):
        c = min(CHUNK_ROWS, n - r)
        g = _gen(_chunk_seed(seed, (first + r) // CHUNK_ROWS), device)
        comp = torch.randint(0, k, (c,), generator=g, device=device)
        x = torch.randn((c, d), generator=g, device=device, dtype=torch.float32)
        x.mul_(within_std).add_(centres[comp])
        out[r:r + c] = _normalise(x)
    return out


def mixture_components(n: int, n_components: int, seed: int, device="cpu") -> torch.Tensor:
    """The mixture component of rows 0 .. n-1 of mixture_rows(seed=seed) on
    the same device type: the same generator draws, replayed."""
    out = torch.empty(n, dtype=torch.int64, device=device)
    for r in range(0, n, CHUNK_ROWS):
        c = min(CHUNK_ROWS, n - r)
        g = _gen(_chunk_seed(seed, r // CHUNK_ROWS), device)
        out[r:r + c] = torch.randint(0, n_components, (c,), generator=g, device=device)
    return out


def mixture_query_components(nq: int, n_components: int, seed: int, device="cpu") -> torch.Tensor:
    """The component of each query of mixture_queries(seed=seed), replayed."""
    g = _gen(_chunk_seed(seed, -2), device)
    return torch.randint(0, n_components, (nq,), generator=g, device=device)


def mixture_queries(nq: int, centres: torch.Tensor, noise_std: float, seed: int) -> torch.Tensor:
    """Queries: a uniformly chosen centre + noise_std * N(0, I), normalised."""
    device = centres.device
    g = _gen(_chunk_seed(seed, -2), device)
    comp = torch.randint(0, centres.shape[0], (nq,), generator=g, device=device)
    x = torch.randn((nq, centres.shape[1]), generator=g, device=device, dtype=torch.float32)
    return _normalise(centres[comp] + noise_std * x)


def near_duplicate_rows(src: torch.Tensor, noise_std: float, seed: int) -> torch.Tensor:
    """Copies of the given rows plus N(0, noise_std^2) noise, normalised."""
    g = _gen(_chunk_seed(seed, -3), src.device)
    x = torch.randn(src.shape, generator=g, device=src.device, dtype=torch.float32)
    return _normalise(src + noise_std * x)


def copula_ranking(proxy_scores: torch.Tensor, tau: float, seed: int) -> torch.Tensor:
    """A complete ranking (int64 ids, best first) of all len(proxy_scores)
    items whose Kendall tau against the proxy-score ranking is about tau:
    key = rho * Phi^-1((n - r + 0.5) / n) + sqrt(1 - rho^2) * eps with
    rho = sin(pi * tau / 2) (Greiner's relation for a Gaussian copula) and
    r the proxy rank."""
    device = proxy_scores.device
    n = proxy_scores.numel()
    rho = math.sin(math.pi * tau / 2.0)
    order = torch.argsort(proxy_scores.double(), descending=True, stable=True)
    ranks = torch.empty(n, dtype=torch.float64, device=device)
    ranks[order] = torch.arange(1, n + 1, dtype=torch.float64, device=device)
    u = (n - ranks + 0.5) / n
    z = torch.special.ndtri(u)
    g = _gen(_chunk_seed(seed, -4), device)
    eps = torch.randn(n, generator=g, device=device, dtype=torch.float64)
    key = rho * z + math.sqrt(max(0.0, 1.0 - rho * rho)) * eps
    return torch.argsort(key, descending=True, stable=True)


def kendall_tau_sample(a: np.ndarray, b: np.ndarray, pairs: int, seed: int) -> float:
    """Kendall tau between two complete rankings (arrays of ids in rank order)
    estimated on random item pairs."""
    n = len(a)
    ra = np.empty(n, np.int64)
    rb = np.empty(n, np.int64)
    ra[np.asarray(a)] = np.arange(n)
    rb[np.asarray(b)] = np.arange(n)
    rng = np.random.default_rng(seed)
    i = rng.integers(0, n, pairs)
    j = rng.integers(0, n, pairs)
    keep = i != j
    s = np.sign(ra[i[keep]] - ra[j[keep]]) * np.sign(rb[i[keep]] - rb[j[keep]])
    return float(s.mean())


def controlled_streams(n: int, relation: str, seed: int):
    """Two complete rankings of n items for the controlled-stream study.
    relation: 'correlated' (second = first permuted within 32-item blocks),
    'partial' (500 random items of the first list's top 1000 plus the 500
    items ranked just below it form the second list's top 1000 in random
    order; the rest follow in the first list's order),
    'independent', 'reversed', 'tied' (equal scores: both lists in id order)."""
    rng = np.random.default_rng(seed)
    if relation == "tied":
        ids = np.arange(n, dtype=np.int64)
        return ids, ids.copy()
    first = rng.permutation(n).astype(np.int64)
    if relation == "correlated":
        second = first.copy()
        for b in range(0, n, 32):
            second[b:b + 32] = rng.permutation(second[b:b + 32])
    elif relation == "partial":
        top = min(1000, n)
        half = top // 2
        inside = rng.choice(first[:top], half, replace=False)
        outside = first[top:top + (top - half)]   # the first list's next 500 items
        head = rng.permutation(np.concatenate([inside, outside]))
        used = np.zeros(n, bool)
        used[head] = True
        rest = first[~used[first]]          # the remaining items keep the first order
        second = np.concatenate([head, rest]).astype(np.int64)
    elif relation == "independent":
        second = rng.permutation(n).astype(np.int64)
    elif relation == "reversed":
        second = first[::-1].copy()
    else:
        raise ValueError(relation)
    return first, second


# --------------------------------------------------------------------------
# sparse (BM25 impact) postings
# --------------------------------------------------------------------------

def _zipf_cdf(n_terms: int, exponent: float, skip: int, device) -> torch.Tensor:
    r = torch.arange(1, n_terms + 1, dtype=torch.float64, device=device) + skip
    w = r.pow(-exponent)
    c = torch.cumsum(w, 0)
    return c / c[-1]


def bm25_postings(n_items: int, n_terms: int, mean_tokens: float, seed: int, device="cpu",
                  exponent: float = 1.0, skip: int = 100, k1: float = 0.9, b: float = 0.4,
                  topic_of=None, topic_terms: int = 0, topic_share: float = 0.0):
    """Term-major postings (term_off int64 [n_terms + 1], docs int32, imps
    float32) of a synthetic corpus with BM25 impacts.

    Each item draws Poisson(mean_tokens) tokens; each token is a term drawn
    from a Zipf law over ranks skip+1 .. skip+n_terms (the first `skip`
    ranks play the removed stopwords).  Repeated draws of a term give its
    term frequency tf.  The impact of term t on item x is the BM25 weight
    idf_t * tf (k1 + 1) / (tf + k1 (1 - b + b dl_x / avgdl)) with
    idf_t = ln(1 + (N - df_t + 0.5) / (df_t + 0.5)), computed in float64 and
    stored as float32.  Postings of a term are in ascending item id.

    Topics (optional): with topic_of[x] the topic of item x (e.g. its mixture
    component), each token is, with probability topic_share, a uniform draw
    from the item's own block of topic_terms terms, numbered after the
    n_terms background terms (the vocabulary then has n_terms +
    n_topics * topic_terms terms, n_topics = max(topic_of) + 1)."""
    cdf = _zipf_cdf(n_terms, exponent, skip, device)
    n_topics = 0
    if topic_of is not None and topic_terms > 0:
        topic_of = topic_of.to(device=device, dtype=torch.int64)
        n_topics = int(topic_of.max().item()) + 1
    vocab = n_terms + n_topics * topic_terms
    g = _gen(_chunk_seed(seed, -11), device)
    dl = torch.poisson(torch.full((n_items,), float(mean_tokens), dtype=torch.float64,
                                  device=device), generator=g).to(torch.int64)
    keys = []
    step = 1 << 16
    for c0 in range(0, n_items, step):
        c1 = min(n_items, c0 + step)
        lens = dl[c0:c1]
        total = int(lens.sum().item())
        if total == 0:
            continue
        gc = _gen(_chunk_seed(seed, c0 // step), device)
        u = torch.rand(total, generator=gc, dtype=torch.float64, device=device)
        terms = torch.searchsorted(cdf, u).clamp_max(n_terms - 1)
        docs = torch.repeat_interleave(torch.arange(c0, c1, device=device), lens)
        if n_topics:
            pick = torch.rand(total, generator=gc, device=device) < topic_share
            j = torch.randint(0, topic_terms, (total,), generator=gc, device=device)
            topical = n_terms + topic_of[docs] * topic_terms + j
            terms = torch.where(pick, topical, terms)
        keys.append(terms * n_items + docs)
    if keys:
        key = torch.sort(torch.cat(keys)).values
        uniq, tf = torch.unique_consecutive(key, return_counts=True)
    else:
        uniq = torch.empty(0, dtype=torch.int64, device=device)
        tf = torch.empty(0, dtype=torch.int64, device=device)
    term = uniq // n_items
    docs = (uniq % n_items).to(torch.int32)
    df = torch.bincount(term, minlength=vocab)
    term_off = torch.zeros(vocab + 1, dtype=torch.int64, device=device)
    term_off[1:] = torch.cumsum(df, 0)
    dlf = dl.to(torch.float64)
    avgdl = float(dlf.mean().item()) if n_items else 1.0
    avgdl = max(avgdl, 1e-9)
    idf = torch.log1p((n_items - df.to(torch.float64) + 0.5) / (df.to(torch.float64) + 0.5))
    tff = tf.to(torch.float64)
    norm = k1 * (1.0 - b + b * dlf[docs.to(torch.int64)] / avgdl)
    imps = (idf[term] * tff * (k1 + 1.0) / (tff + norm)).to(torch.float32)
    return term_off, docs, imps


def sparse_queries(nq: int, term_off: torch.Tensor, seed: int, mean_terms: float = 5.0,
                   min_df: int = 1):
    """nq queries of 1 + Poisson(mean_terms - 1) distinct terms (capped by
    the vocabulary), drawn with probability proportional to the document
    frequency among terms with at least min_df postings, each of weight 1
    (a query term counted once).  Returns a list of (terms int32, weights
    float32) numpy pairs; terms keep the order they were drawn in."""
    off = term_off.detach().cpu().numpy().astype(np.int64)
    df = np.diff(off)
    ok = np.flatnonzero(df >= min_df)
    rng = np.random.default_rng(int(seed) & ((1 << 63) - 1))
    p = df[ok].astype(np.float64)
    p /= p.sum()
    out = []
    for _ in range(nq):
        k = min(ok.size, 1 + int(rng.poisson(max(mean_terms - 1.0, 0.0))))
        t = rng.choice(ok, size=k, replace=False, p=p).astype(np.int32)
        out.append((t, np.ones(k, np.float32)))
    return out


def topical_queries(query_topics, term_off: torch.Tensor, n_terms: int, topic_terms: int,
                    seed: int, mean_topic: float = 2.0, mean_background: float = 2.0,
                    min_df: int = 2):
    """Sparse queries that match the topical corpus of bm25_postings: query i
    takes 1 + Poisson(mean_topic - 1) distinct terms of its topic's block
    (those with postings) and Poisson(mean_background) distinct background
    terms drawn in proportion to their document frequency, all of weight 1,
    topic terms first.  Returns a list of (terms int32, weights float32)."""
    off = term_off.detach().cpu().numpy().astype(np.int64)
    df = np.diff(off)
    bg = np.flatnonzero(df[:n_terms] >= min_df)
    p = df[bg].astype(np.float64)
    p /= p.sum()
    rng = np.random.default_rng(int(seed) & ((1 << 63) - 1))
    out = []
    for c in np.asarray(query_topics.detach().cpu() if hasattr(query_topics, "detach")
                        else query_topics).tolist():
        block = n_terms + int(c) * topic_terms + np.arange(topic_terms)
        block = block[df[block] > 0]
        kt = min(block.size, 1 + int(rng.poisson(max(mean_topic - 1.0, 0.0))))
        kb = min(bg.size, int(rng.poisson(mean_background)))
        t = np.concatenate([rng.choice(block, size=kt, replace=False),
                            rng.choice(bg, size=kb, replace=False, p=p)]).astype(np.int32)
        out.append((t, np.ones(t.size, np.float32)))
    return out
