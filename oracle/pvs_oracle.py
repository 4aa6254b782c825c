"""PVS oracle: quantization, intervals, authoritative scores, dense ranking.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Paper: arXiv 2608.07152.
  * Sec. 2.1   complete ranked list pi_i: items ordered by score, ties broken
               by the identifier order (here: ascending id).
  * Sec. 2.3.1 PVS per-vector Int8 quantization, centre score
               c = s_q s_v <z_q, z_v>, residual bound
               E = ||e_q|| ||v|| + ||q_hat|| ||e_v||.
  * App. A.1   guard G = (|c| + E + ||q||_up ||v||_up) gamma_m,
               gamma_m >= a_m / (1 - a_m), a_m = (8m + 64) eps_f32, outward
               rounded endpoints, failure on non-finite input.

Scalar-quantization intervals (the rank-generator ablation of Sec. 3.5 and
4.4; the paper gives no construction; reading): one scale s = RN(max |v_j| /
127) over the whole corpus in place of every s_v, with the same codes,
residual bounds and intervals (``global_scale``, ``quantize_global``).

Authoritative float32 score (the paper fixes no summation order; reading):
the correctly rounded (to nearest, ties to even) float32 value of the exact
real inner product sum_j q_j v_j.  It lies within every interval the guard
admits, and it does not depend on any summation order.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

from . import _clib

F32_EPS = 2.0 ** -23


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(__import__("ctypes").c_void_p)


# --------------------------------------------------------------------------
# Sec. 2.3.1: per-vector Int8 quantization (bound arithmetic in pvs_ref.c)
# --------------------------------------------------------------------------

@dataclass
class Quantized:
    z: np.ndarray       # int8 [n, ldz]
    s: np.ndarray       # float32 [n]   per-vector scale s_v
    vnorm: np.ndarray   # float32 [n]   ||v||_2 rounded up
    enorm: np.ndarray   # float32 [n]   ||v - s_v z_v||_2 rounded up
    status: int         # 0 ok, 1 non-finite input, 2 norm overflow


def quantize(V: np.ndarray, ldz: int | None = None) -> Quantized:
    """Quantize the rows of a float32 matrix (Sec. 2.3.1)."""
    V = np.ascontiguousarray(V, dtype=np.float32)
    n, m = V.shape
    ldz = m if ldz is None else ldz
    Z = np.zeros((n, ldz), dtype=np.int8)
    s = np.zeros(n, np.float32)
    vn = np.zeros(n, np.float32)
    en = np.zeros(n, np.float32)
    scratch = np.zeros(max(m, 1), np.float64)
    st = _clib.lib().orc_quantize(_ptr(V), n, m, _ptr(Z), ldz, _ptr(s), _ptr(vn),
                                  _ptr(en), _ptr(scratch))
    return Quantized(Z, s, vn, en, int(st))


def global_scale(V: np.ndarray) -> np.float32:
    """Scalar-quantization intervals (the ablation of Sec. 3.5 / 4.4): one
    scale RN(max |v_j| / 127) for the whole corpus (NaN for non-finite input)."""
    V = np.ascontiguousarray(V, dtype=np.float32)
    n, m = V.shape
    return np.float32(_clib.lib().orc_global_scale(_ptr(V), n, m))


def quantize_global(V: np.ndarray, s=None, ldz: int | None = None) -> Quantized:
    """Quantize every row with one scale s (default: global_scale(V)); codes,
    residuals and norm bounds as Sec. 2.3.1 with s in place of s_v.  Status 3
    marks a row whose codes would leave [-127, 127]."""
    V = np.ascontiguousarray(V, dtype=np.float32)
    n, m = V.shape
    ldz = m if ldz is None else ldz
    s = global_scale(V) if s is None else np.float32(s)
    Z = np.zeros((n, ldz), dtype=np.int8)
    sv = np.zeros(n, np.float32)
    vn = np.zeros(n, np.float32)
    en = np.zeros(n, np.float32)
    scratch = np.zeros(max(m, 1), np.float64)
    st = _clib.lib().orc_quantize_fixed(_ptr(V), n, m, _ptr(Z), ldz, float(s), _ptr(sv),
                                        _ptr(vn), _ptr(en), _ptr(scratch))
    return Quantized(Z, sv, vn, en, int(st))


def norm_bound(x) -> np.float32:
    """Upward-rounded ||x||_2 of binary64 values (reading in pvs_ref.c)."""
    x = np.ascontiguousarray(np.asarray(x, dtype=np.float64))
    return np.float32(_clib.lib().orc_norm_bound(_ptr(x), x.size))


def gamma(m: int) -> np.float32:
    """gamma_m = RU(a_m / RD(1 - a_m)), a_m = (8m + 64) 2^-23 (App. A.1)."""
    return np.float32(_clib.lib().orc_gamma(int(m)))


@dataclass
class EncodedQuery:
    z: np.ndarray       # int8 [m]
    s: np.float32       # s_q
    qnorm: np.float32   # ||q||_2 up
    qhat: np.float32    # ||s_q z_q||_2 up
    enorm: np.float32   # ||q - s_q z_q||_2 up
    gamma: np.float32   # gamma_m
    status: int


def encode_query(q: np.ndarray) -> EncodedQuery:
    """Encode the query exactly as a corpus vector (Sec. 2.3.1)."""
    q = np.ascontiguousarray(q, dtype=np.float32).reshape(1, -1)
    m = q.shape[1]
    Q = quantize(q)
    scratch = np.zeros(max(m, 1), np.float64)
    zq = np.ascontiguousarray(Q.z[0])
    qhat = np.float32(_clib.lib().orc_qhat_norm(_ptr(zq), float(Q.s[0]), m, _ptr(scratch)))
    return EncodedQuery(zq, Q.s[0], Q.vnorm[0], qhat, Q.enorm[0], gamma(m), Q.status)


def intervals(qe: EncodedQuery, Q: Quantized, m: int):
    """Score intervals [lo, hi] of every corpus vector (Sec. 2.3.1, App. A.1)."""
    n, ldz = Q.z.shape
    lo = np.zeros(n, np.float32)
    hi = np.zeros(n, np.float32)
    _clib.lib().orc_intervals(_ptr(qe.z), float(qe.s), float(qe.qnorm), float(qe.qhat),
                              float(qe.enorm), float(qe.gamma), _ptr(Q.z), n, m, ldz,
                              _ptr(Q.s), _ptr(Q.vnorm), _ptr(Q.enorm), _ptr(lo), _ptr(hi))
    return lo, hi


def interval_one(dot: int, qe: EncodedQuery, s: float, vnorm: float, enorm: float):
    import ctypes
    lo = ctypes.c_float()
    hi = ctypes.c_float()
    _clib.lib().orc_interval_one(int(dot), float(qe.s), float(qe.qnorm), float(qe.qhat),
                                 float(qe.enorm), float(qe.gamma), float(s), float(vnorm),
                                 float(enorm), ctypes.byref(lo), ctypes.byref(hi))
    return np.float32(lo.value), np.float32(hi.value)


# --------------------------------------------------------------------------
# Authoritative float32 score: RN_f32 of the exact inner product
# --------------------------------------------------------------------------

def round_real_to_f32(s64: float, residual_sign: int) -> np.float32:
    """Round a real x to float32 (nearest, ties to even), given s64 = RN_f64(x)
    and the sign of x - s64.

    RN_f32(x) == RN_f32(s64) unless s64 is exactly halfway between two
    adjacent float32 values (then x's side of s64 decides), because every
    such halfway point is itself a binary64 number.  A result that rounds to
    zero is returned as +0: the score orders by value and -0 == +0, so the
    sign of a zero carries nothing, and one canonical zero makes scores
    comparable bit for bit.
    """
    f = np.float32(s64)
    if f == 0:
        return np.float32(0.0)                  # a score that rounds to zero is +0
    if not np.isfinite(f) or float(f) == s64:
        return f
    g = np.nextafter(f, np.float32(math.inf) if s64 > float(f) else np.float32(-math.inf))
    mid = (float(f) + float(g)) / 2.0          # exact in binary64
    if s64 != mid or residual_sign == 0:
        return f                                # not a tie, or an exact tie
    above = residual_sign > 0
    return max(f, g) if above else min(f, g)


def exact_score_one(q: np.ndarray, v: np.ndarray) -> np.float32:
    """RN_f32(sum_j q_j v_j) computed exactly: every product of two float32
    values is exact in binary64, and math.fsum returns the correctly rounded
    binary64 sum of its (exact) inputs."""
    p = (np.asarray(q, np.float32).astype(np.float64)
         * np.asarray(v, np.float32).astype(np.float64)).tolist()
    s64 = math.fsum(p)
    r = math.fsum(p + [-s64])                  # sign of (exact sum - s64)
    sign = (r > 0) - (r < 0)
    return round_real_to_f32(s64, sign)


def exact_scores(q: np.ndarray, V: np.ndarray, block: int = 1 << 16) -> np.ndarray:
    """Authoritative scores of every row of V.

    A binary64 matrix product (a library step) gives S with
    |S - exact| <= (m u) * sum_j |p_j|, u = 2^-53; rows whose whole error
    interval rounds to one float32 take that value, the others fall back to
    ``exact_score_one``.
    """
    q = np.asarray(q, np.float32)
    V = np.asarray(V, np.float32)
    n, m = V.shape
    q64 = q.astype(np.float64)
    aq = np.abs(q64)
    out = np.empty(n, np.float32)
    factor = 4.0 * max(m, 1) * 2.0 ** -53
    for b0 in range(0, n, block):
        B = V[b0:b0 + block].astype(np.float64)
        S = B @ q64
        A = np.abs(B) @ aq
        beta = A * factor
        lo = (S - beta).astype(np.float32)
        hi = (S + beta).astype(np.float32)
        ok = lo == hi
        out[b0:b0 + block][ok] = lo[ok]
        for i in np.nonzero(~ok)[0]:
            out[b0 + i] = exact_score_one(q, V[b0 + i])
    out[out == 0] = np.float32(0.0)             # canonical +0, as round_real_to_f32
    return out


def dense_ranking(q: np.ndarray, V: np.ndarray, visible: np.ndarray | None = None):
    """Complete dense ranked list (Sec. 2.1): visible ids ordered by
    (authoritative score descending, id ascending).  Returns (ids, scores)."""
    s = exact_scores(q, V)
    ids = np.arange(V.shape[0], dtype=np.int64)
    if visible is not None:
        ids = ids[np.asarray(visible, bool)]
        s = s[ids]
    order = np.lexsort((ids, -s.astype(np.float64)))
    return ids[order], s[order]


def ranking_of_scores(ids: np.ndarray, scores: np.ndarray):
    """Order (id, score) pairs by (score descending, id ascending)."""
    ids = np.asarray(ids, np.int64)
    scores = np.asarray(scores, np.float32)
    order = np.lexsort((ids, -scores.astype(np.float64)))
    return ids[order], scores[order]
