"""GB300-native PVS resumable exact dense ranking and EAHR fusion.

Method: arXiv 2608.07152 (Exact Adaptive Hybrid Retrieval).  Every step of
the ranking path runs in the CUDA kernels of ``libpvs.so`` behind the C ABI of
``include/pvs.h``; this module only marshals arguments.  The functions keep
the C names.  A negative status raises :class:`PvsError`; ``PVS_EXHAUSTED``
is returned, not raised.

Host inputs are numpy arrays; device inputs are CUDA ``torch`` tensors
(torch's current stream is synchronised before their pointers are handed to
the library, which runs on its own stream).
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from ._build import LIB as _LIB_PATH

PVS_OK = 0
PVS_EXHAUSTED = 1
PVS_ERR_INVALID = -1
PVS_ERR_NONFINITE = -2
PVS_ERR_OVERFLOW = -3
PVS_ERR_INTERVAL = -4
PVS_ERR_CUDA = -5
PVS_ERR_OOM = -6
PVS_ERR_TIMEOUT = -7
PVS_ERR_FAILED = -8

PVS_QUANT_PER_VECTOR = 0
PVS_QUANT_GLOBAL = 1
PVS_GEN_INTERVALS = 0
PVS_GEN_FULL_SCAN = 1

PVS_CHILD_DENSE = 0
PVS_CHILD_SPARSE = 1
PVS_CHILD_MERGE = 2

EAHR_RANK_SCALED = 0
EAHR_NUMERATOR = 1
EAHR_POLICY_GEOMETRIC = 0
EAHR_POLICY_EQUAL_DEPTH = 1
EAHR_POLICY_FROZEN = 2
EAHR_POLICY_ADAPTIVE = 3


class PvsError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {pvs_status_string(status)} ({status})")


class pvs_stats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "visible", "emitted", "refined", "exact_fallbacks", "interval_passes",
        "horizon_builds", "pulls", "candidates", "code_bytes")] + [
        ("state", ctypes.c_int32), ("reserved", ctypes.c_int32),
        ("interval_ms", ctypes.c_double), ("batch_passes", ctypes.c_int64),
        ("batch_ms", ctypes.c_double)]


class eahr_params(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("k", ctypes.c_int32), ("form", ctypes.c_int32),
                ("policy", ctypes.c_int32), ("step", ctypes.c_int32),
                ("w_num", ctypes.c_int32 * 2), ("w_den", ctypes.c_int32 * 2)]


class eahr_stats(ctypes.Structure):
    _fields_ = [("depth", ctypes.c_int64 * 2), ("length", ctypes.c_int64 * 2),
                ("exhausted", ctypes.c_int32 * 2), ("pulls", ctypes.c_int32 * 2),
                ("checks", ctypes.c_int32), ("complete", ctypes.c_int32)]


class pbm_stats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "items", "emitted", "ranges", "ranges_expanded", "postings_visited", "items_scored",
        "pulls", "rounds", "pulls_from_window")] + [("state", ctypes.c_int32),
                                                    ("reserved", ctypes.c_int32)]


class pvs_merge_child(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("cursor", ctypes.c_void_p), ("id_offset", ctypes.c_int64)]


class pvs_merge_stats_t(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "emitted", "read", "duplicates", "child_pulls", "id_space", "length")] + [
        ("state", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class pvs_executor_stats_t(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in ("requests", "failed", "pages", "ranks")] + [
        ("workers", ctypes.c_int32), ("group", ctypes.c_int32),
        ("interval_passes", ctypes.c_int64), ("interval_ms", ctypes.c_double),
        ("refined", ctypes.c_int64)]


def _load() -> ctypes.CDLL:
    if not os.path.exists(_LIB_PATH):
        raise ImportError(
            f"libpvs.so not found at {_LIB_PATH}; build it with "
            "`python -c 'import __graft_entry__ as g; g.build()'` (needs nvcc)")
    L = ctypes.CDLL(_LIB_PATH)
    P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    pp = ctypes.POINTER(ctypes.c_void_p)
    sig = {
        "pvs_build": (i32, [P, i64, i32, i32, P, pp]),
        "pvs_build_ex": (i32, [P, i64, i32, i32, P, i32, pp]),
        "pvs_cursor_set_generator": (i32, [P, i32]),
        "pvs_append": (i32, [P, P, i64, i32]),
        "pvs_tombstone": (i32, [P, P, i64]),
        "pvs_index_size": (i64, [P]),
        "pvs_index_live": (i64, [P]),
        "pvs_index_dim": (i32, [P]),
        "pvs_index_export": (i32, [P, i64, i64, P, P, P, P]),
        "pvs_index_free": (None, [P]),
        "pvs_snapshot_create": (i32, [P, pp]),
        "pvs_snapshot_visible": (i64, [P]),
        "pvs_snapshot_free": (None, [P]),
        "pvs_cursor_open": (i32, [P, P, P, i32, pp]),
        "pvs_cursor_open_batch": (i32, [P, P, P, i32, i32, i32, P, pp]),
        "pvs_next": (i32, [P, i32, P, P, P]),
        "pvs_next_device": (i32, [P, i32, P, P, P]),
        "pvs_cursor_sync": (i32, [P]),
        "pvs_cursor_set_stream": (i32, [P, P]),
        "pvs_next_batch": (i32, [P, i32, i32, i32, P, P, P]),
        "pvs_batch_bounds": (i32, [P, P, P, i32, i32, P, P]),
        "pvs_cursor_stats": (i32, [P, ctypes.POINTER(pvs_stats)]),
        "pvs_cursor_bounds": (i32, [P, i64, i64, P, P]),
        "pvs_cursor_score_ids": (i32, [P, P, i32, P]),
        "pvs_cursor_close": (None, [P]),
        "pvs_cursor_sync_batch": (i32, [P, i32, P]),
        "pvs_cursor_stats_batch": (i32, [P, i32, P]),
        "pvs_cursor_close_batch": (None, [P, i32]),
        "pvs_status_string": (ctypes.c_char_p, [i32]),
        "pvs_launch_count": (i64, []),
        "pvs_rank_exact_noalloc": (i32, [P, P, i32, i32, i32, P, P, P]),
        "pvs_index_import": (i32, [P, P, P, P, P, i64, i32, P, pp]),
        "pvs_cursor_open_group": (i32, [P, P, P, i32, i32, P, P, P]),
        "pvs_cursor_set_readahead": (i32, [P, i32]),
        "pvs_index_set_wait_limit": (i32, [P, i64]),
        "eahr_topk": (i32, [P, P, i64, ctypes.POINTER(eahr_params), P, P, P,
                            ctypes.POINTER(eahr_stats)]),
        "eahr_topk_lists": (i32, [P, i64, P, i64, ctypes.POINTER(eahr_params), P, P, P,
                                  ctypes.POINTER(eahr_stats)]),
        "pbm_build": (i32, [P, i32, P, P, i64, i64, i32, i32, P, pp]),
        "pbm_index_items": (i64, [P]),
        "pbm_index_ranges": (i64, [P]),
        "pbm_index_free": (None, [P]),
        "pbm_cursor_open": (i32, [P, P, P, i32, pp]),
        "pbm_cursor_open_snapshot": (i32, [P, P, P, P, i32, pp]),
        "pbm_cursor_open_stream": (i32, [P, P, P, P, i32, P, pp]),
        "pbm_next": (i32, [P, i32, P, P, P]),
        "pbm_cursor_range_bounds": (i32, [P, i64, i64, P]),
        "pbm_cursor_stats": (i32, [P, ctypes.POINTER(pbm_stats)]),
        "pbm_cursor_close": (None, [P]),
        "eahr_topk_pbm": (i32, [P, P, ctypes.POINTER(eahr_params), P, P, P,
                                ctypes.POINTER(eahr_stats)]),
        "pvs_merge_open": (i32, [P, i32, pp]),
        "pvs_merge_next": (i32, [P, i32, P, P, P]),
        "pvs_merge_stats_get": (i32, [P, ctypes.POINTER(pvs_merge_stats_t)]),
        "pvs_merge_close": (None, [P]),
        "eahr_topk_merge": (i32, [P, P, ctypes.POINTER(eahr_params), P, P, P,
                                  ctypes.POINTER(eahr_stats)]),
        "pvs_executor_create": (i32, [P, i32, pp]),
        "pvs_executor_run": (i32, [P, P, P, i32, i32, i32, P, P, P, P]),
        "pvs_executor_run_ex": (i32, [P, P, P, i32, i32, i32, i32, P, P, P, P]),
        "pvs_executor_set_group": (i32, [P, i32]),
        "pvs_executor_stats_get": (i32, [P, ctypes.POINTER(pvs_executor_stats_t)]),
        "pvs_executor_destroy": (None, [P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    return L


_lib = _load()
lib_path = _LIB_PATH
EXPORTED = ("pvs_build", "pvs_build_ex", "pvs_cursor_set_generator", "pvs_append", "pvs_tombstone", "pvs_index_size", "pvs_index_live",
            "pvs_index_dim", "pvs_index_export", "pvs_index_free", "pvs_snapshot_create",
            "pvs_snapshot_visible", "pvs_snapshot_free", "pvs_cursor_open",
            "pvs_cursor_open_batch", "pvs_next", "pvs_next_device", "pvs_cursor_sync",
            "pvs_cursor_set_stream", "pvs_next_batch", "pvs_batch_bounds",
            "pvs_cursor_stats", "pvs_cursor_bounds", "pvs_cursor_score_ids", "pvs_cursor_close",
            "pvs_cursor_sync_batch", "pvs_cursor_stats_batch", "pvs_cursor_close_batch",
            "pvs_status_string", "pvs_launch_count", "pvs_rank_exact_noalloc",
            "pvs_index_import", "pvs_index_set_wait_limit", "pvs_cursor_open_group",
            "pvs_cursor_set_readahead", "eahr_topk",
            "eahr_topk_lists", "pbm_build", "pbm_index_items", "pbm_index_ranges",
            "pbm_index_free", "pbm_cursor_open", "pbm_cursor_open_snapshot", "pbm_cursor_open_stream", "pbm_next", "pbm_cursor_range_bounds",
            "pbm_cursor_stats", "pbm_cursor_close", "eahr_topk_pbm", "pvs_merge_open",
            "pvs_merge_next", "pvs_merge_stats_get", "pvs_merge_close", "eahr_topk_merge",
            "pvs_executor_create", "pvs_executor_run", "pvs_executor_run_ex",
            "pvs_executor_set_group", "pvs_executor_stats_get",
            "pvs_executor_destroy")


def pvs_status_string(status: int) -> str:
    return _lib.pvs_status_string(int(status)).decode()


def pvs_launch_count() -> int:
    return int(_lib.pvs_launch_count())


def _check(status: int, where: str) -> int:
    if status < 0:
        raise PvsError(status, where)
    return status


def _vec_arg(x, dim: int | None = None):
    """(pointer, rows, dim, on_device, keepalive) for numpy or torch input."""
    try:
        import torch
    except ImportError:  # pragma: no cover
        torch = None
    if torch is not None and isinstance(x, torch.Tensor):
        if x.dtype != torch.float32:
            raise TypeError("vectors must be float32")
        x = x.contiguous()
        on_dev = 1 if x.is_cuda else 0
        if x.is_cuda:
            torch.cuda.current_stream(x.device).synchronize()
        shape = tuple(x.shape)
        return ctypes.c_void_p(x.data_ptr()), shape, on_dev, x
    a = np.ascontiguousarray(x, dtype=np.float32)
    return ctypes.c_void_p(a.ctypes.data), a.shape, 0, a


def pvs_build(vecs, stream=None, quantization: int = PVS_QUANT_PER_VECTOR):
    """Build an index over the rows of a 2-D float32 array / tensor
    (quantization: PVS_QUANT_PER_VECTOR, or PVS_QUANT_GLOBAL for the
    scalar-quantization-interval index of the ablation, via pvs_build_ex)."""
    ptr, shape, on_dev, keep = _vec_arg(vecs)
    n, dim = (shape[0], shape[1]) if len(shape) == 2 else (0, shape[-1])
    out = ctypes.c_void_p()
    st = ctypes.c_void_p(stream) if stream else None
    if quantization == PVS_QUANT_PER_VECTOR:
        _check(_lib.pvs_build(ptr, n, dim, on_dev, st, ctypes.byref(out)), "pvs_build")
    else:
        _check(_lib.pvs_build_ex(ptr, n, dim, on_dev, st, int(quantization), ctypes.byref(out)),
               "pvs_build_ex")
    return out


def pvs_build_ex(vecs, quantization: int, stream=None):
    return pvs_build(vecs, stream=stream, quantization=quantization)


def pvs_append(index, vecs) -> None:
    ptr, shape, on_dev, keep = _vec_arg(vecs)
    _check(_lib.pvs_append(index, ptr, shape[0], on_dev), "pvs_append")


def pvs_tombstone(index, ids) -> None:
    a = np.ascontiguousarray(ids, dtype=np.int64)
    _check(_lib.pvs_tombstone(index, a.ctypes.data, a.size), "pvs_tombstone")


def pvs_index_size(index) -> int:
    return int(_lib.pvs_index_size(index))


def pvs_index_live(index) -> int:
    return int(_lib.pvs_index_live(index))


def pvs_index_dim(index) -> int:
    return int(_lib.pvs_index_dim(index))


def pvs_index_export(index, first: int, count: int):
    dim = pvs_index_dim(index)
    codes = np.zeros((count, dim), np.int8)
    scale = np.zeros(count, np.float32)
    vnorm = np.zeros(count, np.float32)
    enorm = np.zeros(count, np.float32)
    _check(_lib.pvs_index_export(index, first, count, codes.ctypes.data, scale.ctypes.data,
                                 vnorm.ctypes.data, enorm.ctypes.data), "pvs_index_export")
    return codes, scale, vnorm, enorm


def pvs_index_import(vecs, codes, scale, vnorm, enorm, stream=None):
    """Index from saved parameters (host arrays): vecs float32 [n, dim],
    codes int8 [n, dim], scale / vnorm / enorm float32 [n].  Nothing is
    re-quantized; a parameter that does not bound its row's score fails the
    pull that scores the row (App. A.1 failure rule)."""
    v = np.ascontiguousarray(vecs, dtype=np.float32)
    z = np.ascontiguousarray(codes, dtype=np.int8)
    s, vn, en = (np.ascontiguousarray(a, dtype=np.float32) for a in (scale, vnorm, enorm))
    n, dim = v.shape
    if z.shape != (n, dim) or s.shape != (n,) or vn.shape != (n,) or en.shape != (n,):
        raise ValueError("codes [n, dim] and scale / vnorm / enorm [n] must match vecs")
    out = ctypes.c_void_p()
    _check(_lib.pvs_index_import(v.ctypes.data, z.ctypes.data, s.ctypes.data, vn.ctypes.data,
                                 en.ctypes.data, n, dim, stream, ctypes.byref(out)),
           "pvs_index_import")
    return out


def pvs_index_set_wait_limit(index, ns: int) -> None:
    _check(_lib.pvs_index_set_wait_limit(index, int(ns)), "pvs_index_set_wait_limit")


def pvs_index_free(index) -> None:
    _lib.pvs_index_free(index)


def pvs_snapshot_create(index):
    out = ctypes.c_void_p()
    _check(_lib.pvs_snapshot_create(index, ctypes.byref(out)), "pvs_snapshot_create")
    return out


def pvs_snapshot_visible(snap) -> int:
    return int(_lib.pvs_snapshot_visible(snap))


def pvs_snapshot_free(snap) -> None:
    _lib.pvs_snapshot_free(snap)


def pvs_cursor_open(index, query, snap=None):
    ptr, shape, on_dev, keep = _vec_arg(query)
    out = ctypes.c_void_p()
    _check(_lib.pvs_cursor_open(index, snap, ptr, on_dev, ctypes.byref(out)), "pvs_cursor_open")
    return out


PVS_GROUP_MAX = 16


def pvs_cursor_open_group(index, queries, snap=None, pass_stream=None, cursor_streams=None):
    """Open one cursor per query row (at most PVS_GROUP_MAX) whose bounds come
    from one grouped pass over the codes -> list of cursors.  pass_stream and
    the entries of cursor_streams: torch.cuda.Stream or raw cudaStream_t
    (None: the index's stream / the pass stream)."""
    ptr, shape, on_dev, keep = _vec_arg(queries)
    nq = shape[0] if len(shape) == 2 else 1
    arr = (ctypes.c_void_p * max(nq, 1))()
    ps = getattr(pass_stream, "cuda_stream", pass_stream)
    streams = None
    if cursor_streams is not None:
        if len(cursor_streams) != nq:
            raise ValueError("one stream per query")
        streams = (ctypes.c_void_p * nq)(*[getattr(s, "cuda_stream", s) for s in cursor_streams])
    _check(_lib.pvs_cursor_open_group(index, snap, ptr, nq, on_dev,
                                      ctypes.c_void_p(ps) if ps else None,
                                      ctypes.cast(streams, ctypes.c_void_p) if streams else None,
                                      ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))),
           "pvs_cursor_open_group")
    return [ctypes.c_void_p(arr[i]) for i in range(nq)]


class CursorBatch(tuple):
    """The cursors of a batched open (immutable), with the C array of their
    handles built once for the batch calls."""

    def __new__(cls, handles):
        self = super().__new__(cls, [ctypes.c_void_p(h) for h in handles])
        self._arr = (ctypes.c_void_p * max(len(handles), 1))(*handles)
        return self


def pvs_cursor_open_batch(index, queries, horizon: int, snap=None, stream=None):
    """Open one cursor per query row -> CursorBatch.  stream: a
    torch.cuda.Stream or raw cudaStream_t for the open and the cursors (None:
    the index's stream)."""
    ptr, shape, on_dev, keep = _vec_arg(queries)
    nq = shape[0]
    arr = (ctypes.c_void_p * max(nq, 1))()
    handle = getattr(stream, "cuda_stream", stream)
    _check(_lib.pvs_cursor_open_batch(index, snap, ptr, nq, on_dev, int(horizon),
                                      ctypes.c_void_p(handle) if handle else None,
                                      ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))),
           "pvs_cursor_open_batch")
    return CursorBatch([arr[i] for i in range(nq)])


def pvs_next(cursor, n: int):
    """Next n exact ranks -> (ids int64[n_out], scores float32[n_out], status)."""
    ids = np.zeros(max(n, 1), np.int64)
    sc = np.zeros(max(n, 1), np.float32)
    got = ctypes.c_int32(0)
    st = _check(_lib.pvs_next(cursor, int(n), ids.ctypes.data, sc.ctypes.data,
                              ctypes.byref(got)), "pvs_next")
    return ids[:got.value], sc[:got.value], st


def pvs_next_device(cursor, n: int, ids, scores):
    """Enqueue the next n ranks into CUDA tensors ids (int64) / scores
    (float32); returns (n_out, status)."""
    got = ctypes.c_int32(0)
    st = _check(_lib.pvs_next_device(cursor, int(n), ctypes.c_void_p(ids.data_ptr()),
                                     ctypes.c_void_p(scores.data_ptr()), ctypes.byref(got)),
                "pvs_next_device")
    return got.value, st


def _cursor_array(cursors):
    if isinstance(cursors, CursorBatch):
        return cursors._arr
    return (ctypes.c_void_p * max(len(cursors), 1))(
        *[c.value if isinstance(c, ctypes.c_void_p) else c for c in cursors])


def pvs_next_batch(cursors, n: int, ids=None, scores=None):
    """Next n ranks of every cursor.  Without ids/scores: host outputs, returns
    (ids int64[nc, n], scores float32[nc, n], n_out int32[nc]); with CUDA
    tensors ids / scores of shape [nc, >= n] (row stride n): queued, returns
    n_out."""
    nc = len(cursors)
    arr = _cursor_array(cursors)
    n_out = np.zeros(max(nc, 1), np.int32)
    if ids is None:
        h_ids = np.zeros((max(nc, 1), max(n, 1)), np.int64)
        h_sc = np.zeros((max(nc, 1), max(n, 1)), np.float32)
        _check(_lib.pvs_next_batch(arr, nc, int(n), 0, h_ids.ctypes.data, h_sc.ctypes.data,
                                   n_out.ctypes.data), "pvs_next_batch")
        return h_ids[:nc, :n], h_sc[:nc, :n], n_out[:nc]
    _check(_lib.pvs_next_batch(arr, nc, int(n), 1, ctypes.c_void_p(ids.data_ptr()),
                               ctypes.c_void_p(scores.data_ptr()), n_out.ctypes.data),
           "pvs_next_batch")
    return n_out[:nc]


def pvs_batch_bounds(index, queries, snap=None, rows=None):
    """Tensor-core intervals of every row for nq <= 256 queries ->
    (lo, hi) float32[nq, rows]; `rows` is the snapshot's row count (default:
    the index's current size, right for snap=None)."""
    ptr, shape, on_dev, keep = _vec_arg(queries)
    nq = shape[0]
    rows = int(_lib.pvs_index_size(index)) if rows is None else int(rows)
    lo = np.zeros((nq, max(rows, 1)), np.float32)
    hi = np.zeros((nq, max(rows, 1)), np.float32)
    _check(_lib.pvs_batch_bounds(index, snap, ptr, nq, on_dev, lo.ctypes.data, hi.ctypes.data),
           "pvs_batch_bounds")
    return lo[:, :rows], hi[:, :rows]


def pvs_cursor_sync(cursor) -> int:
    return _check(_lib.pvs_cursor_sync(cursor), "pvs_cursor_sync")


def pvs_cursor_set_generator(cursor, generator: int) -> None:
    """PVS_GEN_INTERVALS (default) or PVS_GEN_FULL_SCAN, before the first pull."""
    _check(_lib.pvs_cursor_set_generator(cursor, int(generator)), "pvs_cursor_set_generator")


def pvs_cursor_set_readahead(cursor, pages: int) -> None:
    _check(_lib.pvs_cursor_set_readahead(cursor, int(pages)), "pvs_cursor_set_readahead")


def pvs_cursor_set_stream(cursor, stream) -> None:
    """stream: a torch.cuda.Stream, a raw cudaStream_t handle, or None."""
    handle = getattr(stream, "cuda_stream", stream)
    _check(_lib.pvs_cursor_set_stream(cursor, ctypes.c_void_p(handle) if handle else None),
           "pvs_cursor_set_stream")


def pvs_cursor_stats(cursor) -> dict:
    s = pvs_stats()
    _check(_lib.pvs_cursor_stats(cursor, ctypes.byref(s)), "pvs_cursor_stats")
    return {name: getattr(s, name) for name, _ in pvs_stats._fields_ if name != "reserved"}


def pvs_cursor_bounds(cursor, first: int, count: int):
    lo = np.zeros(max(count, 1), np.float32)
    hi = np.zeros(max(count, 1), np.float32)
    _check(_lib.pvs_cursor_bounds(cursor, first, count, lo.ctypes.data, hi.ctypes.data),
           "pvs_cursor_bounds")
    return lo[:count], hi[:count]


def pvs_cursor_score_ids(cursor, ids):
    a = np.ascontiguousarray(ids, dtype=np.int64)
    out = np.zeros(max(a.size, 1), np.float32)
    _check(_lib.pvs_cursor_score_ids(cursor, a.ctypes.data, a.size, out.ctypes.data),
           "pvs_cursor_score_ids")
    return out[:a.size]


def pvs_cursor_close(cursor) -> None:
    _lib.pvs_cursor_close(cursor)


def pvs_cursor_sync_batch(cursors):
    """States (int32[nc]) of many cursors after one wait per stream."""
    states = np.zeros(max(len(cursors), 1), np.int32)
    _check(_lib.pvs_cursor_sync_batch(_cursor_array(cursors), len(cursors),
                                      states.ctypes.data), "pvs_cursor_sync_batch")
    return states[:len(cursors)]


def pvs_cursor_stats_batch(cursors) -> list:
    out = (pvs_stats * max(len(cursors), 1))()
    _check(_lib.pvs_cursor_stats_batch(_cursor_array(cursors), len(cursors),
                                       ctypes.cast(out, ctypes.c_void_p)),
           "pvs_cursor_stats_batch")
    return [{name: getattr(out[i], name) for name, _ in pvs_stats._fields_ if name != "reserved"}
            for i in range(len(cursors))]


def pvs_cursor_close_batch(cursors) -> None:
    _lib.pvs_cursor_close_batch(_cursor_array(cursors), len(cursors))


PVS_NOALLOC_MAX_VECTORS = 8192


def pvs_rank_exact_noalloc(query, vecs, top: int, out_ids, out_scores) -> int:
    """Allocation-free exact ranking of the rows of `vecs` (float32 [n, dim])
    against `query` (float32 [dim]) into the caller's tensors out_ids (int64,
    at least `top` entries) and out_scores (float32, at least `top` entries).
    All four are contiguous CUDA tensors on one device.  Neither this wrapper
    nor the library allocates device memory: callers whose device memory
    belongs to a pool or budget of their own pass tensors they already own.
    Runs on torch's current stream of that device and returns once the
    stream has finished the work.

    The library cannot see tensor shapes or types through raw pointers, so
    every size and type is checked here before the call."""
    import torch
    ts = (query, vecs, out_ids, out_scores)
    for t in ts:
        if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous()):
            raise TypeError("pvs_rank_exact_noalloc takes contiguous CUDA tensors")
    if any(t.device != vecs.device for t in ts):
        raise ValueError("query, vecs, out_ids and out_scores must be on one device")
    if query.dtype != torch.float32 or vecs.dtype != torch.float32:
        raise TypeError("query and vecs must be float32")
    if out_ids.dtype != torch.int64 or out_scores.dtype != torch.float32:
        raise TypeError("out_ids must be int64 and out_scores float32")
    if vecs.dim() != 2:
        raise ValueError("vecs must be a 2-D tensor [n, dim]")
    n, dim = int(vecs.shape[0]), int(vecs.shape[1])
    top = int(top)
    if query.numel() != dim:
        raise ValueError(f"query has {query.numel()} entries, vecs rows have {dim}")
    if top < 0 or top > n:
        raise ValueError(f"top = {top} outside [0, {n}]")
    if out_ids.numel() < top or out_scores.numel() < top:
        raise ValueError(f"out_ids and out_scores must hold at least top = {top} entries")
    with torch.cuda.device(vecs.device):
        stream = torch.cuda.current_stream(vecs.device).cuda_stream
        return _check(_lib.pvs_rank_exact_noalloc(
            ctypes.c_void_p(query.data_ptr()), ctypes.c_void_p(vecs.data_ptr()), n, dim, top,
            ctypes.c_void_p(out_ids.data_ptr()), ctypes.c_void_p(out_scores.data_ptr()),
            ctypes.c_void_p(stream) if stream else None), "pvs_rank_exact_noalloc")


def _params(K, k, form, policy, step, weights):
    p = eahr_params()
    p.K, p.k, p.form, p.policy, p.step = int(K), int(k), int(form), int(policy), int(step)
    for i, w in enumerate(weights):
        num, den = (w, 1) if np.isscalar(w) else w
        p.w_num[i], p.w_den[i] = int(num), int(den)
    return p


def _eahr_result(st, ids, F, got, stats):
    s = {"depth": list(stats.depth), "length": list(stats.length),
         "exhausted": list(stats.exhausted), "pulls": list(stats.pulls),
         "checks": stats.checks, "complete": stats.complete}
    return ids[:got.value], F[:got.value], s


def eahr_topk(cursor, sparse_ids, K: int = 20, k: int = 60, form: int = EAHR_NUMERATOR,
              policy: int = EAHR_POLICY_GEOMETRIC, step: int = 0, weights=(1, 1)):
    """Ordered Top-K of complete-list weighted RRF (dense cursor + host sparse
    ranking) -> (ids int64[q_K], F float64[q_K], stats)."""
    sp = np.ascontiguousarray(sparse_ids, dtype=np.int64)
    p = _params(K, k, form, policy, step, weights)
    ids = np.zeros(K, np.int64)
    F = np.zeros(K, np.float64)
    got = ctypes.c_int32(0)
    stats = eahr_stats()
    _check(_lib.eahr_topk(cursor, sp.ctypes.data, sp.size, ctypes.byref(p), ids.ctypes.data,
                          F.ctypes.data, ctypes.byref(got), ctypes.byref(stats)), "eahr_topk")
    return _eahr_result(0, ids, F, got, stats)


def eahr_topk_lists(list0, list1, K: int = 20, k: int = 60, form: int = EAHR_RANK_SCALED,
                    policy: int = EAHR_POLICY_GEOMETRIC, step: int = 0, weights=(1, 1)):
    a = np.ascontiguousarray(list0, dtype=np.int64)
    b = np.ascontiguousarray(list1, dtype=np.int64)
    p = _params(K, k, form, policy, step, weights)
    ids = np.zeros(K, np.int64)
    F = np.zeros(K, np.float64)
    got = ctypes.c_int32(0)
    stats = eahr_stats()
    _check(_lib.eahr_topk_lists(a.ctypes.data, a.size, b.ctypes.data, b.size, ctypes.byref(p),
                                ids.ctypes.data, F.ctypes.data, ctypes.byref(got),
                                ctypes.byref(stats)), "eahr_topk_lists")
    return _eahr_result(0, ids, F, got, stats)


# --------------------------------------------------------------------------
# PBM sparse rank generator (Sec. 2.3.2, App. A.2; include/pbm.h)
# --------------------------------------------------------------------------

def _array_arg(x, dtype):
    """(pointer, size, on_device, keepalive) of a 1-D numpy or torch array."""
    try:
        import torch
    except ImportError:  # pragma: no cover
        torch = None
    if torch is not None and isinstance(x, torch.Tensor):
        tdt = {np.int64: torch.int64, np.int32: torch.int32, np.float32: torch.float32}[dtype]
        if x.dtype != tdt:
            raise TypeError(f"expected {tdt}")
        x = x.contiguous()
        if x.is_cuda:
            torch.cuda.current_stream(x.device).synchronize()
        return ctypes.c_void_p(x.data_ptr()), x.numel(), 1 if x.is_cuda else 0, x
    a = np.ascontiguousarray(x, dtype=dtype)
    return ctypes.c_void_p(a.ctypes.data), a.size, 0, a


def pbm_build(term_off, docs, imps, n_items: int, block: int = 0, stream=None):
    """PBM index from term-major postings (numpy or torch; all three on the
    same side): term_off int64 [n_terms + 1], docs int32, imps float32."""
    o, n_off, dev_o, ko = _array_arg(term_off, np.int64)
    d, n_d, dev_d, kd = _array_arg(docs, np.int32)
    p, n_p, dev_p, kp = _array_arg(imps, np.float32)
    if not (dev_o == dev_d == dev_p):
        raise ValueError("postings arrays must all be on the host or all on the device")
    if n_d != n_p:
        raise ValueError("one impact per posting")
    out = ctypes.c_void_p()
    st = ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else stream)
    _check(_lib.pbm_build(o, n_off - 1, d, p, n_d, int(n_items), int(block), dev_o, st,
                          ctypes.byref(out)), "pbm_build")
    return out


def pbm_index_items(index) -> int:
    return int(_lib.pbm_index_items(index))


def pbm_index_ranges(index) -> int:
    return int(_lib.pbm_index_ranges(index))


def pbm_index_free(index) -> None:
    _lib.pbm_index_free(index)


def pbm_cursor_open(index, terms, weights, snap=None, stream=None):
    """PBM cursor for the query (terms, weights); with `snap` (a PVS snapshot
    of the same id space) the items it deletes are left out of the ranking;
    `stream` (a CUDA stream handle, or an object with .cuda_stream) carries
    the cursor's device work."""
    t = np.ascontiguousarray(terms, dtype=np.int32)
    w = np.ascontiguousarray(weights, dtype=np.float32)
    if t.shape != w.shape:
        raise ValueError("one weight per query term")
    out = ctypes.c_void_p()
    if stream is not None:
        handle = getattr(stream, "cuda_stream", stream)
        _check(_lib.pbm_cursor_open_stream(index, snap, t.ctypes.data, w.ctypes.data, t.size,
                                           ctypes.c_void_p(int(handle)), ctypes.byref(out)),
               "pbm_cursor_open_stream")
    elif snap is None:
        _check(_lib.pbm_cursor_open(index, t.ctypes.data, w.ctypes.data, t.size,
                                    ctypes.byref(out)), "pbm_cursor_open")
    else:
        _check(_lib.pbm_cursor_open_snapshot(index, snap, t.ctypes.data, w.ctypes.data, t.size,
                                             ctypes.byref(out)), "pbm_cursor_open_snapshot")
    return out


def pbm_next(cursor, n: int):
    """Next up to n sparse ranks -> (ids int64, scores float32, status)."""
    ids = np.empty(max(int(n), 1), np.int64)
    sc = np.empty(max(int(n), 1), np.float32)
    got = ctypes.c_int32(0)
    s = _check(_lib.pbm_next(cursor, int(n), ids.ctypes.data, sc.ctypes.data,
                             ctypes.byref(got)), "pbm_next")
    return ids[:got.value], sc[:got.value], s


def pbm_cursor_range_bounds(cursor, first: int, count: int):
    """H_hat(R) of ranges first .. first+count-1 as computed at open."""
    H = np.empty(max(int(count), 1), np.float32)
    _check(_lib.pbm_cursor_range_bounds(cursor, int(first), int(count), H.ctypes.data),
           "pbm_cursor_range_bounds")
    return H[:int(count)]


def pbm_cursor_stats(cursor) -> dict:
    st = pbm_stats()
    _check(_lib.pbm_cursor_stats(cursor, ctypes.byref(st)), "pbm_cursor_stats")
    return {n: getattr(st, n) for n, _ in pbm_stats._fields_ if n != "reserved"}


def pbm_cursor_close(cursor) -> None:
    _lib.pbm_cursor_close(cursor)


def eahr_topk_pbm(cursor, sparse_cursor, K: int = 20, k: int = 60, form: int = EAHR_NUMERATOR,
                  policy: int = EAHR_POLICY_GEOMETRIC, step: int = 0, weights=(1, 1)):
    """Ordered Top-K of complete-list weighted RRF with the sparse ranks pulled
    from a PBM cursor -> (ids int64[q_K], F float64[q_K], stats)."""
    p = _params(K, k, form, policy, step, weights)
    ids = np.zeros(K, np.int64)
    F = np.zeros(K, np.float64)
    got = ctypes.c_int32(0)
    stats = eahr_stats()
    _check(_lib.eahr_topk_pbm(cursor, sparse_cursor, ctypes.byref(p), ids.ctypes.data,
                              F.ctypes.data, ctypes.byref(got), ctypes.byref(stats)),
           "eahr_topk_pbm")
    return _eahr_result(0, ids, F, got, stats)


# --------------------------------------------------------------------------
# hierarchical Segment / Shard merging (Sec. 2.4; include/merge.h)
# --------------------------------------------------------------------------

def pvs_merge_open(children):
    """children: a list of (kind, cursor, id_offset) with kind PVS_CHILD_DENSE
    (pvs cursor), PVS_CHILD_SPARSE (pbm cursor) or PVS_CHILD_MERGE."""
    arr = (pvs_merge_child * len(children))()
    for i, (kind, cur, off) in enumerate(children):
        arr[i].kind = int(kind)
        arr[i].cursor = cur.value if isinstance(cur, ctypes.c_void_p) else cur
        arr[i].id_offset = int(off)
    out = ctypes.c_void_p()
    _check(_lib.pvs_merge_open(arr, len(children), ctypes.byref(out)), "pvs_merge_open")
    return out


def pvs_merge_next(merge, n: int):
    ids = np.empty(max(int(n), 1), np.int64)
    sc = np.empty(max(int(n), 1), np.float32)
    got = ctypes.c_int32(0)
    s = _check(_lib.pvs_merge_next(merge, int(n), ids.ctypes.data, sc.ctypes.data,
                                   ctypes.byref(got)), "pvs_merge_next")
    return ids[:got.value], sc[:got.value], s


def pvs_merge_stats(merge) -> dict:
    st = pvs_merge_stats_t()
    _check(_lib.pvs_merge_stats_get(merge, ctypes.byref(st)), "pvs_merge_stats_get")
    return {n: getattr(st, n) for n, _ in pvs_merge_stats_t._fields_ if n != "reserved"}


def pvs_merge_close(merge) -> None:
    _lib.pvs_merge_close(merge)


def eahr_topk_merge(dense_merge, sparse_merge, K: int = 20, k: int = 60,
                    form: int = EAHR_NUMERATOR, policy: int = EAHR_POLICY_GEOMETRIC, step: int = 0,
                    weights=(1, 1)):
    p = _params(K, k, form, policy, step, weights)
    ids = np.zeros(K, np.int64)
    F = np.zeros(K, np.float64)
    got = ctypes.c_int32(0)
    stats = eahr_stats()
    _check(_lib.eahr_topk_merge(dense_merge, sparse_merge, ctypes.byref(p), ids.ctypes.data,
                                F.ctypes.data, ctypes.byref(got), ctypes.byref(stats)),
           "eahr_topk_merge")
    return _eahr_result(0, ids, F, got, stats)


# --------------------------------------------------------------------------
# native request executor (Sec. 2.1 paging over PVS cursors; include/executor.h)
# --------------------------------------------------------------------------

def pvs_executor_create(index, workers: int = 8):
    """Start `workers` native worker threads (one CUDA stream each) for index."""
    out = ctypes.c_void_p()
    _check(_lib.pvs_executor_create(index, int(workers), ctypes.byref(out)), "pvs_executor_create")
    return out


def _host_buffer(x, dtype, shape, what):
    """A host numpy array or CPU torch tensor of dtype and shape -> (pointer, array)."""
    if x is None:
        a = np.empty(shape, dtype)
        return a.ctypes.data, a
    if hasattr(x, "data_ptr"):
        import torch
        want = {np.int64: torch.int64, np.float32: torch.float32, np.int32: torch.int32}[dtype]
        if x.is_cuda or x.dtype != want or tuple(x.shape) != tuple(shape) or not x.is_contiguous():
            raise ValueError(f"{what}: want a contiguous CPU {want} tensor of shape {shape}")
        return x.data_ptr(), x
    if (not isinstance(x, np.ndarray) or x.dtype != dtype or x.shape != tuple(shape)
            or not x.flags.c_contiguous):
        raise ValueError(f"{what}: want a C-contiguous {np.dtype(dtype)} array of shape {shape}")
    return x.ctypes.data, x


def pvs_executor_run(ex, queries, ranks: int, page: int, snap=None, ids=None, scores=None,
                     n_out=None, status=None):
    """Serve one request per row of `queries` (host: numpy float32 or a CPU,
    preferably pinned, torch float32 tensor): `ranks` ranks each, read in
    pages of `page` through the host path.  Outputs may be given as host
    buffers (numpy / CPU torch) to be filled in place.  Returns (ids [nq,
    ranks], scores [nq, ranks], n_out [nq], status [nq], rc); raises
    PvsError when the arguments are rejected (then nothing ran)."""
    if hasattr(queries, "data_ptr"):
        if queries.is_cuda or queries.dtype.itemsize != 4 or queries.dim() != 2:
            raise ValueError("queries: want a 2-D CPU float32 tensor")
        q = queries.contiguous()
        qptr, nq = q.data_ptr(), q.shape[0]
    else:
        q = np.ascontiguousarray(queries, dtype=np.float32)
        if q.ndim != 2:
            raise ValueError("queries: want a 2-D array")
        qptr, nq = q.ctypes.data, q.shape[0]
    pi, ids = _host_buffer(ids, np.int64, (nq, ranks), "ids")
    ps, scores = _host_buffer(scores, np.float32, (nq, ranks), "scores")
    pn, n_out = _host_buffer(n_out, np.int32, (nq,), "n_out")
    pst, status = _host_buffer(status, np.int32, (nq,), "status")
    status[:] = 0
    rc = _lib.pvs_executor_run(ex, snap, qptr, int(nq), int(ranks), int(page), pi, ps, pn, pst)
    if rc < 0 and not any(int(v) == rc for v in status):
        raise PvsError(rc, "pvs_executor_run")
    return ids, scores, n_out, status, rc


def pvs_executor_set_group(ex, group: int) -> None:
    """Serve requests `group` at a time from one grouped pass over the codes."""
    _check(_lib.pvs_executor_set_group(ex, int(group)), "pvs_executor_set_group")


def pvs_executor_run_device(ex, queries, ranks: int, page: int, ids, scores, snap=None):
    """pvs_executor_run with device-resident buffers: queries (CUDA float32
    [nq, dim]), ids (CUDA int64 [nq, ranks]) and scores (CUDA float32 [nq,
    ranks]), all contiguous on the index's device.  Returns (n_out [nq],
    status [nq], rc) as host arrays."""
    import torch
    for t, dt, shape, what in ((queries, torch.float32, None, "queries"),
                               (ids, torch.int64, None, "ids"),
                               (scores, torch.float32, None, "scores")):
        if not (isinstance(t, torch.Tensor) and t.is_cuda and t.is_contiguous() and
                t.dtype == dt and t.dim() == 2):
            raise ValueError(f"{what}: want a contiguous 2-D CUDA {dt} tensor")
    nq = int(queries.shape[0])
    if tuple(ids.shape) != (nq, ranks) or tuple(scores.shape) != (nq, ranks):
        raise ValueError(f"ids and scores: want shape ({nq}, {ranks})")
    n_out = np.zeros(nq, np.int32)
    status = np.zeros(nq, np.int32)
    rc = _lib.pvs_executor_run_ex(ex, snap, ctypes.c_void_p(queries.data_ptr()), nq, int(ranks),
                                  int(page), 1, ctypes.c_void_p(ids.data_ptr()),
                                  ctypes.c_void_p(scores.data_ptr()), n_out.ctypes.data,
                                  status.ctypes.data)
    if rc < 0 and not any(int(v) == rc for v in status):
        raise PvsError(rc, "pvs_executor_run_ex")
    return n_out, status, rc


def pvs_executor_stats(ex) -> dict:
    st = pvs_executor_stats_t()
    _check(_lib.pvs_executor_stats_get(ex, ctypes.byref(st)), "pvs_executor_stats_get")
    return {n: getattr(st, n) for n, _ in pvs_executor_stats_t._fields_}


def pvs_executor_destroy(ex) -> None:
    _lib.pvs_executor_destroy(ex)
