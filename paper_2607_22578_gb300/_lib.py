"""Thin ctypes binding of libhs.so with the C ABI's names.

Argument marshalling only: every function passes device pointers
(``tensor.data_ptr()``), sizes and the current torch CUDA stream to the
library and returns the tensors it wrote.  Workspaces and outputs are torch
allocations when the caller does not pass them.  Every step of the path runs
in the library's kernels; if the library cannot be built or loaded, these
functions raise instead of computing anything another way.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

HS_OK = 0
HS_ERR_INVALID_ARG = 1
HS_ERR_UNSUPPORTED = 2
HS_ERR_CUDA = 3
HS_ERR_WORKSPACE = 4
HS_ERR_TIMEOUT = 5
HS_FNV64_OFFSET_BASIS = 0xCBF29CE484222325
HS_TOPK_MAX_K = 1024
HS_MERGE_QUERIES_MAX = 256

_STATUS = {0: "HS_OK", 1: "HS_ERR_INVALID_ARG", 2: "HS_ERR_UNSUPPORTED", 3: "HS_ERR_CUDA",
           4: "HS_ERR_WORKSPACE", 5: "HS_ERR_TIMEOUT"}

_lock = threading.Lock()
_lib = None


class HsError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__("%s: %s" % (_STATUS.get(status, str(status)), msg))
        self.status = status


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libhs.so (building it first if it is missing or stale)."""
    global _lib
    with _lock:
        if _lib is None:
            if build_if_missing:
                _build.build()
            if not os.path.exists(_build.LIB):
                raise RuntimeError("libhs.so is missing: run paper_2607_22578_gb300.build.build()")
            lib = ctypes.CDLL(_build.LIB)
            P, i64, i32, u64, sz = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32,
                                    ctypes.c_uint64, ctypes.c_size_t)
            st = ctypes.c_int
            lib.hs_last_error.restype = ctypes.c_char_p
            lib.hs_version.restype = ctypes.c_char_p
            lib.hs_fingerprint.argtypes = [P, i64, i32, P, u64, P, P]
            lib.hs_fingerprint.restype = st
            lib.hs_unique_inverse_workspace.argtypes = [i64]
            lib.hs_unique_inverse_workspace.restype = sz
            lib.hs_unique_inverse.argtypes = [P, P, i64, i32, P, P, P, P, P, sz, P]
            lib.hs_unique_inverse.restype = st
            lib.hs_unique_inverse_noalloc.argtypes = [P, P, i64, i32, P, P, P, P, P]
            lib.hs_unique_inverse_noalloc.restype = st
            lib.hs_retrieve_topk_workspace.argtypes = [i64, i64, i32, i32]
            lib.hs_retrieve_topk_workspace.restype = sz
            lib.hs_retrieve_topk.argtypes = [P, i64, P, i64, i32, i32, P, P, P, sz, P]
            lib.hs_retrieve_topk.restype = st
            lib.hs_retrieve_topk_n.argtypes = [P, i64, P, P, i64, i32, i32, P, P, P, sz, P]
            lib.hs_retrieve_topk_n.restype = st
            lib.hs_retrieve_topk_fanout.argtypes = [P, i64, P, P, i64, P, i64, i32, i32, P, P,
                                                    P, sz, P]
            lib.hs_retrieve_topk_fanout.restype = st
            lib.hs_merge_queries.argtypes = [P, i64, i32, u64, P, P, P, P, P, P, P]
            lib.hs_merge_queries.restype = st
            lib.hs_rerank_topk.argtypes = [P, i64, P, P, i64, i32, P, i32, i32, P, i64, P, P, P]
            lib.hs_rerank_topk.restype = st
            lib.hs_cache_bytes.argtypes = [i64, i32, i32]
            lib.hs_cache_bytes.restype = sz
            lib.hs_cache_init.argtypes = [P, sz, i64, i32, i32, P]
            lib.hs_cache_init.restype = st
            lib.hs_cache_lookup.argtypes = [P, sz, i64, i32, i32, P, P, P, i64, P, P, P, P, P, P, P]
            lib.hs_cache_lookup.restype = st
            lib.hs_cache_insert.argtypes = [P, sz, i64, i32, i32, P, P, i64, P, P, P, P, P, P, P, P]
            lib.hs_cache_insert.restype = st
            lib.hs_cache_stats.argtypes = [P, P, P, P]
            lib.hs_cache_stats.restype = st
            lib.hs_segment_sum.argtypes = [P, P, i64, P, i64, P, P]
            lib.hs_segment_sum.restype = st
            lib.hs_scatter_results.argtypes = [P, i64, i64, P, i64, P, P]
            lib.hs_scatter_results.restype = st
            lib.hs_get_device_error.argtypes = [P]
            lib.hs_get_device_error.restype = st
            lib.hs_launch_count.restype = ctypes.c_uint64
            lib.hs_debug_scan_wait.argtypes = [u64, i64]
            lib.hs_debug_scan_wait.restype = st
            lib.hs_merge_rows_workspace.argtypes = [i64]
            lib.hs_merge_rows_workspace.restype = sz
            lib.hs_merge_rows.argtypes = [P, i64, i32, P, u64, P, P, P, P, P, sz, P]
            lib.hs_merge_rows.restype = st
            lib.hs_debug_merge_key_mask.argtypes = [u64]
            lib.hs_debug_merge_key_mask.restype = st
            lib.hs_debug_retrieve_wait.argtypes = [u64, i32]
            lib.hs_debug_retrieve_wait.restype = st
            lib.hs_memcpy_async.argtypes = [P, P, sz, P]
            lib.hs_memcpy_async.restype = st
            lib.hs_debug_stream_rows.argtypes = [P, i64, i32, P, i32, P, i32, P]
            lib.hs_debug_stream_rows.restype = st
            _lib = lib
    return _lib


def _check(status: int) -> None:
    if status != HS_OK:
        raise HsError(status, load().hs_last_error().decode())


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _ptr(t):
    return None if t is None else t.data_ptr()


def _cuda(t: torch.Tensor, name: str) -> torch.Tensor:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError("%s must be a CUDA tensor" % name)
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    return t


def hs_version() -> str:
    return load().hs_version().decode()


def hs_fingerprint(tokens: torch.Tensor, lens: torch.Tensor | None = None,
                   seed_state: int = HS_FNV64_OFFSET_BASIS, fp_out: torch.Tensor | None = None,
                   stream=None) -> torch.Tensor:
    """fp[i] = FNV-1a-64 over row i's little-endian token octets (int64 tensor
    holding the uint64 bit patterns)."""
    _cuda(tokens, "tokens")
    if tokens.dtype != torch.int32 or tokens.dim() != 2:
        raise TypeError("tokens must be a 2-D int32 tensor")
    n, stride = tokens.shape
    if lens is not None:
        _cuda(lens, "lens")
        if lens.dtype != torch.int32 or lens.numel() != n:
            raise TypeError("lens must be int32 [n_rows]")
    if fp_out is None:
        fp_out = torch.empty(n, dtype=torch.int64, device=tokens.device)
    _check(load().hs_fingerprint(_ptr(tokens), n, stride, _ptr(lens), seed_state & (2**64 - 1),
                                 _ptr(fp_out), _stream(stream)))
    return fp_out


def hs_unique_inverse_workspace(n_rows: int) -> int:
    return int(load().hs_unique_inverse_workspace(n_rows))


def hs_unique_inverse(fp: torch.Tensor, tokens: torch.Tensor, lens: torch.Tensor | None = None,
                      workspace: torch.Tensor | None = None, out: tuple | None = None,
                      stream=None):
    """Exact unique rows.  Returns (n_unique_dev [1] int32, unique_idx [n]
    int32, inverse [n] int32); only the first n_unique entries of unique_idx
    are meaningful."""
    _cuda(fp, "fp")
    _cuda(tokens, "tokens")
    n, stride = tokens.shape
    dev = tokens.device
    if out is None:
        out = (torch.empty(1, dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev))
    nu, uidx, inv = out
    need = hs_unique_inverse_workspace(n)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=dev)
    _check(load().hs_unique_inverse(_ptr(fp), _ptr(tokens), n, stride, _ptr(lens), _ptr(nu),
                                    _ptr(uidx), _ptr(inv), _ptr(workspace), workspace.numel(),
                                    _stream(stream)))
    return nu, uidx[:n], inv[:n]


def hs_merge_rows_workspace(n_rows: int) -> int:
    return int(load().hs_merge_rows_workspace(int(n_rows)))


def hs_merge_rows(tokens: torch.Tensor, lens: torch.Tensor | None = None,
                  seed_state: int = HS_FNV64_OFFSET_BASIS, workspace: torch.Tensor | None = None,
                  out: tuple | None = None, stream=None):
    """Fingerprint and exact merge in one pass.  Returns (fp [n] int64 (uint64
    bits), n_unique_dev [1] int32, unique_idx [n] int32, inverse [n] int32);
    `out`, if given, is that tuple of preallocated tensors."""
    _cuda(tokens, "tokens")
    n, stride = tokens.shape
    dev = tokens.device
    if out is None:
        out = (torch.empty(max(n, 1), dtype=torch.int64, device=dev),
               torch.empty(1, dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev))
    fp, nu, uidx, inv = out
    need = hs_merge_rows_workspace(n)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=dev)
    _check(load().hs_merge_rows(_ptr(tokens), n, stride, _ptr(lens), int(seed_state), _ptr(fp),
                                _ptr(nu), _ptr(uidx), _ptr(inv), _ptr(workspace),
                                workspace.numel(), _stream(stream)))
    return fp[:n], nu, uidx[:n], inv[:n]


def hs_debug_merge_key_mask(mask: int = 0) -> None:
    """Test hook of hs_merge_rows: key the table by fp & mask (0 restores
    all ones; see hs.h)."""
    _check(load().hs_debug_merge_key_mask(int(mask)))


def hs_memcpy_async(dst: torch.Tensor, src: torch.Tensor, stream=None) -> torch.Tensor:
    """Copy src into dst (equal byte sizes, contiguous; host, pinned host or
    device on either side) on `stream` through the C ABI.  Returns dst."""
    if not dst.is_contiguous() or not src.is_contiguous():
        raise ValueError("dst and src must be contiguous")
    nbytes = dst.numel() * dst.element_size()
    if nbytes != src.numel() * src.element_size():
        raise ValueError("dst and src differ in size")
    if not (dst.is_cuda or src.is_cuda):
        raise ValueError("one side must be on the GPU")
    _check(load().hs_memcpy_async(ctypes.c_void_p(dst.data_ptr()), ctypes.c_void_p(src.data_ptr()),
                                  nbytes, _stream(stream)))
    return dst


def hs_debug_retrieve_wait(limit_ns: int = 0, withhold_first: int = 0) -> None:
    """Test hook of the retrieval's bounded waits: the wait limit (0: 2 s)
    and whether every CTA withholds its first stage (see hs.h)."""
    _check(load().hs_debug_retrieve_wait(int(limit_ns), int(withhold_first)))


def hs_unique_inverse_noalloc(fp: torch.Tensor, tokens: torch.Tensor,
                              lens: torch.Tensor | None = None, out: tuple | None = None,
                              stream=None):
    """hs_unique_inverse without a workspace, for callers that cannot
    allocate device memory (at most 65536 rows; the scratch is a fixed array
    inside the library).  Pass preallocated `out` = (n_unique_dev [1],
    unique_idx [n], inverse [n]) int32 tensors to allocate nothing here
    either."""
    _cuda(fp, "fp")
    _cuda(tokens, "tokens")
    n, stride = tokens.shape
    dev = tokens.device
    if out is None:
        out = (torch.empty(1, dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev))
    nu, uidx, inv = out
    _check(load().hs_unique_inverse_noalloc(_ptr(fp), _ptr(tokens), n, stride, _ptr(lens),
                                            _ptr(nu), _ptr(uidx), _ptr(inv), _stream(stream)))
    return nu, uidx[:n], inv[:n]


def hs_retrieve_topk_workspace(n_queries: int, n_corpus: int, dim: int, k: int) -> int:
    return int(load().hs_retrieve_topk_workspace(n_queries, n_corpus, dim, k))


def hs_retrieve_topk(queries: torch.Tensor, corpus: torch.Tensor, k: int,
                     workspace: torch.Tensor | None = None, out: tuple | None = None,
                     stream=None):
    """Top-k inner products of bf16 query rows against bf16 corpus rows.
    Returns (scores fp32 [Q, k], ids int32 [Q, k])."""
    _cuda(queries, "queries")
    _cuda(corpus, "corpus")
    if queries.element_size() != 2 or corpus.element_size() != 2:
        raise TypeError("queries and corpus must hold bf16 (2-byte) elements")
    Q, d = queries.shape
    N, d2 = corpus.shape
    if d != d2:
        raise ValueError("dimension mismatch")
    dev = queries.device
    if out is None:
        out = (torch.empty((Q, k), dtype=torch.float32, device=dev),
               torch.empty((Q, k), dtype=torch.int32, device=dev))
    scores, ids = out
    if workspace is None:
        workspace = torch.empty(hs_retrieve_topk_workspace(Q, N, d, k), dtype=torch.uint8,
                                device=dev)
    _check(load().hs_retrieve_topk(_ptr(queries), Q, _ptr(corpus), N, d, k, _ptr(scores),
                                   _ptr(ids), _ptr(workspace), workspace.numel(), _stream(stream)))
    return scores, ids


def hs_retrieve_topk_n(queries: torch.Tensor, n_queries_dev: torch.Tensor, corpus: torch.Tensor,
                       k: int, workspace: torch.Tensor | None = None, out: tuple | None = None,
                       stream=None):
    """hs_retrieve_topk over the first n_queries_dev[0] rows of `queries`
    (a device int32 scalar, read when the kernels run).  Returns (scores,
    ids) shaped like `queries` rows x k; rows past the count are left as
    they were."""
    _cuda(queries, "queries")
    _cuda(corpus, "corpus")
    _cuda(n_queries_dev, "n_queries_dev")
    if n_queries_dev.dtype != torch.int32:
        raise TypeError("n_queries_dev must be int32")
    if queries.element_size() != 2 or corpus.element_size() != 2:
        raise TypeError("queries and corpus must hold bf16 (2-byte) elements")
    Q, d = queries.shape
    N, d2 = corpus.shape
    if d != d2:
        raise ValueError("dimension mismatch")
    dev = queries.device
    if out is None:
        out = (torch.empty((Q, k), dtype=torch.float32, device=dev),
               torch.empty((Q, k), dtype=torch.int32, device=dev))
    scores, ids = out
    if workspace is None:
        workspace = torch.empty(hs_retrieve_topk_workspace(Q, N, d, k), dtype=torch.uint8,
                                device=dev)
    _check(load().hs_retrieve_topk_n(_ptr(queries), Q, _ptr(n_queries_dev), _ptr(corpus), N, d,
                                     k, _ptr(scores), _ptr(ids), _ptr(workspace),
                                     workspace.numel(), _stream(stream)))
    return scores, ids


def hs_retrieve_topk_fanout(queries: torch.Tensor, n_queries_dev: torch.Tensor | None,
                            inverse: torch.Tensor, corpus: torch.Tensor, k: int,
                            workspace: torch.Tensor | None = None, out: tuple | None = None,
                            stream=None):
    """Retrieval whose results go to every merged row: row o of the returned
    (scores [n_out, k], ids [n_out, k]) is the top-k of query inverse[o]
    (n_out = inverse.numel()).  n_queries_dev (device int32 scalar) or None
    gives the query count, as for hs_retrieve_topk_n."""
    _cuda(queries, "queries")
    _cuda(corpus, "corpus")
    _cuda(inverse, "inverse")
    if inverse.dtype != torch.int32:
        raise TypeError("inverse must be int32")
    if n_queries_dev is not None:
        _cuda(n_queries_dev, "n_queries_dev")
        if n_queries_dev.dtype != torch.int32:
            raise TypeError("n_queries_dev must be int32")
    if queries.element_size() != 2 or corpus.element_size() != 2:
        raise TypeError("queries and corpus must hold bf16 (2-byte) elements")
    Q, d = queries.shape
    N, d2 = corpus.shape
    if d != d2:
        raise ValueError("dimension mismatch")
    n_out = inverse.numel()
    dev = queries.device
    if out is None:
        out = (torch.empty((n_out, k), dtype=torch.float32, device=dev),
               torch.empty((n_out, k), dtype=torch.int32, device=dev))
    scores, ids = out
    if workspace is None:
        workspace = torch.empty(hs_retrieve_topk_workspace(Q, N, d, k), dtype=torch.uint8,
                                device=dev)
    _check(load().hs_retrieve_topk_fanout(_ptr(queries), Q, _ptr(n_queries_dev), _ptr(inverse),
                                          n_out, _ptr(corpus), N, d, k, _ptr(scores), _ptr(ids),
                                          _ptr(workspace), workspace.numel(), _stream(stream)))
    return scores, ids


def hs_merge_queries(queries: torch.Tensor, seed_state: int = HS_FNV64_OFFSET_BASIS,
                     fp_in: torch.Tensor | None = None, out: tuple | None = None, stream=None):
    """Fingerprint, exact merge and gather of a query batch (at most
    HS_MERGE_QUERIES_MAX rows of bf16 vectors) in one launch.  Returns
    (fp [n] int64, n_unique_dev [1] int32, unique_idx [n] int32,
    inverse [n] int32, unique_queries [n, dim]); the first n_unique rows of
    unique_queries are the unique query vectors.  ``out`` may supply those
    five tensors preallocated; ``fp_in`` replaces the computed fingerprints."""
    _cuda(queries, "queries")
    if queries.element_size() != 2 or queries.dim() != 2:
        raise TypeError("queries must be a 2-D tensor of bf16 (2-byte) elements")
    n, d = queries.shape
    dev = queries.device
    if fp_in is not None:
        _cuda(fp_in, "fp_in")
        if fp_in.dtype != torch.int64 or fp_in.numel() != n:
            raise TypeError("fp_in must be int64 [n]")
    if out is None:
        out = (torch.empty(max(n, 1), dtype=torch.int64, device=dev),
               torch.empty(1, dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               torch.empty((max(n, 1), d), dtype=queries.dtype, device=dev))
    fp, nu, uidx, inv, uq = out
    _check(load().hs_merge_queries(_ptr(queries), n, d, seed_state & (2**64 - 1), _ptr(fp_in),
                                   _ptr(fp), _ptr(nu), _ptr(uidx), _ptr(inv), _ptr(uq),
                                   _stream(stream)))
    return fp[:n], nu, uidx[:n], inv[:n], uq[:n]


def hs_scatter_results(src: torch.Tensor, mapping: torch.Tensor, dst: torch.Tensor | None = None,
                       stream=None) -> torch.Tensor:
    """dst[i] = src[mapping[i]] row-wise (rows are the first dimension)."""
    _cuda(src, "src")
    _cuda(mapping, "map")
    if mapping.dtype != torch.int32:
        raise TypeError("map must be int32")
    n = mapping.numel()
    row_bytes = src[0].numel() * src.element_size() if src.dim() > 1 else src.element_size()
    if dst is None:
        dst = torch.empty((n,) + tuple(src.shape[1:]), dtype=src.dtype, device=src.device)
    _check(load().hs_scatter_results(_ptr(src), src.shape[0], row_bytes, _ptr(mapping), n,
                                     _ptr(dst), _stream(stream)))
    return dst


def hs_rerank_topk(rerank_queries: torch.Tensor, rerank_corpus: torch.Tensor,
                   candidates: torch.Tensor, k2: int, n_queries_dev: torch.Tensor | None = None,
                   inverse: torch.Tensor | None = None, out: tuple | None = None, stream=None):
    """Rescore each query's candidates (int32 [Q, k1] corpus ids) by the
    inner product of bf16 rerank vectors and keep the best k2.  Returns
    (scores fp32, ids int32), one row per query, or one per entry of
    ``inverse`` (row o = query inverse[o]) when it is given."""
    _cuda(rerank_queries, "rerank_queries")
    _cuda(rerank_corpus, "rerank_corpus")
    _cuda(candidates, "candidates")
    if rerank_queries.element_size() != 2 or rerank_corpus.element_size() != 2:
        raise TypeError("rerank vectors must hold bf16 (2-byte) elements")
    if candidates.dtype != torch.int32 or candidates.dim() != 2:
        raise TypeError("candidates must be int32 [Q, k1]")
    Q, d = rerank_queries.shape
    N, d2 = rerank_corpus.shape
    if d != d2:
        raise ValueError("dimension mismatch")
    if candidates.shape[0] != Q:
        raise ValueError("candidates must have one row per query")
    k1 = candidates.shape[1]
    for t, name in ((n_queries_dev, "n_queries_dev"), (inverse, "inverse")):
        if t is not None:
            _cuda(t, name)
            if t.dtype != torch.int32:
                raise TypeError("%s must be int32" % name)
    rows = inverse.numel() if inverse is not None else Q
    dev = rerank_queries.device
    if out is None:
        out = (torch.empty((rows, k2), dtype=torch.float32, device=dev),
               torch.empty((rows, k2), dtype=torch.int32, device=dev))
    scores, ids = out
    _check(load().hs_rerank_topk(_ptr(rerank_queries), Q, _ptr(n_queries_dev),
                                 _ptr(rerank_corpus), N, d, _ptr(candidates), k1, int(k2),
                                 _ptr(inverse), rows if inverse is not None else 0, _ptr(scores),
                                 _ptr(ids), _stream(stream)))
    return scores, ids


class ResultCache:
    """Device-resident fingerprint -> retrieval result table that persists
    across batches (asynchronous cache reuse, Section 3.3 (II)): ``capacity``
    entries of a dim-wide query vector and its k scores and ids, in one
    uint8 tensor allocated here (the library itself allocates nothing)."""

    def __init__(self, capacity: int, dim: int, k: int, device=None, stream=None):
        self.capacity, self.dim, self.k = int(capacity), int(dim), int(k)
        nbytes = int(load().hs_cache_bytes(self.capacity, self.dim, self.k))
        if nbytes == 0:
            raise ValueError("invalid cache shape")
        self.mem = torch.empty(nbytes, dtype=torch.uint8, device=device or "cuda")
        hs_cache_init(self, stream)

    def _args(self):
        return (_ptr(self.mem), self.mem.numel(), self.capacity, self.dim, self.k)


def hs_cache_init(cache: ResultCache, stream=None) -> None:
    """Empty the cache (every entry free, counters zero)."""
    _check(load().hs_cache_init(*cache._args(), _stream(stream)))


def hs_cache_bytes(capacity: int, dim: int, k: int) -> int:
    return int(load().hs_cache_bytes(capacity, dim, k))


def hs_cache_lookup(cache: ResultCache, queries: torch.Tensor, fp: torch.Tensor,
                    fp_rows: torch.Tensor | None = None, n_queries_dev: torch.Tensor | None = None,
                    out: tuple | None = None, miss: tuple | None = None, stream=None):
    """Look the merged queries up in the cache.  Hits get their cached
    (scores, ids) rows in ``out``; misses are listed in ``miss`` =
    (miss_list [Q] int32, n_miss_dev [1] int32, miss_queries [Q, dim]) with
    their vectors gathered for retrieval.  Query u's key is fp[fp_rows[u]]
    (fp[u] if fp_rows is None).  Returns (out, miss)."""
    for t, name in ((queries, "queries"), (fp, "fp")):
        _cuda(t, name)
    Q, d = queries.shape
    dev = queries.device
    if out is None:
        out = (torch.empty((Q, cache.k), dtype=torch.float32, device=dev),
               torch.empty((Q, cache.k), dtype=torch.int32, device=dev))
    if miss is None:
        miss = (torch.empty(max(Q, 1), dtype=torch.int32, device=dev),
                torch.empty(1, dtype=torch.int32, device=dev),
                torch.empty((max(Q, 1), d), dtype=queries.dtype, device=dev))
    _check(load().hs_cache_lookup(*cache._args(), _ptr(queries), _ptr(fp), _ptr(fp_rows), Q,
                                  _ptr(n_queries_dev), _ptr(out[0]), _ptr(out[1]), _ptr(miss[0]),
                                  _ptr(miss[1]), _ptr(miss[2]), _stream(stream)))
    return out, miss


def hs_cache_insert(cache: ResultCache, miss: tuple, fp: torch.Tensor, miss_scores: torch.Tensor,
                    miss_ids: torch.Tensor, out: tuple, fp_rows: torch.Tensor | None = None,
                    stream=None):
    """Insert the retrieved results of the misses of ``hs_cache_lookup``
    (rows of miss_scores / miss_ids follow the miss list) into the cache and
    write them to the queries' rows of ``out``."""
    miss_list, n_miss, miss_q = miss
    _check(load().hs_cache_insert(*cache._args(), _ptr(miss_list), _ptr(n_miss),
                                  miss_list.numel(), _ptr(miss_q), _ptr(fp), _ptr(fp_rows),
                                  _ptr(miss_scores), _ptr(miss_ids), _ptr(out[0]), _ptr(out[1]),
                                  _stream(stream)))
    return out


def hs_cache_stats(cache: ResultCache, stream=None):
    """(hits, misses) counted since the cache was initialised (synchronises)."""
    h, m = ctypes.c_uint64(0), ctypes.c_uint64(0)
    _check(load().hs_cache_stats(_ptr(cache.mem), ctypes.addressof(h), ctypes.addressof(m),
                                 _stream(stream)))
    return int(h.value), int(m.value)


def hs_segment_sum(phi: torch.Tensor, inverse: torch.Tensor, max_groups: int,
                   n_groups_dev: torch.Tensor | None = None, out: torch.Tensor | None = None,
                   stream=None) -> torch.Tensor:
    """out[u] = sum of phi[i] over rows with inverse[i] == u (float64
    [max_groups]; entries past the group count, n_groups_dev[0] if given,
    are 0): the priority contribution of each fused node."""
    _cuda(phi, "phi")
    _cuda(inverse, "inverse")
    if phi.dtype != torch.float64 or inverse.dtype != torch.int32:
        raise TypeError("phi must be float64 and inverse int32")
    if phi.numel() != inverse.numel():
        raise ValueError("phi and inverse differ in length")
    if n_groups_dev is not None:
        _cuda(n_groups_dev, "n_groups_dev")
        if n_groups_dev.dtype != torch.int32:
            raise TypeError("n_groups_dev must be int32")
    if out is None:
        out = torch.empty(max(int(max_groups), 1), dtype=torch.float64, device=phi.device)
    _check(load().hs_segment_sum(_ptr(phi), _ptr(inverse), phi.numel(), _ptr(n_groups_dev),
                                 int(max_groups), _ptr(out), _stream(stream)))
    return out[: int(max_groups)]


def hs_launch_count() -> int:
    """Kernels launched by the library in this process (diagnostics)."""
    return int(load().hs_launch_count())


def hs_get_device_error(stream=None) -> None:
    """Synchronise the stream; raise HsError if a kernel reported a problem."""
    _check(load().hs_get_device_error(_stream(stream)))


def hs_debug_scan_wait(limit_ns: int = 0, withhold_tile: int = -1) -> None:
    """Test hook of hs_unique_inverse's bounded look-back wait (see hs.h);
    hs_debug_scan_wait() restores the defaults."""
    _check(load().hs_debug_scan_wait(int(limit_ns), int(withhold_tile)))


def hs_debug_stream_rows(tokens: torch.Tensor, lens: torch.Tensor | None = None, pattern: int = 0,
                         checksum: torch.Tensor | None = None, blocks_per_sm: int = 4,
                         stream=None) -> torch.Tensor:
    """Read the rows' valid prefixes with one access pattern (diagnostics,
    see hs.h); returns the xor checksum tensor it folded them into."""
    n, stride = tokens.shape
    if checksum is None:
        checksum = torch.zeros(1, dtype=torch.int32, device=tokens.device)
    _check(load().hs_debug_stream_rows(tokens.data_ptr(), n, stride,
                                        None if lens is None else lens.data_ptr(), int(pattern),
                                        checksum.data_ptr(), int(blocks_per_sm), _stream(stream)))
    return checksum
