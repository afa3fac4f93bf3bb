"""Oracle for the embed-and-retrieve hot path (test infrastructure).

Plain, slow CPU implementations of what the GPU library computes; see
``hs_oracle.cpp`` for the definition each function follows and the paper
passage it comes from (Section 3.3 Eq. 2, "Dynamic Fusion and Reuse
Mechanism" and Eq. 3; Appendix A.2; Section 4.1 "Workloads", retrieval and
rerank).

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg may import this package.  The library under ``paper_2607_22578_gb300``
never does: the two share no code.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hs_oracle.cpp")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

FNV64_OFFSET_BASIS = 14695981039346656037


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (portable flags: it runs on x86 and Arm)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp%d" % os.getpid()
        cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-pthread",
               "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            P = ctypes.c_void_p
            i64, i32, u64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_uint64
            lib.oracle_fnv1a64_bytes.argtypes = [P, i64, u64]
            lib.oracle_fnv1a64_bytes.restype = u64
            lib.oracle_fingerprint.argtypes = [P, i64, i32, P, u64, P]
            lib.oracle_fingerprint.restype = ctypes.c_int
            lib.oracle_unique_inverse.argtypes = [P, i64, i32, P, P, P, P]
            lib.oracle_unique_inverse.restype = ctypes.c_int
            lib.oracle_topk.argtypes = [P, i64, P, i64, i32, i32, P, P, i32]
            lib.oracle_topk.restype = ctypes.c_int
            lib.oracle_pair_scores.argtypes = [P, P, i32, P, P, i64, P]
            lib.oracle_pair_scores.restype = None
            lib.oracle_scatter.argtypes = [P, i64, i64, P, i64, P]
            lib.oracle_scatter.restype = ctypes.c_int
            lib.oracle_rerank.argtypes = [P, i64, P, i64, i32, P, i32, i32, P, P]
            lib.oracle_rerank.restype = ctypes.c_int
            lib.oracle_segment_sum.argtypes = [P, P, i64, i64, P]
            lib.oracle_segment_sum.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data


def fnv1a64_bytes(data: bytes, h0: int = FNV64_OFFSET_BASIS) -> int:
    buf = np.frombuffer(data, dtype=np.uint8) if len(data) else np.zeros(1, np.uint8)
    return int(_load().oracle_fnv1a64_bytes(_ptr(buf), len(data), h0))


def fingerprint(tokens: np.ndarray, lens: np.ndarray | None = None,
                seed: int = FNV64_OFFSET_BASIS) -> np.ndarray:
    """FNV-1a-64 over the little-endian octets of tokens[i, :lens[i]]."""
    tokens = np.ascontiguousarray(tokens, dtype=np.int32)
    n, stride = tokens.shape
    if lens is not None:
        lens = np.ascontiguousarray(lens, dtype=np.int32)
    out = np.empty(n, dtype=np.uint64)
    rc = _load().oracle_fingerprint(_ptr(tokens), n, stride, _ptr(lens), seed, _ptr(out))
    if rc:
        raise ValueError("row length outside [0, stride]")
    return out


def unique_inverse(tokens: np.ndarray, lens: np.ndarray | None = None):
    """Exact unique rows (first occurrence, ascending) and the inverse map."""
    tokens = np.ascontiguousarray(tokens, dtype=np.int32)
    n, stride = tokens.shape
    if lens is not None:
        lens = np.ascontiguousarray(lens, dtype=np.int32)
    nu = np.zeros(1, dtype=np.int32)
    uidx = np.empty(max(n, 1), dtype=np.int32)
    inv = np.empty(max(n, 1), dtype=np.int32)
    rc = _load().oracle_unique_inverse(_ptr(tokens), n, stride, _ptr(lens), _ptr(nu),
                                       _ptr(uidx), _ptr(inv))
    if rc:
        raise ValueError("row length outside [0, stride]")
    return uidx[: int(nu[0])].copy(), inv[:n].copy()


def topk(queries: np.ndarray, corpus: np.ndarray, k: int, nthreads: int = 0):
    """Exact fp64 top-k by inner product over bf16 bit patterns (uint16)."""
    queries = np.ascontiguousarray(queries, dtype=np.uint16)
    corpus = np.ascontiguousarray(corpus, dtype=np.uint16)
    nq, d = queries.shape
    N, d2 = corpus.shape
    assert d == d2
    scores = np.empty((nq, k), dtype=np.float64)
    ids = np.empty((nq, k), dtype=np.int32)
    rc = _load().oracle_topk(_ptr(queries), nq, _ptr(corpus), N, d, k, _ptr(scores),
                             _ptr(ids), nthreads)
    if rc:
        raise ValueError("k outside [1, N]")
    return scores, ids


def pair_scores(queries: np.ndarray, corpus: np.ndarray, qi: np.ndarray,
                cj: np.ndarray) -> np.ndarray:
    """fp64 inner products of the listed (query row, corpus row) pairs."""
    queries = np.ascontiguousarray(queries, dtype=np.uint16)
    corpus = np.ascontiguousarray(corpus, dtype=np.uint16)
    qi = np.ascontiguousarray(qi, dtype=np.int64)
    cj = np.ascontiguousarray(cj, dtype=np.int64)
    assert qi.shape == cj.shape
    out = np.empty(qi.shape, dtype=np.float64)
    _load().oracle_pair_scores(_ptr(queries), _ptr(corpus), queries.shape[1], _ptr(qi),
                               _ptr(cj), qi.size, _ptr(out))
    return out


def scatter(src: np.ndarray, mapping: np.ndarray) -> np.ndarray:
    """dst[i] = src[mapping[i]] row-wise (rows are the first axis)."""
    src = np.ascontiguousarray(src)
    mapping = np.ascontiguousarray(mapping, dtype=np.int32)
    row_bytes = src.strides[0] if src.ndim > 1 else src.itemsize
    n = mapping.shape[0]
    dst = np.empty((n,) + src.shape[1:], dtype=src.dtype)
    rc = _load().oracle_scatter(_ptr(src), src.shape[0], row_bytes, _ptr(mapping), n,
                                _ptr(dst))
    if rc:
        raise IndexError("map entry outside [0, n_src)")
    return dst


def segment_sum(phi: np.ndarray, inverse: np.ndarray, n_groups: int) -> np.ndarray:
    """out[u] = sum of phi[i] over rows with inverse[i] == u (fp64, ascending
    row order): the priority contribution of a fused node (Section 3.3,
    Eq. 3)."""
    phi = np.ascontiguousarray(phi, dtype=np.float64)
    inverse = np.ascontiguousarray(inverse, dtype=np.int32)
    assert phi.shape == inverse.shape
    out = np.empty(max(int(n_groups), 1), dtype=np.float64)
    rc = _load().oracle_segment_sum(_ptr(phi), _ptr(inverse), phi.size, int(n_groups), _ptr(out))
    if rc:
        raise IndexError("inverse entry outside [0, n_groups)")
    return out[: int(n_groups)].copy()


def rerank(rq: np.ndarray, rc: np.ndarray, cand: np.ndarray, k2: int):
    """Second-stage rerank of retrieved candidates (Section 4.1, RAG with
    rerank): fp64 inner products of bf16 rerank vectors over cand[q, :]
    (negative entries absent), ordered by descending score, ties to the lower
    id; returns the first k2 (scores fp64, ids int32)."""
    rq = np.ascontiguousarray(rq, dtype=np.uint16)
    rc = np.ascontiguousarray(rc, dtype=np.uint16)
    cand = np.ascontiguousarray(cand, dtype=np.int32)
    nq, d = rq.shape
    assert rc.shape[1] == d and cand.shape[0] == nq
    k1 = cand.shape[1]
    scores = np.empty((nq, k2), dtype=np.float64)
    ids = np.empty((nq, k2), dtype=np.int32)
    rc_ = _load().oracle_rerank(_ptr(rq), nq, _ptr(rc), rc.shape[0], d, _ptr(cand), k1, k2,
                                _ptr(scores), _ptr(ids))
    if rc_:
        raise IndexError("candidate id outside [0, n_rc)")
    return scores, ids


def cache_reuse(batches):
    """Asynchronous cache reuse across batches (Section 3.3, "Dynamic Fusion
    and Reuse Mechanism" (II)) with unbounded capacity: a node of a later
    batch that equals a node completed in an earlier batch takes that
    node's result instead of executing.  ``batches`` is a sequence of 2-D
    arrays of rows (the merged nodes of each batch); returns, per batch, a
    bool array: True where the row equals a row of an earlier batch."""
    seen = set()
    out = []
    for rows in batches:
        rows = np.ascontiguousarray(rows)
        hit = np.array([r.tobytes() in seen for r in rows], dtype=bool)
        for r in rows:
            seen.add(r.tobytes())
        out.append(hit)
    return out
