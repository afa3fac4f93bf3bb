"""Seeded synthetic workloads for the embed-and-retrieve hot path.

Inputs only: this package draws random numbers (``gen.c``, a counter-based
SplitMix64 generator) and lays them out in the shapes of the paper's
concurrent-workflow mixes (Section 4.1, "Workloads": duplicate queries
targeting hot documents with Zipfian reuse, many concurrent clients).  It
holds none of the method's arithmetic.  Both the oracle and the GPU library
read what it returns, and each builder also returns the ground-truth
partition it planted, which the tests use to pin the oracle.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gen.c")
_LIB = os.path.join(_HERE, "libsynth.so")
_lock = threading.Lock()
_lib = None

VOCAB = 32000

# Stream ids: one independent random stream per purpose.
_S_TOKENS, _S_LENS, _S_COPYPOS, _S_COPYSRC, _S_ZIPF, _S_PERM = 1, 2, 3, 4, 5, 6
_S_VECTORS, _S_CENTRES, _S_MEMBERS, _S_QCLUSTER, _S_QNOISE, _S_MEMBERNOISE = 7, 8, 9, 10, 11, 12


def build(force: bool = False) -> str:
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp%d" % os.getpid()
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
                        "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp, "-lm"],
                       check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            P, i64, i32, u64, f64 = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32,
                                     ctypes.c_uint64, ctypes.c_double)
            lib.synth_u64.argtypes = [u64, u64, u64]
            lib.synth_u64.restype = u64
            lib.synth_normal.argtypes = [u64, u64, u64]
            lib.synth_normal.restype = f64
            lib.synth_token_rows.argtypes = [P, i64, i32, P, i32, u64, u64, i64, ctypes.c_int]
            lib.synth_token_rows.restype = None
            lib.synth_uniform_ints.argtypes = [P, i64, i32, i32, u64, u64]
            lib.synth_uniform_ints.restype = None
            lib.synth_unit_rows_bf16.argtypes = [P, i64, i32, u64, u64, i64, ctypes.c_int]
            lib.synth_unit_rows_bf16.restype = None
            lib.synth_rows_near_bf16.argtypes = [P, i64, i32, P, P, f64, u64, u64, i64,
                                                 ctypes.c_int]
            lib.synth_rows_near_bf16.restype = None
            lib.synth_unit_centres_f64.argtypes = [P, i64, i32, u64, u64]
            lib.synth_unit_centres_f64.restype = None
            lib.synth_choose_distinct.argtypes = [P, i64, i64, u64, u64]
            lib.synth_choose_distinct.restype = ctypes.c_int
            lib.synth_zipf_ranks.argtypes = [P, i64, i64, f64, u64, u64]
            lib.synth_zipf_ranks.restype = ctypes.c_int
            lib.synth_below.argtypes = [P, P, i64, u64, u64]
            lib.synth_below.restype = None
            _lib = lib
    return _lib


def _threads() -> int:
    return max(1, min(64, os.cpu_count() or 1))


def _p(a):
    return None if a is None else a.ctypes.data


# ---- primitive draws ---------------------------------------------------------

def token_rows(n: int, stride: int, seed: int, lens: np.ndarray | None = None,
               vocab: int = VOCAB, ordinal0: int = 0, stream: int = _S_TOKENS) -> np.ndarray:
    """Pairwise-distinct token rows (the first two tokens spell the ordinal)."""
    out = np.empty((n, stride), dtype=np.int32)
    if lens is not None:
        lens = np.ascontiguousarray(lens, dtype=np.int32)
    if n:
        _load().synth_token_rows(_p(out), n, stride, _p(lens), vocab, seed, stream,
                                 ordinal0, _threads())
    return out


def uniform_ints(n: int, lo: int, hi: int, seed: int, stream: int = _S_LENS) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    if n:
        _load().synth_uniform_ints(_p(out), n, lo, hi, seed, stream)
    return out


def unit_rows(n: int, d: int, seed: int, stream: int = _S_VECTORS,
              counter0: int = 0) -> np.ndarray:
    """n unit-norm bf16 rows (uint16 bit patterns), Gaussian then normalised."""
    out = np.empty((n, d), dtype=np.uint16)
    if n:
        _load().synth_unit_rows_bf16(_p(out), n, d, seed, stream, counter0, _threads())
    return out


def choose_distinct(n: int, m: int, seed: int, stream: int) -> np.ndarray:
    out = np.empty(max(m, 1), dtype=np.int64)
    rc = _load().synth_choose_distinct(_p(out), n, m, seed, stream)
    if rc:
        raise ValueError("choose_distinct failed (%d)" % rc)
    return out[:m].copy()


def below(bounds: np.ndarray, seed: int, stream: int) -> np.ndarray:
    bounds = np.ascontiguousarray(bounds, dtype=np.int64)
    out = np.empty(bounds.shape[0], dtype=np.int64)
    if bounds.size:
        _load().synth_below(_p(out), _p(bounds), bounds.shape[0], seed, stream)
    return out


def zipf_ranks(n: int, pool: int, s: float, seed: int, stream: int = _S_ZIPF) -> np.ndarray:
    out = np.empty(n, dtype=np.int64)
    rc = _load().synth_zipf_ranks(_p(out), n, pool, s, seed, stream)
    if rc:
        raise MemoryError("zipf_ranks")
    return out


# ---- planted duplicates --------------------------------------------------------

def copy_plan(n: int, n_copies: int, seed: int, block: int | None = None,
              stream_pos: int = _S_COPYPOS, stream_src: int = _S_COPYSRC) -> np.ndarray:
    """Ground-truth roots for a row array with exactly n_copies copy rows.

    Copy positions are distinct and drawn uniformly among eligible rows.  A
    copy row takes the content of a uniformly drawn earlier row: any earlier
    row when ``block`` is None, otherwise a row of an earlier workflow
    (workflow w owns rows [w*block, (w+1)*block)), so the copy crosses
    workflows.  Returns root[i] = the non-copy row whose content row i holds
    (root[i] == i for non-copy rows).
    """
    first = 1 if block is None else block
    eligible = max(0, n - first)
    if n_copies > eligible:
        raise ValueError("more copies than eligible rows")
    pos = np.sort(choose_distinct(eligible, n_copies, seed, stream_pos) + first)
    bound = pos if block is None else (pos // block) * block
    src = below(bound, seed, stream_src)
    root = np.arange(n, dtype=np.int64)
    for p, s in zip(pos.tolist(), src.tolist()):   # ascending: sources are final
        root[p] = root[s]
    return root


def chunks_with_copies(n: int, stride: int, copy_frac: float, seed: int,
                       block: int | None = None):
    """Token rows where exactly round(copy_frac*n) rows copy earlier rows."""
    n_copies = int(round(copy_frac * n))
    tokens = token_rows(n, stride, seed)
    root = copy_plan(n, n_copies, seed, block)
    cp = np.nonzero(root != np.arange(n))[0]
    tokens[cp] = tokens[root[cp]]
    return tokens, root


def chunks_zipf(n: int, stride: int, pool: int, s: float, len_lo: int, len_hi: int,
                seed: int):
    """Rows drawn i.i.d. from a pool of distinct rows with Zipf(s) reuse.

    Pool row lengths are uniform in [len_lo, len_hi]; rows are zero-padded to
    stride.  The Zipf rank is mapped to a pool row through a seeded
    permutation.  Returns (tokens, lens, pool_index_per_row).
    """
    pool_lens = uniform_ints(pool, len_lo, len_hi, seed, _S_LENS)
    pool_tokens = token_rows(pool, stride, seed, lens=pool_lens)
    perm = choose_distinct(pool, pool, seed, _S_PERM)
    pidx = perm[zipf_ranks(n, pool, s, seed)]
    return pool_tokens[pidx], pool_lens[pidx].copy(), pidx


def queries_with_copies(n: int, d: int, dup_frac: float, seed: int,
                        block: int | None = None, stream: int = _S_VECTORS + 100):
    """Unit-norm bf16 query vectors; exactly round(dup_frac*n) are copies."""
    n_copies = int(round(dup_frac * n))
    q = unit_rows(n, d, seed, stream=stream)
    root = copy_plan(n, n_copies, seed, block, stream_pos=_S_COPYPOS + 100,
                     stream_src=_S_COPYSRC + 100)
    cp = np.nonzero(root != np.arange(n))[0]
    q[cp] = q[root[cp]]
    return q, root


def clustered_corpus(N: int, d: int, n_clusters: int, members: int, sigma: float,
                     seed: int):
    """Unit-norm Gaussian corpus with planted near-duplicate clusters.

    Cluster c has a unit-norm centre; its members sit at distinct seeded
    positions and equal normalise(centre + (sigma/sqrt(d)) * z), z ~ N(0, I),
    so the noise vector has norm about sigma.  Returns (corpus, centres,
    member_positions[n_clusters, members]).
    """
    centres = np.empty((n_clusters, d), dtype=np.float64)
    _load().synth_unit_centres_f64(_p(centres), n_clusters, d, seed, _S_CENTRES)
    pos = choose_distinct(N, n_clusters * members, seed, _S_MEMBERS).reshape(n_clusters,
                                                                            members)
    centre_of_row = np.full(N, -1, dtype=np.int64)
    centre_of_row[pos.reshape(-1)] = np.repeat(np.arange(n_clusters), members)
    out = np.empty((N, d), dtype=np.uint16)
    _load().synth_rows_near_bf16(_p(out), N, d, _p(centres), _p(centre_of_row),
                                 sigma / np.sqrt(d), seed, _S_VECTORS, 0, _threads())
    return out, centres, pos


def queries_near_centres(nq: int, centres: np.ndarray, sigma: float, seed: int):
    """Queries normalise(centre[c] + (sigma/sqrt(d)) z), c uniform per query."""
    n_clusters, d = centres.shape
    cl = below(np.full(nq, n_clusters, dtype=np.int64), seed, _S_QCLUSTER)
    out = np.empty((nq, d), dtype=np.uint16)
    centres = np.ascontiguousarray(centres, dtype=np.float64)
    _load().synth_rows_near_bf16(_p(out), nq, d, _p(centres), _p(cl), sigma / np.sqrt(d),
                                 seed, _S_QNOISE, 0, _threads())
    return out, cl


def partition_of(root: np.ndarray):
    """(unique_idx, inverse) induced by a ground-truth root array: groups are
    the rows sharing a root, listed by first occurrence.  Plain bookkeeping on
    planted labels, used to pin the oracle."""
    root = np.asarray(root)
    n = root.shape[0]
    first = {}
    uidx, inv = [], np.empty(n, dtype=np.int32)
    for i, r in enumerate(root.tolist()):
        if r not in first:
            first[r] = len(uidx)
            uidx.append(i)
        inv[i] = first[r]
    return np.asarray(uidx, dtype=np.int32), inv
