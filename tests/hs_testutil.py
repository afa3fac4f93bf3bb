"""Shared helpers for the parity tests: host<->device marshalling and the
top-k parity rule."""
from __future__ import annotations

import numpy as np

TOL = 2e-2          # score tolerance for unit-norm bf16 rows with fp32 sums
STRICT = 1e-3       # bound derived from fp32 accumulation error (d <= 1024)
ORDER_EPS = 1e-5    # oracle scores closer than this may swap order


def to_dev(a: np.ndarray):
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)
    if a.dtype == np.uint64:
        return torch.from_numpy(a.view(np.int64)).cuda()
    return torch.from_numpy(a).cuda()


def fp_host(t) -> np.ndarray:
    return t.cpu().numpy().view(np.uint64)


def bf16_f64(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint32) << 16).view(np.float32).astype(np.float64)


def check_topk(gs, gi, os_, oi, exact_g, N, k, tol=TOL, strict=STRICT):
    """Parity of one query's GPU top-k (scores gs, ids gi) with the oracle.

    os_, oi: the oracle's first min(k+1, N) (score, id) pairs in order;
    exact_g: the oracle's fp64 scores of the GPU ids.
    (i)   ids distinct and in range, scores non-increasing;
    (ii)  |gs_j - exact(g_j)| <= tol (and <= strict);
    (iii) if the oracle's k-th and (k+1)-th scores differ by >= tol, the id
          sets are equal and the order matches except between oracle scores
          closer than ORDER_EPS;
    (iv)  otherwise every oracle id whose score exceeds s_k + tol is returned
          and every returned id scores >= s_k - tol.
    Returns the max score error."""
    gs = np.asarray(gs, dtype=np.float64)
    gi = np.asarray(gi)
    assert len(set(gi.tolist())) == k, "duplicate ids"
    assert gi.min() >= 0 and gi.max() < N, "id out of range"
    assert (np.diff(gs) <= 0).all(), "scores not non-increasing"
    err = np.abs(gs - exact_g).max()
    assert err <= tol, "score error %g > %g" % (err, tol)
    assert err <= strict, "score error %g > %g (fp32 accumulation bound)" % (err, strict)
    s_k = os_[k - 1]
    s_next = os_[k] if len(os_) > k else -np.inf
    if s_k - s_next >= tol:
        assert set(gi.tolist()) == set(oi[:k].tolist()), "id sets differ"
        pos = {int(j): r for r, j in enumerate(oi[:k].tolist())}
        for a in range(k - 1):
            ra, rb = pos[int(gi[a])], pos[int(gi[a + 1])]
            if ra > rb:
                assert abs(os_[ra] - os_[rb]) < ORDER_EPS, "order differs"
    else:
        must = [int(j) for j, s in zip(oi[:k], os_[:k]) if s > s_k + tol]
        assert set(must) <= set(gi.tolist()), "a clearly-better oracle id is missing"
        assert (exact_g >= s_k - tol).all(), "a returned id is clearly worse than the k-th"
    return err


_TOPK_MEMO: dict = {}


def oracle_topk_memo(tag: str, Q: np.ndarray, C: np.ndarray, k: int):
    """oracle.topk(Q, C, k), remembered for the rest of the test session.

    The full-size parity tests of several modules need the oracle's top-k of
    the same merged queries against the same corpus (minutes of fp64 work
    on the host); the key is the caller's name for the corpus, the corpus
    shape, k and a digest of the query rows."""
    import hashlib

    import oracle
    key = (tag, C.shape, int(k), hashlib.sha1(np.ascontiguousarray(Q).tobytes()).hexdigest())
    if key not in _TOPK_MEMO:
        _TOPK_MEMO[key] = oracle.topk(Q, C, k)
    return _TOPK_MEMO[key]


def check_rows(Q, C, k, gs, gi, rows, tag=None):
    """check_topk on each listed query row of a GPU result (gs, gi indexed
    like Q); the oracle's first k + 1 entries come from oracle.topk (through
    oracle_topk_memo when a corpus tag is given).  Returns the max score
    error."""
    import oracle
    rows = np.asarray(rows, dtype=np.int64)
    N = C.shape[0]
    kk = min(k + 1, N)
    Qs = np.ascontiguousarray(Q[rows])
    os_, oi = oracle_topk_memo(tag, Qs, C, kk) if tag else oracle.topk(Qs, C, kk)
    exact = oracle.pair_scores(Q, C, np.repeat(rows, k), gi[rows].reshape(-1)).reshape(-1, k)
    worst = 0.0
    for r, q in enumerate(rows):
        worst = max(worst, check_topk(gs[q], gi[q], os_[r], oi[r], exact[r], N, k))
    return worst
