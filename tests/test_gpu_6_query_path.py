"""The fused query path against the oracle.

hs_merge_queries: fingerprint (Section 3.3, Eq. 2), exact merge of equal
query rows (Section 3.3 (I)) and the gather of the unique rows in one
launch — fingerprints, unique sets and inverse maps bit-exact, gathered rows
byte-exact.  hs_retrieve_topk_fanout: the merged query's results written to
every row merged into it (Section 3.3 (I), Appendix A.2) — bit-identical to
retrieval followed by two scatters, and within the top-k parity rule of the
oracle."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
import synth
from hs_testutil import check_topk, to_dev

pytestmark = pytest.mark.gpu


def query_batch(n, d, dup_frac, seed):
    q, _ = synth.queries_with_copies(n, d, dup_frac, seed)
    return q


def merged(q, seed_state=hs.HS_FNV64_OFFSET_BASIS, fp_in=None, fill=None):
    n, d = q.shape
    out = None
    if fill is not None:
        dev = torch.device("cuda")
        out = (torch.empty(max(n, 1), dtype=torch.int64, device=dev),
               torch.empty(1, dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev),
               torch.full((max(n, 1), d), fill, dtype=torch.int16, device=dev).view(torch.bfloat16))
    fp, nu, uidx, inv, uq = hs.hs_merge_queries(
        to_dev(q), seed_state, None if fp_in is None else to_dev(fp_in.astype(np.uint64)), out=out)
    hs.hs_get_device_error()
    n_u = int(nu.item())
    return (fp.cpu().numpy().view(np.uint64), n_u, uidx.cpu().numpy(), inv.cpu().numpy(),
            uq.view(torch.int16).cpu().numpy().view(np.uint16))


def check_merge(q, seed_state=hs.HS_FNV64_OFFSET_BASIS, fp_in=None):
    n = q.shape[0]
    fp, n_u, uidx, inv, uq = merged(q, seed_state, fp_in, fill=0x7F7F)
    words = q.view(np.int32)
    if fp_in is None:
        assert (fp == oracle.fingerprint(words, seed=seed_state)).all()
    else:
        assert (fp == fp_in.astype(np.uint64)).all()
    ou, oi = oracle.unique_inverse(words)
    assert n_u == len(ou)
    assert (uidx[:n_u] == ou).all() and (uidx[n_u:] == 0).all()
    assert (inv == oi).all()
    assert (uq[:n_u] == q[ou]).all()
    assert (uq[n_u:] == 0x7F7F).all(), "rows past the unique count must stay untouched"
    return n_u


@pytest.mark.parametrize("n", [1, 2, 8, 31, 32, 33, 64, 100, 200, 255, 256])
def test_merge_queries_matches_oracle(n):
    q = query_batch(n, 768, 0.2, seed=n)
    assert check_merge(q) == n - int(round(0.2 * n))


@pytest.mark.parametrize("n,d", [(5, 8), (70, 40), (33, 1032), (256, 64), (3, 4096)])
def test_merge_queries_dims(n, d):
    check_merge(query_batch(n, d, 0.3, seed=d))


def test_merge_queries_degenerate():
    base = query_batch(1, 768, 0.0, seed=7)
    assert check_merge(np.repeat(base, 256, axis=0)) == 1          # every row equal
    assert check_merge(query_batch(256, 768, 0.0, seed=8)) == 256   # every row distinct
    zero = np.zeros((40, 16), np.uint16)
    zero[20:] = 1
    assert check_merge(zero) == 2
    assert check_merge(query_batch(64, 768, 0.5, seed=9), seed_state=0x1234567890ABCDEF) == 32


def test_merge_queries_empty_and_limits():
    dev = torch.device("cuda")
    nu = torch.full((1,), 99, dtype=torch.int32, device=dev)
    q = torch.zeros((0, 768), dtype=torch.bfloat16, device=dev)
    out = (torch.empty(1, dtype=torch.int64, device=dev), nu,
           torch.empty(1, dtype=torch.int32, device=dev),
           torch.empty(1, dtype=torch.int32, device=dev),
           torch.empty((1, 768), dtype=torch.bfloat16, device=dev))
    hs.hs_merge_queries(q, out=out)
    hs.hs_get_device_error()
    assert int(nu.item()) == 0
    with pytest.raises(hs.HsError):
        hs.hs_merge_queries(torch.zeros((hs.HS_MERGE_QUERIES_MAX + 1, 768),
                                        dtype=torch.bfloat16, device=dev))
    with pytest.raises(hs.HsError):
        hs.hs_merge_queries(torch.zeros((4, 12), dtype=torch.bfloat16, device=dev))


def test_merge_queries_collisions_resolved_exactly():
    """Fingerprints supplied with planted collisions: rows with different
    contents share a fingerprint; the merge must still follow contents."""
    rng = np.random.default_rng(3)
    classes = rng.integers(0, 40, size=200)
    table = query_batch(40, 768, 0.0, seed=11)
    q = table[classes]
    for fp_in in (classes % 3, np.zeros(200, np.int64), np.where(classes % 2 == 0, -1, classes),
                  classes.astype(np.int64)):
        fp_in = np.asarray(fp_in).astype(np.int64).view(np.uint64)
        assert check_merge(q, fp_in=fp_in) == len(np.unique(classes))


def test_merge_queries_matches_separate_calls():
    q = query_batch(96, 768, 0.25, seed=21)
    fp, n_u, uidx, inv, uq = merged(q)
    t = to_dev(q)
    fp2 = hs.hs_fingerprint(t.view(torch.int32))
    nu2, uidx2, inv2 = hs.hs_unique_inverse(fp2, t.view(torch.int32))
    uq2 = hs.hs_scatter_results(t, uidx2)
    hs.hs_get_device_error()
    n2 = int(nu2.item())
    assert n_u == n2 and (fp == fp2.cpu().numpy().view(np.uint64)).all()
    assert (uidx == uidx2.cpu().numpy()).all() and (inv == inv2.cpu().numpy()).all()
    assert (uq[:n_u] == uq2.view(torch.int16).cpu().numpy().view(np.uint16)[:n_u]).all()


def fanout_case(Q_max, n_real, n_out, N, d, k, seed):
    corpus = synth.unit_rows(N, d, seed)
    queries = synth.unit_rows(Q_max, d, seed + 1)
    rng = np.random.default_rng(seed)
    inv = rng.integers(0, n_real, size=n_out).astype(np.int32)
    qd, cd = to_dev(queries), to_dev(corpus)
    cnt = to_dev(np.array([n_real], np.int32))
    ws = torch.empty(hs.hs_retrieve_topk_workspace(Q_max, N, d, k), dtype=torch.uint8,
                     device="cuda")
    s, i = hs.hs_retrieve_topk_fanout(qd, cnt, to_dev(inv), cd, k, workspace=ws)
    hs.hs_get_device_error()
    s, i = s.cpu().numpy(), i.cpu().numpy()
    # the same kernels followed by two scatters
    s_u, i_u = hs.hs_retrieve_topk_n(qd, cnt, cd, k, workspace=ws)
    s2 = hs.hs_scatter_results(s_u, to_dev(inv)).cpu().numpy()
    i2 = hs.hs_scatter_results(i_u, to_dev(inv)).cpu().numpy()
    hs.hs_get_device_error()
    assert (s == s2).all() and (i == i2).all()
    # oracle parity on the distinct queries referenced
    used = np.unique(inv)[:24]
    os_, oi_ = oracle.topk(queries[used], corpus, min(k + 1, N))
    for r, qi in enumerate(used):
        o = int(np.nonzero(inv == qi)[0][0])
        exact = oracle.pair_scores(queries, corpus, np.full(k, qi), i[o])
        check_topk(s[o], i[o], os_[r], oi_[r], exact, N, k)
        rows = np.nonzero(inv == qi)[0]
        assert (s[rows] == s[o]).all() and (i[rows] == i[o]).all()


@pytest.mark.parametrize("Q_max,n_real,n_out,N,d,k", [
    (12, 9, 20, 5000, 768, 10),        # small-batch kernel
    (1, 1, 3, 300, 64, 5),
    (300, 250, 400, 20000, 768, 10),   # CTA-pair kernel, register lists
    (64, 64, 70, 9000, 256, 32),
    (40, 33, 50, 70000, 128, 100),     # large k over >= 64 tiles: the optimistic pass
    (20, 20, 21, 3000, 128, 300),      # large k, one pass
])
def test_fanout_matches_scatter_and_oracle(Q_max, n_real, n_out, N, d, k):
    fanout_case(Q_max, n_real, n_out, N, d, k, seed=Q_max + N)


def test_fanout_rejects_bad_map_entries():
    corpus = to_dev(synth.unit_rows(1000, 64, 1))
    queries = to_dev(synth.unit_rows(4, 64, 2))
    inv = to_dev(np.array([0, 3, 4, -1, 2], np.int32))
    s = torch.full((5, 7), 5.0, device="cuda")
    i = torch.full((5, 7), -7, dtype=torch.int32, device="cuda")
    hs.hs_retrieve_topk_fanout(queries, None, inv, corpus, 7, out=(s, i))
    with pytest.raises(hs.HsError):
        hs.hs_get_device_error()
    s, i = s.cpu().numpy(), i.cpu().numpy()
    assert (s[[2, 3]] == 5.0).all() and (i[[2, 3]] == -7).all()
    assert (i[[0, 1, 4]] >= 0).all()
    # n_out = 0 enqueues nothing
    hs.hs_retrieve_topk_fanout(queries, None, inv[:0], corpus, 7)
    hs.hs_get_device_error()


def test_fanout_large_k_flagged_blocks_with_device_count():
    """k > 32 with the exact fallback taken (a query whose top-k crowds into
    one list's rows), a device-side query count and a fan-out map."""
    N, d, k, Qmax, n_real = 64 * 256 * 2, 64, 100, 200, 150
    corpus = synth.unit_rows(N, d, 61)
    q = synth.unit_rows(Qmax, d, 62)
    rng = np.random.default_rng(63)
    base = (q[3].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    rows = base / np.linalg.norm(base) + rng.standard_normal((180, d)) * 0.02
    rows /= np.linalg.norm(rows, axis=1, keepdims=True)
    corpus[5000:5180] = (rows.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    inv = rng.integers(0, n_real, size=260).astype(np.int32)
    inv[:4] = 3
    cnt = to_dev(np.array([n_real], np.int32))
    s, i = hs.hs_retrieve_topk_fanout(to_dev(q), cnt, to_dev(inv), to_dev(corpus), k)
    hs.hs_get_device_error()
    s, i = s.cpu().numpy(), i.cpu().numpy()
    used = np.unique(np.concatenate([[3], inv[::29]]))
    os_, oi = oracle.topk(q[used], corpus, k + 1)
    for r, qi in enumerate(used):
        o = int(np.nonzero(inv == qi)[0][0])
        exact = oracle.pair_scores(q, corpus, np.full(k, qi), i[o])
        check_topk(s[o], i[o], os_[r], oi[r], exact, N, k)
        rows_o = np.nonzero(inv == qi)[0]
        assert (s[rows_o] == s[o]).all() and (i[rows_o] == i[o]).all()
