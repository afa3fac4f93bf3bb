"""hs_rerank_topk against the oracle: the second stage of the RAG-with-rerank
workflow (Section 4.1, "Workloads": the initial top-12 chunks rescored, the
top-8 kept).  Scores within the fp32 accumulation bound of the exact fp64
inner products; ids identical except where the oracle's k2-th and
(k2+1)-th scores are closer than the tolerance."""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
import synth
from hs_testutil import check_topk, to_dev

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "rerank_hand.txt")


def run(rq, rc, cand, k2, count=None, inv=None):
    s, i = hs.hs_rerank_topk(to_dev(rq), to_dev(rc), to_dev(cand.astype(np.int32)), k2,
                             n_queries_dev=None if count is None else to_dev(np.array([count], np.int32)),
                             inverse=None if inv is None else to_dev(inv.astype(np.int32)))
    hs.hs_get_device_error()
    return s.cpu().numpy(), i.cpu().numpy()


def test_hand_example():
    from test_oracle_rerank import read_golden
    rq, rc, cand, expect = read_golden()
    pad = lambda a: np.concatenate([a, np.zeros((a.shape[0], 8 - a.shape[1]), np.uint16)], 1)
    s, i = run(pad(rq), pad(rc), cand, 3)          # zero columns up to the 16-byte row
    for q, (ids, sc) in expect.items():
        assert i[q].tolist() == ids and s[q].tolist() == sc


@pytest.mark.parametrize("Q,N,d,k1,k2", [(300, 5000, 1024, 12, 8), (33, 2000, 768, 32, 1),
                                         (7, 100, 8, 1, 1), (40, 3000, 4096, 20, 20),
                                         (64, 10000, 64, 16, 5)])
def test_matches_oracle(Q, N, d, k1, k2):
    rng = np.random.default_rng(Q + d)
    rc = synth.unit_rows(N, d, 1)
    rq = synth.unit_rows(Q, d, 2)
    cand = np.stack([rng.choice(N, k1, replace=False) for _ in range(Q)]).astype(np.int32)
    s, i = run(rq, rc, cand, k2)
    os_, oi = oracle.rerank(rq, rc, cand, min(k2 + 1, k1))
    for q in range(Q):
        exact = oracle.pair_scores(rq, rc, np.full(k2, q), i[q])
        check_topk(s[q], i[q], os_[q], oi[q], exact, N, k2)


def test_rerank_of_retrieval_candidates():
    """The two stages in sequence: retrieval top-12 ids as candidates of a
    rerank over different vectors, top-8 kept."""
    corpus = to_dev(synth.unit_rows(20000, 768, 3))
    rc = synth.unit_rows(20000, 1024, 4)
    q = synth.unit_rows(50, 768, 5)
    rq = synth.unit_rows(50, 1024, 6)
    _, ids12 = hs.hs_retrieve_topk(to_dev(q), corpus, 12)
    cand = ids12.cpu().numpy()
    s, i = run(rq, rc, cand, 8)
    os_, oi = oracle.rerank(rq, rc, cand, 9)
    for r in range(50):
        exact = oracle.pair_scores(rq, rc, np.full(8, r), i[r])
        check_topk(s[r], i[r], os_[r], oi[r], exact, 20000, 8)


def test_absent_duplicate_and_bad_candidates():
    rc = synth.unit_rows(100, 32, 7)
    rq = synth.unit_rows(3, 32, 8)
    cand = np.array([[5, -1, 7, -7, 9],      # three present, k2 = 4
                     [4, 4, 8, 12, 16],      # a duplicated id is scored twice
                     [-1, -2, -2147483648, -1, -1]], np.int32)   # any negative is absent
    s, i = run(rq, rc, cand, 4)
    os_, oi = oracle.rerank(rq, rc, cand, 4)
    assert (i == oi).all()
    assert np.isinf(s[0, 3]) and (s[2] == -np.inf).all() and (i[2] == -1).all()
    assert np.abs(s[np.isfinite(os_)] - os_[np.isfinite(os_)]).max() < 1e-5
    bad = cand.copy()
    bad[0, 0] = 100                          # >= n_corpus: error, treated as absent
    s2, i2 = hs.hs_rerank_topk(to_dev(rq), to_dev(rc), to_dev(bad), 4)
    with pytest.raises(hs.HsError):
        hs.hs_get_device_error()
    assert 100 not in i2.cpu().numpy()[0].tolist()


def test_fanout_and_device_count():
    rc = synth.unit_rows(3000, 256, 9)
    rq = synth.unit_rows(20, 256, 10)
    rng = np.random.default_rng(11)
    cand = np.stack([rng.choice(3000, 12, replace=False) for _ in range(20)]).astype(np.int32)
    inv = rng.integers(0, 15, size=45)
    s, i = run(rq, rc, cand, 8, count=15, inv=inv)
    s0, i0 = run(rq[:15], rc, cand[:15], 8)
    assert (s == s0[inv]).all() and (i == i0[inv]).all()


def test_stage_retrieve_rerank_matches_oracle():
    """The whole rerank workflow through the stage: merged retrieval of the
    top-12, rescoring of the 12 with the rerank vectors, top-8 kept and
    fanned out to every query (merged queries share their representative's
    rerank)."""
    q, root = synth.queries_with_copies(60, 768, 0.25, 12)
    rq = synth.unit_rows(60, 1024, 13)
    rq[np.nonzero(root != np.arange(60))[0]] = rq[root[root != np.arange(60)]]
    corpus = synth.unit_rows(30000, 768, 14)
    rc = synth.unit_rows(30000, 1024, 15)
    stage = hs.EmbedRetrieveStage(to_dev(corpus), 12, max_queries=60, rerank_corpus=to_dev(rc),
                                  rerank_k=8)
    s, i, nu = stage.retrieve_rerank(to_dev(q), to_dev(rq))
    hs.hs_get_device_error()
    s, i = s.cpu().numpy(), i.cpu().numpy()
    assert int(nu.item()) == 45
    _, cand = oracle.topk(q, corpus, 12)
    os_, oi = oracle.rerank(rq, rc, cand, 9)
    for r in range(60):
        exact = oracle.pair_scores(rq, rc, np.full(8, r), i[r])
        check_topk(s[r], i[r], os_[r], oi[r], exact, 30000, 8)
