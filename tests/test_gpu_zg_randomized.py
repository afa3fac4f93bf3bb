"""Randomized parity sweeps over the shapes the §8(f) entry points accept:
seeded draws of batch sizes, dimensions, duplicate patterns, k values and
group structures, each checked against the oracle (bit-exact where the
result is integer or exactly representable)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
import synth
from hs_testutil import check_topk, to_dev

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed", range(12))
def test_merge_queries_random_shapes(seed):
    rng = np.random.default_rng(1000 + seed)
    n = int(rng.integers(1, hs.HS_MERGE_QUERIES_MAX + 1))
    d = int(rng.choice([8, 16, 24, 64, 200, 768, 1024]))
    dup = float(rng.choice([0.0, 0.1, 0.5, 0.9]))
    q, _ = synth.queries_with_copies(n, d, dup, seed + 50)
    if rng.random() < 0.3:                      # rows differing in one word only
        q[n // 2] = q[0]
        q[n // 2, -1] ^= 1
    fp, nu, uidx, inv, uq = hs.hs_merge_queries(to_dev(q))
    hs.hs_get_device_error()
    n_u = int(nu.item())
    ou, oi = oracle.unique_inverse(q.view(np.int32))
    assert (fp.cpu().numpy().view(np.uint64) == oracle.fingerprint(q.view(np.int32))).all()
    assert n_u == len(ou) and (uidx.cpu().numpy()[:n_u] == ou).all()
    assert (inv.cpu().numpy() == oi).all()
    assert (uq.view(torch.int16).cpu().numpy().view(np.uint16)[:n_u] == q[ou]).all()


@pytest.mark.parametrize("seed", range(8))
def test_segment_sum_random_groups(seed):
    rng = np.random.default_rng(2000 + seed)
    n = int(rng.integers(1, 200_000))
    G = int(rng.integers(1, max(2, n // int(rng.choice([1, 3, 50, 5000])))))
    skew = float(rng.choice([0.0, 1.1, 2.0]))
    if skew:
        p = np.arange(1, G + 1, dtype=np.float64) ** -skew
        inv = rng.choice(G, n, p=p / p.sum()).astype(np.int32)
    else:
        inv = rng.integers(0, G, n).astype(np.int32)
    inv = rng.permutation(G).astype(np.int32)[inv]          # hot groups anywhere
    phi = rng.integers(-(1 << 24), 1 << 24, n).astype(np.float64)
    out = hs.hs_segment_sum(to_dev(phi), to_dev(inv), G)
    hs.hs_get_device_error()
    assert (out.cpu().numpy() == oracle.segment_sum(phi, inv, G)).all()


@pytest.mark.parametrize("seed", range(6))
def test_rerank_random_shapes(seed):
    rng = np.random.default_rng(3000 + seed)
    Q = int(rng.integers(1, 400))
    N = int(rng.integers(64, 20000))
    d = int(rng.choice([8, 64, 256, 1024, 2048]))
    k1 = int(rng.integers(1, min(32, N) + 1))
    k2 = int(rng.integers(1, k1 + 1))
    rc = synth.unit_rows(N, d, seed + 70)
    rq = synth.unit_rows(Q, d, seed + 71)
    cand = np.stack([rng.choice(N, k1, replace=False) for _ in range(Q)]).astype(np.int32)
    s, i = hs.hs_rerank_topk(to_dev(rq), to_dev(rc), to_dev(cand), k2)
    hs.hs_get_device_error()
    s, i = s.cpu().numpy(), i.cpu().numpy()
    os_, oi = oracle.rerank(rq, rc, cand, min(k2 + 1, k1))
    for q in range(Q):
        exact = oracle.pair_scores(rq, rc, np.full(k2, q), i[q])
        check_topk(s[q], i[q], os_[q], oi[q], exact, N, k2)


@pytest.mark.parametrize("seed", range(4))
def test_cache_random_streams(seed):
    rng = np.random.default_rng(4000 + seed)
    d = int(rng.choice([64, 256, 768]))
    k = int(rng.integers(1, 33))
    B = int(rng.integers(5, 600))
    pool = synth.unit_rows(int(rng.integers(20, 2000)), d, seed + 90)
    corpus = to_dev(synth.unit_rows(int(rng.integers(k, 30000)), d, seed + 91))
    cap = int(rng.choice([8, 64, 100000]))
    cached = hs.EmbedRetrieveStage(corpus, k, max_queries=B, cache_capacity=cap)
    plain = hs.EmbedRetrieveStage(corpus, k, max_queries=B)
    total = 0
    for _ in range(5):
        qb = to_dev(pool[rng.integers(0, len(pool), B)])
        s, i, nu = cached.retrieve(qb)
        s2, i2, _ = plain.retrieve(qb)
        hs.hs_get_device_error()
        assert torch.equal(s.cpu(), s2.cpu()) and torch.equal(i.cpu(), i2.cpu())
        total += int(nu.item())
    hits, misses = cached.cache_stats()
    assert hits + misses == total
