"""The §8(f) rows at the benchmark's full sizes, in the configuration
bench.py times: the fused query path on batch-sweep batches against the
2,097,152-row corpus, the result cache on a stream of RAG-mix batches, and
the rerank of RAG-mix candidates against 1,048,576 rerank vectors, each on
sampled outputs the oracle computes one by one."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
import synth
from hs_testutil import check_rows, check_topk, to_dev
from synth import configs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rag():
    w = configs.build_retrieval_mix(configs.RAG_MIX)
    return w, to_dev(w["corpus"])


def test_fused_query_path_batch_sweep_sizes():
    C = configs.sweep_corpus()
    corpus = to_dev(C)
    stage = hs.EmbedRetrieveStage(corpus, configs.BATCH_SWEEP["k"], max_queries=256)
    for B in (1, 64, 256):
        q = configs.build_sweep_batch(B, seed=77)["queries"]
        s, i, nu = stage.retrieve(to_dev(q))
        hs.hs_get_device_error()
        ou, oi = oracle.unique_inverse(q.view(np.int32))
        assert int(nu.item()) == len(ou)
        s, i = s.cpu().numpy(), i.cpu().numpy()
        assert (s == s[ou][oi]).all() and (i == i[ou][oi]).all()   # merged rows share results
        # every merged query of the batch against the oracle
        check_rows(q, C, configs.BATCH_SWEEP["k"], s, i, ou)


def test_cache_on_rag_mix_stream(rag):
    w, corpus = rag
    pool = synth.unit_rows(3000, corpus.shape[1], 41)
    rng = np.random.default_rng(42)
    p = np.arange(1, 3001, dtype=np.float64) ** -1.1
    p /= p.sum()
    cached = hs.EmbedRetrieveStage(corpus, w["k"], max_queries=2048, cache_capacity=65536)
    plain = hs.EmbedRetrieveStage(corpus, w["k"], max_queries=2048)
    checked = 0
    for b in range(3):
        qh = pool[rng.choice(3000, 2048, p=p)]
        qb = to_dev(qh)
        s, i, nu = cached.retrieve(qb)
        n_u = int(nu.item())
        n_miss = int(cached.miss[1].item())
        hit = np.ones(n_u, bool)
        hit[cached.miss[0][:n_miss].cpu().numpy()] = False
        s2, i2, _ = plain.retrieve(qb)
        hs.hs_get_device_error()
        assert torch.equal(s.cpu(), s2.cpu()) and torch.equal(i.cpu(), i2.cpu())
        # rows served from the cache against the oracle (a seeded sample)
        uidx, _ = oracle.unique_inverse(qh.view(np.int32))
        hit_rows = uidx[hit]
        if len(hit_rows):
            pick = np.random.default_rng(b).choice(len(hit_rows), min(96, len(hit_rows)),
                                                   replace=False)
            check_rows(qh, w["corpus"], w["k"], s.cpu().numpy(), i.cpu().numpy(),
                       hit_rows[pick])
            checked += len(pick)
    hits, misses = cached.cache_stats()
    assert hits > 0 and misses > 0 and checked > 0


def test_rerank_full_size_sampled(rag):
    w, corpus = rag
    N, d2 = corpus.shape[0], 1024
    g = torch.Generator(device="cuda").manual_seed(5)
    rc = torch.nn.functional.normalize(torch.randn(N, d2, device="cuda", generator=g), dim=1)
    rc = rc.to(torch.bfloat16)
    q = to_dev(w["queries"])
    rq = torch.nn.functional.normalize(torch.randn(q.shape[0], d2, device="cuda", generator=g),
                                       dim=1).to(torch.bfloat16)
    _, i12 = hs.hs_retrieve_topk(q, corpus, 12)
    s8, i8 = hs.hs_rerank_topk(rq, rc, i12, 8)
    hs.hs_get_device_error()
    rows = np.arange(0, q.shape[0], 97)
    cand = i12.cpu().numpy()[rows]
    used = np.unique(cand)
    rc_h = rc[torch.from_numpy(used).cuda()].view(torch.int16).cpu().numpy().view(np.uint16)
    rq_h = rq[torch.from_numpy(rows).cuda()].view(torch.int16).cpu().numpy().view(np.uint16)
    local = np.searchsorted(used, cand).astype(np.int32)      # candidates in the gathered rows
    os_, oi = oracle.rerank(rq_h, rc_h, local, 9)
    s8, i8 = s8.cpu().numpy()[rows], i8.cpu().numpy()[rows]
    for r in range(len(rows)):
        got = np.searchsorted(used, i8[r]).astype(np.int64)
        exact = oracle.pair_scores(rq_h, rc_h, np.full(8, r), got)
        check_topk(s8[r], got, os_[r], oi[r], exact, len(used), 8)
