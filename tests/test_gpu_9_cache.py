"""The result cache (asynchronous cache reuse across batches, Section 3.3,
"Dynamic Fusion and Reuse Mechanism" (II)) against the oracle: with room for
every query, a merged query hits exactly when an equal query was retrieved
in an earlier batch (the oracle's reuse model); hit or miss, every result
is bit-identical to retrieving the query afresh; fingerprint collisions
never return another query's result."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
import synth
from hs_testutil import check_rows, to_dev

pytestmark = pytest.mark.gpu


def zipf_batches(pool, n_batches, B, seed):
    rng = np.random.default_rng(seed)
    ranks = np.arange(1, len(pool) + 1, dtype=np.float64)
    p = ranks ** -1.1
    p /= p.sum()
    return [pool[rng.choice(len(pool), B, p=p)] for _ in range(n_batches)]


def miss_flags(stage, Q):
    n_miss = int(stage.miss[1].item())
    flags = np.zeros(Q, bool)
    flags[stage.miss[0][:n_miss].cpu().numpy()] = True
    return flags


@pytest.mark.parametrize("B", [40, 700])
def test_hits_follow_the_reuse_model_and_results_match(B):
    """B = 40 takes the fused query path; B = 700 the separate calls."""
    pool = synth.unit_rows(300, 256, 1)
    corpus_h = synth.unit_rows(20000, 256, 2)
    corpus = to_dev(corpus_h)
    batches = zipf_batches(pool, 6, B, seed=B)
    cached = hs.EmbedRetrieveStage(corpus, 10, max_queries=B, cache_capacity=4096)
    plain = hs.EmbedRetrieveStage(corpus, 10, max_queries=B)
    uniq_rows = []
    for qb in batches:
        s, i, nu = cached.retrieve(to_dev(qb))
        n_u = int(nu.item())
        flags = miss_flags(cached, n_u)
        s2, i2, _ = plain.retrieve(to_dev(qb))
        hs.hs_get_device_error()
        assert torch.equal(s.cpu(), s2.cpu()) and torch.equal(i.cpu(), i2.cpu())
        uidx, _ = oracle.unique_inverse(qb.view(np.int32))
        # hit rows (from the cache) and miss rows (retrieved now) alike
        # against the oracle
        check_rows(qb, corpus_h, 10, s.cpu().numpy(), i.cpu().numpy(), uidx)
        uniq_rows.append((qb[uidx], ~flags))
    model = oracle.cache_reuse([u for u, _ in uniq_rows])
    for (_, hit), want in zip(uniq_rows, model):
        assert (hit == want).all()
    hits, misses = cached.cache_stats()
    assert hits == sum(int(m.sum()) for m in model)
    assert misses == sum(int((~m).sum()) for m in model)


def test_small_cache_evicts_but_stays_correct():
    pool = synth.unit_rows(400, 128, 3)
    corpus_h = synth.unit_rows(5000, 128, 4)
    corpus = to_dev(corpus_h)
    batches = zipf_batches(pool, 8, 200, seed=5)
    cached = hs.EmbedRetrieveStage(corpus, 8, max_queries=200, cache_capacity=16)
    plain = hs.EmbedRetrieveStage(corpus, 8, max_queries=200)
    total_unique = 0
    for qb in batches:
        s, i, nu = cached.retrieve(to_dev(qb))
        s2, i2, _ = plain.retrieve(to_dev(qb))
        hs.hs_get_device_error()
        assert torch.equal(s.cpu(), s2.cpu()) and torch.equal(i.cpu(), i2.cpu())
        check_rows(qb, corpus_h, 8, s.cpu().numpy(), i.cpu().numpy(),
                   oracle.unique_inverse(qb.view(np.int32))[0])
        total_unique += int(nu.item())
    hits, misses = cached.cache_stats()
    assert hits + misses == total_unique
    unbounded = oracle.cache_reuse([qb[oracle.unique_inverse(qb.view(np.int32))[0]]
                                    for qb in batches])
    assert 0 < hits <= sum(int(m.sum()) for m in unbounded)


def test_fingerprint_collisions_never_share_results():
    """All queries given the same key: every distinct vector is its own
    entry (up to the set's 8 ways), and each lookup returns its own top-k."""
    d, k = 64, 5
    corpus_h = synth.unit_rows(2000, d, 6)
    corpus = to_dev(corpus_h)
    q = synth.unit_rows(6, d, 7)
    cache = hs.ResultCache(64, d, k)
    fp = torch.zeros(6, dtype=torch.int64, device="cuda")
    qd = to_dev(q)
    want_s, want_i = hs.hs_retrieve_topk(qd, corpus, k)
    check_rows(q, corpus_h, k, want_s.cpu().numpy(), want_i.cpu().numpy(), np.arange(6))
    for _ in range(2):
        out, miss = hs.hs_cache_lookup(cache, qd, fp)
        ms, mi = hs.hs_retrieve_topk_n(miss[2], miss[1], corpus, k)
        hs.hs_cache_insert(cache, miss, fp, ms, mi, out)
        hs.hs_get_device_error()
        assert torch.equal(out[0].cpu(), want_s.cpu()) and torch.equal(out[1].cpu(), want_i.cpu())
    assert hs.hs_cache_stats(cache) == (6, 6)       # second pass: six hits


def test_uninitialised_cache_is_rejected():
    cache = hs.ResultCache(16, 64, 4)
    cache.mem.zero_()                                # header wiped
    q = to_dev(synth.unit_rows(3, 64, 8))
    hs.hs_cache_lookup(cache, q, torch.zeros(3, dtype=torch.int64, device="cuda"))
    with pytest.raises(hs.HsError):
        hs.hs_get_device_error()


def test_two_streams_share_a_cache_without_torn_results():
    """Two streams look up and insert into one small cache at the same time,
    so inserts on one stream evict entries that lookups on the other may be
    reading.  Every row, hit or miss, must be exactly its own query's top-k."""
    d, k, pool_n, B = 256, 10, 48, 12
    corpus_h = synth.unit_rows(400000, d, 21)
    pool_h = synth.unit_rows(pool_n, d, 22)
    corpus = to_dev(corpus_h)
    pd = to_dev(pool_h)
    fp_all = hs.hs_fingerprint(pd.view(torch.int32))
    want_s = torch.empty((pool_n, k), dtype=torch.float32, device="cuda")
    want_i = torch.empty((pool_n, k), dtype=torch.int32, device="cuda")
    for c0 in range(0, pool_n, B):                   # the kernel the misses take (<= 16 rows)
        s, i = hs.hs_retrieve_topk(pd[c0:c0 + B], corpus, k)
        want_s[c0:c0 + B], want_i[c0:c0 + B] = s, i
    check_rows(pool_h, corpus_h, k, want_s.cpu().numpy(), want_i.cpu().numpy(),
               np.arange(pool_n))
    rng = np.random.default_rng(23)
    sels = torch.from_numpy(np.stack([rng.choice(pool_n, B, replace=False)
                                      for _ in range(120)])).to("cuda")
    torch.cuda.synchronize()
    cache = hs.ResultCache(16, d, k)                 # two sets of eight ways: steady eviction
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    for st in streams:
        st.wait_stream(torch.cuda.current_stream())
    outs = []
    for it in range(sels.shape[0]):
        st = streams[it % 2]
        with torch.cuda.stream(st):
            sel = sels[it]
            q, f = pd[sel], fp_all[sel]
            out, miss = hs.hs_cache_lookup(cache, q, f)
            ms, mi = hs.hs_retrieve_topk_n(miss[2], miss[1], corpus, k)
            hs.hs_cache_insert(cache, miss, f, ms, mi, out)
            outs.append((it, out))
    torch.cuda.synchronize()
    hs.hs_get_device_error()
    for it, (s, i) in outs:
        sel = sels[it]
        assert torch.equal(i, want_i[sel]), "batch %d returned another query's ids" % it
        assert torch.equal(s, want_s[sel]), "batch %d returned another query's scores" % it
    hits, misses = hs.hs_cache_stats(cache)
    assert hits + misses == sels.numel() and hits > 0 and misses > 0
