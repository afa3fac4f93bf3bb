"""hs_retrieve_topk vs the oracle (the retrieval node shared by merged
queries, Section 4.1 "Workloads"; merged execution, Section 3.3).

Scores must be within 2e-2 of the oracle's fp64 scores (and within 1e-3, the
fp32-accumulation bound for unit-norm rows with d <= 1024); ids must match
except where the oracle's k-th and (k+1)-th scores are closer than 2e-2 (the
parity rule in hs_testutil.check_topk).  At full size the oracle checks every
merged query of the RAG mix and of the batch-sweep batches up to B = 512, and
a seeded sample of at least 256 queries of the batch of 4096 and of the large
corpus; the properties that hold at any size are checked on every query."""
import gc

import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
import synth
from hs_testutil import check_rows, check_topk, to_dev
from synth import configs

pytestmark = pytest.mark.gpu


def gpu_topk(Qd, Cd, k):
    s, i = hs.hs_retrieve_topk(Qd, Cd, k)
    hs.hs_get_device_error()
    return s.cpu().numpy(), i.cpu().numpy()


def parity(Q, C, k, gs, gi, rows):
    return check_rows(Q, C, k, gs, gi, rows)


def all_rows_properties(Q, C, k, gs, gi):
    """(i) and (ii) of the parity rule on every query."""
    N = C.shape[0]
    nq = Q.shape[0]
    assert (gi >= 0).all() and (gi < N).all()
    assert (np.diff(gs, axis=1) <= 0).all()
    srt = np.sort(gi, axis=1)
    assert (np.diff(srt, axis=1) > 0).all(), "duplicate ids within a query"
    exact = oracle.pair_scores(Q, C, np.repeat(np.arange(nq), k), gi.reshape(-1)).reshape(nq, k)
    err = np.abs(exact - gs).max()
    assert err <= 1e-3, err
    return err


def unit_pair(nq, N, d, seed):
    return synth.unit_rows(nq, d, seed, stream=901), synth.unit_rows(N, d, seed, stream=902)


def test_single_tile_single_kblock():
    Q, C = unit_pair(128, 256, 64, 1)
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), 10)
    parity(Q, C, 10, gs, gi, range(128))


def test_tiny_config():
    w = configs.build_retrieval_mix(configs.TINY)
    uidx, _ = oracle.unique_inverse(w["queries"].view(np.int32))
    Q, C = w["queries"][uidx], w["corpus"]
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), 10)
    parity(Q, C, 10, gs, gi, range(len(uidx)))


@pytest.mark.parametrize("nq,N,d,k", [
    (1, 1000, 384, 10),       # one query, ragged last corpus tile
    (130, 777, 72, 5),        # two query blocks, d not a multiple of 64
    (3, 300, 1024, 1),        # k = 1
    (257, 4096, 768, 16),     # largest register-list k
    (64, 40, 128, 40),        # k = N (full sort)
    (33, 5000, 256, 20),      # 32-slot register list
    (17, 3000, 256, 100),     # candidate-buffer path
    (5, 2000, 64, 33),        # smallest buffered k
    (40, 20000, 128, 1024),   # HS_TOPK_MAX_K
    (600, 100, 64, 12),       # CTA pairs, N < 128: the odd CTA's corpus half is past N
    (417, 3000, 1024, 32),    # CTA pairs over two query-block groups, k = 32, d = 1024
    (1000, 4096, 128, 16),    # four query-block groups, ragged last block
    (300, 30000, 128, 1024),  # CTA pairs at HS_TOPK_MAX_K: optimistic pass, flags, exact passes
])
def test_shapes(nq, N, d, k):
    Q, C = unit_pair(nq, N, d, nq * 7 + N)
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), k)
    parity(Q, C, k, gs, gi, range(nq))


def test_exact_ties_resolve_to_lower_index():
    Q, C = unit_pair(4, 3000, 256, 11)
    for q in range(4):               # three exact copies of each query
        for j in (2900 - q, 1500 + q, 10 + q):
            C[j] = Q[q]
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), 5)
    for q in range(4):
        assert gi[q, :3].tolist() == [10 + q, 1500 + q, 2900 - q]
        assert gs[q, 0] == gs[q, 1] == gs[q, 2]
    parity(Q, C, 5, gs, gi, range(4))


def test_integer_valued_exact_scores():
    # Small integers: bf16 products and fp32 sums are exact, so the GPU
    # scores must equal the oracle's exactly and ids must match exactly.
    rng = np.random.default_rng(2)
    Qf = rng.integers(-2, 3, size=(70, 128)).astype(np.float32)
    Cf = rng.integers(-2, 3, size=(900, 128)).astype(np.float32)
    Q = (Qf.view(np.uint32) >> 16).astype(np.uint16)
    C = (Cf.view(np.uint32) >> 16).astype(np.uint16)
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), 12)
    os_, oi = oracle.topk(Q, C, 12)
    assert (gs == os_).all() and (gi == oi).all()


def test_rag_mix_full_size():
    w = configs.build_retrieval_mix(configs.RAG_MIX)
    uidx, _ = oracle.unique_inverse(w["queries"].view(np.int32))
    Q, C = w["queries"][uidx], w["corpus"]
    assert Q.shape == (1434, 768) and C.shape == (1048576, 768)
    Cd = to_dev(C)
    gs, gi = gpu_topk(to_dev(Q), Cd, 10)
    del Cd
    all_rows_properties(Q, C, 10, gs, gi)
    # every merged query against the oracle's exact fp64 top-10
    check_rows(Q, C, 10, gs, gi, np.arange(len(Q)), tag="rag_mix_corpus_seed0")
    gc.collect()
    torch.cuda.empty_cache()


def test_batch_sweep_corpus():
    C = configs.sweep_corpus()
    assert C.shape == (2097152, 768)
    Cd = to_dev(C)
    for B in configs.BATCH_SWEEP["batches"]:
        b = configs.build_sweep_batch(B, seed=B)
        uidx, _ = oracle.unique_inverse(b["queries"].view(np.int32))
        Q = b["queries"][uidx]
        gs, gi = gpu_topk(to_dev(Q), Cd, 10)
        all_rows_properties(Q, C, 10, gs, gi)
        if len(Q) <= 512:
            rows = np.arange(len(Q))                 # every merged query
        else:                                        # a seeded sample of 256 + both ends
            rows = np.random.default_rng(B).choice(len(Q), size=256, replace=False)
            rows = np.union1d(rows, [0, len(Q) - 1])
        check_rows(Q, C, 10, gs, gi, rows)
    del Cd
    gc.collect()
    torch.cuda.empty_cache()


def test_large_corpus_planted_clusters():
    w = configs.build_large_corpus()
    C, Q = w["corpus"], w["queries"]
    assert C.shape == (8388608, 1024) and Q.shape == (4096, 1024)
    Cd = to_dev(C)
    gs, gi = gpu_topk(to_dev(Q), Cd, 100)
    del Cd
    # Structure at full size: every query's top-100 lies inside its own
    # cluster's 128 planted near-duplicates.
    members = w["members"]
    cl = w["query_cluster"]
    for q in range(Q.shape[0]):
        own = members[cl[q]]
        assert np.isin(gi[q], own).all()
    all_rows_properties(Q, C, 100, gs, gi)
    # a seeded sample of 256 queries (plus both ends) against the oracle's
    # exact top-100: the optimistic large-k pass must return exactly it
    rows = np.random.default_rng(4).choice(Q.shape[0], size=256, replace=False)
    rows = np.union1d(rows, [0, 1234, Q.shape[0] - 1])
    check_rows(Q, C, 100, gs, gi, rows)
    gc.collect()
    torch.cuda.empty_cache()


def test_argument_errors():
    C = torch.zeros((100, 64), dtype=torch.bfloat16, device="cuda")
    Q = torch.zeros((4, 64), dtype=torch.bfloat16, device="cuda")
    for k in (0, 101, 2000):
        with pytest.raises(hs.HsError):
            hs.hs_retrieve_topk(Q, C, k)
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    with pytest.raises(hs.HsError) as e:
        hs.hs_retrieve_topk(Q, C, 5, workspace=ws)
    assert e.value.status == hs.HS_ERR_WORKSPACE
    s, i = hs.hs_retrieve_topk(Q[:0], C, 5)
    assert s.shape == (0, 5)


def test_deterministic():
    Q, C = unit_pair(300, 20000, 256, 5)
    Qd, Cd = to_dev(Q), to_dev(C)
    a = hs.hs_retrieve_topk(Qd, Cd, 10)
    b = hs.hs_retrieve_topk(Qd, Cd, 10)
    hs.hs_get_device_error()
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])


def test_device_count_matches_host_count():
    Q, C = unit_pair(300, 5000, 256, 9)
    Qd, Cd = to_dev(Q), to_dev(C)
    for k in (10, 20, 40):
        ref_s, ref_i = hs.hs_retrieve_topk(Qd[:177], Cd, k)
        cnt = torch.tensor([177], dtype=torch.int32, device="cuda")
        s = torch.full((300, k), -7.0, device="cuda")
        i = torch.full((300, k), -7, dtype=torch.int32, device="cuda")
        hs.hs_retrieve_topk_n(Qd, cnt, Cd, k, out=(s, i))
        hs.hs_get_device_error()
        assert torch.equal(s[:177], ref_s) and torch.equal(i[:177], ref_i)
        assert (s[177:] == -7.0).all() and (i[177:] == -7).all()   # rows past the count untouched


def test_device_count_zero_and_clamped():
    Q, C = unit_pair(64, 3000, 128, 10)
    Qd, Cd = to_dev(Q), to_dev(C)
    s = torch.full((64, 5), 3.0, device="cuda")
    i = torch.full((64, 5), 3, dtype=torch.int32, device="cuda")
    hs.hs_retrieve_topk_n(Qd, torch.zeros(1, dtype=torch.int32, device="cuda"), Cd, 5, out=(s, i))
    hs.hs_get_device_error()
    assert (s == 3.0).all() and (i == 3).all()
    big = torch.tensor([1 << 30], dtype=torch.int32, device="cuda")
    s2, i2 = hs.hs_retrieve_topk_n(Qd, big, Cd, 5)
    ref_s, ref_i = hs.hs_retrieve_topk(Qd, Cd, 5)
    hs.hs_get_device_error()
    assert torch.equal(s2, ref_s) and torch.equal(i2, ref_i)


def test_large_k_floor_with_ties_beyond_k():
    # 60 exact copies of each query, some inside the first eighth of the
    # corpus (the floor sample): the floor equals the copies' score, every
    # copy ties with it, and the top 40 must be the 40 lowest-index copies.
    nq, N, d, k = 6, 40000, 128, 40
    Q, C = unit_pair(nq, N, d, 21)
    rng = np.random.default_rng(3)
    for q in range(nq):
        pos = rng.choice(N, size=60, replace=False)
        C[pos] = Q[q]
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), k)
    parity(Q, C, k, gs, gi, range(nq))
    os_, oi = oracle.topk(Q, C, k)
    assert (gi == oi).all()


def test_large_k_best_rows_outside_the_sample():
    # The best rows of every query sit in the last part of the corpus, so the
    # floor from the first eighth is far below the final k-th score.
    nq, N, d, k = 5, 40000, 128, 64
    Q, C = unit_pair(nq, N, d, 22)
    for q in range(nq):
        C[N - 200 - 30 * q: N - 30 * q] = Q[q]
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), k)
    parity(Q, C, k, gs, gi, range(nq))


def test_shared_floor_keeps_ties_across_splits():
    # 50 exact copies of each query spread over a corpus of many splits: every
    # list that holds >= k copies raises the query's shared floor to the copy
    # score, and lists elsewhere must still keep their copies (ties at the
    # floor), so the top 10 are the 10 lowest-index copies.
    nq, N, d, k = 6, 300000, 128, 10
    Q, C = unit_pair(nq, N, d, 31)
    rng = np.random.default_rng(7)
    for q in range(nq):
        pos = np.sort(rng.choice(N, size=50, replace=False))
        C[pos] = Q[q]
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), k)
    os_, oi = oracle.topk(Q, C, k)
    assert (gi == oi).all()
    parity(Q, C, k, gs, gi, range(nq))


@pytest.mark.parametrize("nq,N,d,k", [
    (1, 50000, 768, 10),      # one query, ragged last 128-row tile
    (16, 20000, 1024, 32),    # a full batch of 16, largest k and d of the small path
    (7, 777, 72, 5),          # d not a multiple of 64, few tiles
    (2, 130, 128, 1),         # two tiles, k = 1
])
def test_small_batch_path(nq, N, d, k):
    Q, C = unit_pair(nq, N, d, nq * 11 + N)
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), k)
    parity(Q, C, k, gs, gi, range(nq))


def test_small_batch_ties_and_device_count():
    nq, N, d, k = 16, 60000, 256, 10
    Q, C = unit_pair(nq, N, d, 41)
    rng = np.random.default_rng(5)
    for q in range(nq):
        C[np.sort(rng.choice(N, size=25, replace=False))] = Q[q]
    Qd, Cd = to_dev(Q), to_dev(C)
    os_, oi = oracle.topk(Q, C, k)
    gs, gi = gpu_topk(Qd, Cd, k)
    assert (gi == oi).all()
    for cnt_ in (0, 5, 16):
        s = torch.full((nq, k), -7.0, device="cuda")
        i = torch.full((nq, k), -7, dtype=torch.int32, device="cuda")
        hs.hs_retrieve_topk_n(Qd, torch.tensor([cnt_], dtype=torch.int32, device="cuda"), Cd, k,
                              out=(s, i))
        hs.hs_get_device_error()
        assert (i[:cnt_].cpu().numpy() == oi[:cnt_]).all()
        assert (i[cnt_:] == -7).all()


@pytest.mark.parametrize("nq,N,d,k", [
    (4, 40, 128, 10),         # small-batch path, corpus shorter than one 128-row tile
    (300, 200, 256, 10),      # CTA pairs, corpus shorter than one 256-row tile
    (260, 300, 64, 20),       # CTA pairs, 2 tiles, odd query-block count, 32-slot lists
    (129, 1000, 768, 12),     # two query blocks (one pair), 12-slot lists, k = 12
])
def test_tiny_corpus_edges(nq, N, d, k):
    Q, C = unit_pair(nq, N, d, nq + 3 * N)
    gs, gi = gpu_topk(to_dev(Q), to_dev(C), k)
    parity(Q, C, k, gs, gi, range(nq))


@pytest.mark.parametrize("hot", [0, 150])
def test_large_k_optimistic_pass_and_exact_fallback(hot):
    """k > 32 over >= 64 tiles: the optimistic register-list pass is exact
    when no list is cut; queries whose top-k crowds into one list's corpus
    range (here 200 contiguous near-copies of their direction) are flagged
    and recomputed by the exact two-pass path."""
    N, d, k, Q = 64 * 256 * 2, 128, 100, 300
    rng = np.random.default_rng(7 + hot)
    corpus = synth.unit_rows(N, d, 31)
    q = synth.unit_rows(Q, d, 32)
    if hot:
        base = (q[0].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        noise = rng.standard_normal((200, d)) * 0.02
        rows = base / np.linalg.norm(base) + noise
        rows /= np.linalg.norm(rows, axis=1, keepdims=True)
        corpus[1000:1200] = (rows.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
        q[1:hot] = q[0]
    s, i = hs.hs_retrieve_topk(to_dev(q), to_dev(corpus), k)
    hs.hs_get_device_error()
    s, i = s.cpu().numpy(), i.cpu().numpy()
    sample = np.unique(np.concatenate([np.arange(0, Q, 37), [0, 1, hot]]))
    sample = sample[sample < Q]
    os_, oi = oracle.topk(q[sample], corpus, k + 1)
    for r, qq in enumerate(sample):
        exact = oracle.pair_scores(q, corpus, np.full(k, qq), i[qq])
        check_topk(s[qq], i[qq], os_[r], oi[r], exact, N, k)
    if hot:
        assert set(range(1000, 1100)) & set(i[0].tolist())   # the crowded rows are found


@pytest.mark.parametrize("nq", [300, 8])    # CTA pairs; the small-batch kernel
def test_pipeline_wait_runs_out_and_reports_timeout(nq):
    """Failure detection without a fault: with a 1 ms wait limit and every
    CTA withholding the copies of its first corpus stage, the retrieval
    kernel's pipeline waits run out.  The CTA that counts the copies still
    waits for those it armed, and for its MMAs, before tensor memory is
    freed; the call returns in well under the default 2 s limit,
    hs_get_device_error reports HS_ERR_TIMEOUT (and clears it), and a
    normal call on the same stream then meets the parity rule."""
    import time
    N, d, k = 8192, 128, 10
    Q, C = unit_pair(nq, N, d, 21)
    Qd, Cd = to_dev(Q), to_dev(C)
    torch.cuda.synchronize()
    try:
        hs.hs_debug_retrieve_wait(1_000_000, 1)
        t0 = time.perf_counter()
        hs.hs_retrieve_topk(Qd, Cd, k)
        with pytest.raises(hs.HsError) as e:
            hs.hs_get_device_error()          # synchronises
        elapsed = time.perf_counter() - t0
        assert e.value.status == hs.HS_ERR_TIMEOUT
        assert elapsed < 1.0, elapsed
    finally:
        hs.hs_debug_retrieve_wait(0, 0)
    hs.hs_get_device_error()                  # cleared
    gs, gi = gpu_topk(Qd, Cd, k)
    parity(Q, C, k, gs, gi, range(nq))
