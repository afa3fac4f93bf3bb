"""Pins for the oracle's rerank (RAG with rerank, Section 4.1 "Workloads":
the initial top-12 chunks are rescored and the top-8 kept)."""
import os

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "rerank_hand.txt")


def bf16(x):
    return (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)


def read_golden():
    rq, rc, cand, expect = {}, {}, {}, {}
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        key, rest = line.split(":", 1)
        kind, idx = key.split()
        vals = rest.split()
        if kind == "expect":
            ids, sc = rest.split("|")
            expect[int(idx)] = ([int(v) for v in ids.split()], [float(v) for v in sc.split()])
        else:
            {"rq": rq, "rc": rc, "cand": cand}[kind][int(idx)] = [float(v) for v in vals]
    as_rows = lambda d: np.array([d[i] for i in sorted(d)])
    return (bf16(as_rows(rq)), bf16(as_rows(rc)), as_rows(cand).astype(np.int32), expect)


def test_hand_example():
    rq, rc, cand, expect = read_golden()
    s, i = oracle.rerank(rq, rc, cand, 3)
    for q, (ids, sc) in expect.items():
        assert i[q].tolist() == ids and s[q].tolist() == sc


def test_rerank_of_retrieval_prefix_is_retrieval():
    """With the retrieval vectors as rerank vectors, reranking the top-k1
    keeps its first k2 entries: the rerank agrees with the whole-corpus
    top-k oracle."""
    corpus = synth.unit_rows(3000, 64, 1)
    q = synth.unit_rows(20, 64, 2)
    s12, i12 = oracle.topk(q, corpus, 12)
    s8, i8 = oracle.rerank(q, corpus, i12, 8)
    assert (i8 == i12[:, :8]).all() and (s8 == s12[:, :8]).all()


def test_candidate_order_and_absent_entries():
    rc = synth.unit_rows(500, 32, 3)
    rq = synth.unit_rows(6, 32, 4)
    rng = np.random.default_rng(5)
    cand = np.stack([rng.choice(500, 12, replace=False) for _ in range(6)]).astype(np.int32)
    s, i = oracle.rerank(rq, rc, cand, 8)
    perm = cand[:, rng.permutation(12)]
    s2, i2 = oracle.rerank(rq, rc, perm, 8)
    assert (i == i2).all() and (s == s2).all()
    holes = cand.copy()
    holes[:, 5:] = -1                            # only 5 present
    s3, i3 = oracle.rerank(rq, rc, holes, 8)
    assert (i3[:, 5:] == -1).all() and np.isinf(s3[:, 5:]).all()
    assert (np.sort(i3[:, :5], axis=1) == np.sort(cand[:, :5], axis=1)).all()


def test_bad_candidate():
    rc = synth.unit_rows(10, 16, 1)
    with pytest.raises(IndexError):
        oracle.rerank(rc[:1], rc, np.array([[3, 10]], np.int32), 1)
