"""Property checks of the oracle's segment sum and rerank on small random
inputs (hypothesis), against brute-force restatements that share nothing
with the oracle's code: every group summed exactly with Python fractions,
and every candidate ranked by sorting all of them."""
from fractions import Fraction

import numpy as np
import pytest

import oracle

hyp = pytest.importorskip("hypothesis")
from hypothesis import given, settings  # noqa: E402
from hypothesis import strategies as st  # noqa: E402


@settings(max_examples=60, deadline=None)
@given(st.lists(st.tuples(st.integers(0, 9), st.integers(-2**20, 2**20)), min_size=0, max_size=80),
       st.integers(10, 14))
def test_segment_sum_matches_exact_fractions(rows, groups):
    inv = np.array([g for g, _ in rows], np.int32)
    phi = np.array([v / 8.0 for _, v in rows], np.float64)      # dyadic: exact in fp64
    out = oracle.segment_sum(phi, inv, groups)
    want = [Fraction(0)] * groups
    for g, v in rows:
        want[g] += Fraction(v, 8)
    assert [Fraction(x) for x in out] == want


def bf16(x):
    return (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)


@settings(max_examples=40, deadline=None)
@given(st.integers(1, 4), st.integers(1, 8), st.integers(1, 6), st.data())
def test_rerank_matches_sort_of_all_candidates(nq, k1, d, data):
    n = 12
    vals = st.integers(-3, 3)
    rc = bf16(np.array(data.draw(st.lists(st.lists(vals, min_size=d, max_size=d),
                                          min_size=n, max_size=n)), np.float32))
    rq = bf16(np.array(data.draw(st.lists(st.lists(vals, min_size=d, max_size=d),
                                          min_size=nq, max_size=nq)), np.float32))
    cand = np.array(data.draw(st.lists(st.lists(st.integers(-1, n - 1), min_size=k1,
                                                max_size=k1), min_size=nq, max_size=nq)),
                    np.int32)
    k2 = data.draw(st.integers(1, k1))
    s, i = oracle.rerank(rq, rc, cand, k2)
    for q in range(nq):
        qv = (rq[q].astype(np.uint32) << 16).view(np.float32).astype(int)
        scored = []
        for c in cand[q]:
            if c < 0:
                continue
            cv = (rc[c].astype(np.uint32) << 16).view(np.float32).astype(int)
            scored.append((-int(np.dot(qv, cv)), int(c)))
        scored.sort()
        for j in range(k2):
            if j < len(scored):
                assert i[q, j] == scored[j][1] and s[q, j] == -scored[j][0]
            else:
                assert i[q, j] == -1 and np.isinf(s[q, j])
