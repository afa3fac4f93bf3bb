"""Pins for the oracle's exact top-k (the retrieval node of the RAG workloads,
Section 4.1 "Workloads": top-k chunks by similarity; exact inner product,
ties to the lower corpus index).

Checked against a hand-computed example, against the k = N special case
computed by numpy (fp64 matmul + stable lexsort), against planted exact
duplicate rows, and against the cluster structure the generator plants.
"""
import os

import numpy as np
import pytest

import oracle
from synth import configs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "topk_hand.txt")


def to_bf16_bits(x):
    f = np.asarray(x, dtype=np.float32)
    bits = f.view(np.uint32)
    assert ((bits & 0xFFFF) == 0).all(), "value not exact in bf16"
    return (bits >> 16).astype(np.uint16)


def bf16_to_f64(bits):
    return (np.asarray(bits, dtype=np.uint32) << 16).view(np.float32).astype(np.float64)


def load_golden():
    Q, C, exp = [], [], []
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            head, rest = line.split(":", 1)
            if head.startswith("query"):
                Q.append([float(x) for x in rest.split()])
            elif head.startswith("corpus"):
                C.append([float(x) for x in rest.split()])
            else:
                _, q, k = head.split()
                ids, sc = rest.split("|")
                exp.append((int(q), int(k), [int(x) for x in ids.split()],
                            [float(x) for x in sc.split()]))
    return to_bf16_bits(Q), to_bf16_bits(C), exp


def test_hand_computed():
    Q, C, exp = load_golden()
    for q, k, ids, sc in exp:
        s, i = oracle.topk(Q[q:q + 1], C, k)
        assert i[0].tolist() == ids
        assert s[0].tolist() == sc


def numpy_full_order(Q, C):
    s = bf16_to_f64(Q) @ bf16_to_f64(C).T
    N = C.shape[0]
    order = np.stack([np.lexsort((np.arange(N), -row)) for row in s])
    return s, order


@pytest.mark.parametrize("seed", [0, 1])
def test_k_equals_n_is_a_full_sort(seed):
    rng = np.random.default_rng(seed)
    # Small integers -> exact products and sums, so numpy's summation order
    # cannot differ from the oracle's; many ties exercise the index rule.
    Q = to_bf16_bits(rng.integers(-3, 4, size=(7, 16)).astype(np.float32))
    C = to_bf16_bits(rng.integers(-3, 4, size=(50, 16)).astype(np.float32))
    s, order = numpy_full_order(Q, C)
    os_, oi = oracle.topk(Q, C, 50)
    assert (oi == order).all()
    assert (os_ == np.take_along_axis(s, order, 1)).all()


def test_prefix_of_full_sort_on_unit_vectors():
    w = configs.build_retrieval_mix(configs.TINY)
    Q, C = w["queries"][:6], w["corpus"]
    s, order = numpy_full_order(Q, C)
    os_, oi = oracle.topk(Q, C, 10)
    assert (oi == order[:, :10]).all()
    assert np.abs(os_ - np.take_along_axis(s, order[:, :10], 1)).max() < 1e-12


def test_planted_duplicate_row_ties_to_lower_index():
    w = configs.build_retrieval_mix(configs.TINY)
    C = w["corpus"].copy()
    q = w["queries"][:1]
    C[3000] = q[0]                 # exact copy of the query: the best match
    C[1234] = q[0]                 # an earlier copy: must come first
    s, i = oracle.topk(q, C, 3)
    assert i[0, 0] == 1234 and i[0, 1] == 3000 and s[0, 0] == s[0, 1]
    assert abs(s[0, 0] - (bf16_to_f64(q[0]) ** 2).sum()) < 1e-12


def test_negative_and_zero_scores():
    Q = to_bf16_bits([[1.0, 0.0]])
    C = to_bf16_bits([[-1.0, 0.0], [-2.0, 0.0], [0.0, 5.0]])
    s, i = oracle.topk(Q, C, 3)
    assert i[0].tolist() == [2, 0, 1] and s[0].tolist() == [0.0, -1.0, -2.0]


def test_planted_clusters_dominate():
    cfg = dict(configs.LARGE_CORPUS, N=16384, n_clusters=16, members=128, nq=12)
    w = configs.build_large_corpus(cfg)
    s, i = oracle.topk(w["queries"], w["corpus"], 100)
    for q in range(w["queries"].shape[0]):
        own = set(w["members"][w["query_cluster"][q]].tolist())
        assert set(i[q].tolist()) <= own          # all 100 from its own cluster
        assert s[q, -1] > 0.98                    # near-duplicates: cos ~ 0.997


def test_pair_scores_agree():
    w = configs.build_retrieval_mix(configs.TINY)
    Q, C = w["queries"][:3], w["corpus"]
    s, i = oracle.topk(Q, C, 5)
    qi = np.repeat(np.arange(3), 5)
    ps = oracle.pair_scores(Q, C, qi, i.reshape(-1))
    assert (ps == s.reshape(-1)).all()


def test_bad_k_is_rejected():
    Q = to_bf16_bits([[1.0]])
    C = to_bf16_bits([[1.0], [2.0]])
    with pytest.raises(ValueError):
        oracle.topk(Q, C, 3)
    with pytest.raises(ValueError):
        oracle.topk(Q, C, 0)



def test_corpus_permutation_maps_ids():
    """Reordering the corpus rows maps each returned id through the
    permutation and leaves the scores unchanged (distinct scores, so no
    tie-break depends on the order)."""
    rng = np.random.default_rng(11)
    Q = rng.integers(-8, 9, size=(5, 16)).astype(np.float32)
    C = rng.integers(-8, 9, size=(300, 16)).astype(np.float32)
    # every score distinct: column 0 takes 300 distinct bf16-exact values
    # (8 significant bits) spaced 1024 or more apart, beyond what the other
    # columns can add (|sum| <= 15 * 64 = 960), and q[0] >= 1
    k = np.arange(300)
    C[:, 0] = (128 + k % 128) * 2.0 ** (10 + k // 128)
    Q[:, 0] = rng.integers(1, 9, size=5)
    q_bits, c_bits = to_bf16_bits(Q), to_bf16_bits(C)
    perm = rng.permutation(300)
    s1, i1 = oracle.topk(q_bits, c_bits, 12)
    s2, i2 = oracle.topk(q_bits, c_bits[perm], 12)
    assert (s1 == s2).all()
    assert (perm[i2] == i1).all()
