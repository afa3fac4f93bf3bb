"""Pins for the oracle's exact unique-with-inverse (the merge step of
topological fusion, Section 3.3 "Dynamic Fusion and Reuse Mechanism" (I), and
the merge sets M(v*) of Appendix A.2).

Checked against an O(n^2) brute-force pairwise row comparison written
independently here, against the structural invariants of a unique/inverse
pair, and against the partitions the generator planted.
"""
import numpy as np
import pytest

import oracle
import synth
from synth import configs


def brute_force(tokens, lens):
    """rep[i] = smallest j <= i whose row equals row i (same length, same
    tokens below the length); ordinals by first occurrence."""
    n, stride = tokens.shape
    L = [int(x) for x in (lens if lens is not None else [stride] * n)]
    rows = [tuple(tokens[i, : L[i]].tolist()) for i in range(n)]
    uidx, inv, ordinal = [], [], {}
    for i in range(n):
        rep = next(j for j in range(i + 1) if rows[j] == rows[i])
        if rep == i:
            ordinal[i] = len(uidx)
            uidx.append(i)
        inv.append(ordinal[rep])
    return np.array(uidx, dtype=np.int32), np.array(inv, dtype=np.int32)


def check_invariants(tokens, lens, uidx, inv):
    n, stride = tokens.shape
    L = lens if lens is not None else np.full(n, stride)
    assert len(uidx) <= n
    assert (np.diff(uidx) > 0).all()                     # ascending, distinct
    assert (inv[uidx] == np.arange(len(uidx))).all()     # representatives map home
    if n:
        assert inv.min() >= 0 and inv.max() < len(uidx)
    for i in range(n):                                   # unique o inverse = input
        r = uidx[inv[i]]
        assert L[r] == L[i] and (tokens[r, : L[i]] == tokens[i, : L[i]]).all()


@pytest.mark.parametrize("seed", range(6))
def test_matches_brute_force_on_small_inputs(seed):
    rng = np.random.default_rng(seed)
    n, stride = 300, 6
    tokens = rng.integers(0, 3, size=(n, stride)).astype(np.int32)   # tiny vocab: many dups
    lens = rng.integers(0, stride + 1, size=n).astype(np.int32)
    for i in range(n):                                   # garbage beyond len
        tokens[i, lens[i]:] = rng.integers(-5, 5, size=stride - lens[i])
    u, v = oracle.unique_inverse(tokens, lens)
    bu, bv = brute_force(tokens, lens)
    assert (u == bu).all() and (v == bv).all()
    check_invariants(tokens, lens, u, v)


def test_matches_brute_force_full_rows():
    rng = np.random.default_rng(11)
    tokens = rng.integers(0, 2, size=(500, 5)).astype(np.int32)
    u, v = oracle.unique_inverse(tokens)
    bu, bv = brute_force(tokens, None)
    assert (u == bu).all() and (v == bv).all()


def test_edge_cases():
    z = np.zeros((0, 4), dtype=np.int32)
    u, v = oracle.unique_inverse(z)
    assert len(u) == 0 and len(v) == 0
    one = np.array([[7, 8]], dtype=np.int32)
    u, v = oracle.unique_inverse(one)
    assert u.tolist() == [0] and v.tolist() == [0]
    same = np.tile(np.array([[1, 2, 3]], dtype=np.int32), (50, 1))
    u, v = oracle.unique_inverse(same)
    assert u.tolist() == [0] and (v == 0).all()
    distinct = np.arange(60, dtype=np.int32).reshape(20, 3)
    u, v = oracle.unique_inverse(distinct)
    assert (u == np.arange(20)).all() and (v == np.arange(20)).all()


def test_length_and_padding_semantics():
    tokens = np.array([[1, 2, 0, 0],     # len 2
                       [1, 2, 9, 9],     # len 2, different padding -> equal to row 0
                       [1, 2, 0, 0],     # len 3 (token 0 counts) -> different
                       [1, 2, 0, 5],     # len 3 -> equal to row 2
                       [1, 2, 0, 6],     # len 4 -> new
                       [1, 2, 0, 0]],    # len 0 -> new (empty row)
                      dtype=np.int32)
    lens = np.array([2, 2, 3, 3, 4, 0], dtype=np.int32)
    u, v = oracle.unique_inverse(tokens, lens)
    assert u.tolist() == [0, 2, 4, 5]
    assert v.tolist() == [0, 0, 1, 1, 2, 3]


def test_rows_differing_in_last_token_only():
    base = np.arange(64, dtype=np.int32)
    tokens = np.tile(base, (4, 1))
    tokens[1, -1] += 1
    tokens[3, -1] += 1
    u, v = oracle.unique_inverse(tokens)
    assert u.tolist() == [0, 1] and v.tolist() == [0, 1, 0, 1]


def test_generator_ground_truth_tiny():
    w = configs.build_retrieval_mix(configs.TINY, corpus=False)
    u, v = oracle.unique_inverse(w["tokens"])
    gu, gv = synth.partition_of(w["chunk_root"])
    assert (u == gu).all() and (v == gv).all()
    assert len(u) == 256 - 128
    q32 = w["queries"].view(np.int32)
    u, v = oracle.unique_inverse(q32)
    gu, gv = synth.partition_of(w["query_root"])
    assert (u == gu).all() and (v == gv).all()
    assert len(u) == 32 - 8


def test_generator_ground_truth_rag_mix_scaled():
    w = configs.build_retrieval_mix(configs.RAG_MIX, scale=0.1, corpus=False)
    n = w["tokens"].shape[0]
    u, v = oracle.unique_inverse(w["tokens"])
    gu, gv = synth.partition_of(w["chunk_root"])
    assert (u == gu).all() and (v == gv).all()
    assert len(u) == n - int(round(0.4 * n))
    u, v = oracle.unique_inverse(w["queries"].view(np.int32))
    assert len(u) == 2048 - 614


def test_generator_ground_truth_dedup_heavy_scaled():
    w = configs.build_dedup_heavy(scale=0.02)
    u, v = oracle.unique_inverse(w["tokens"], w["lens"])
    gu, gv = synth.partition_of(w["chunk_root"])
    assert (u == gu).all() and (v == gv).all()
    check_invariants(w["tokens"][:2000], w["lens"][:2000],
                     *oracle.unique_inverse(w["tokens"][:2000], w["lens"][:2000]))


def test_out_of_range_len_is_rejected():
    with pytest.raises(ValueError):
        oracle.unique_inverse(np.zeros((2, 3), np.int32), np.array([4, 0], np.int32))


@pytest.mark.parametrize("seed", range(4))
def test_partition_is_invariant_under_row_permutation(seed):
    """Reordering the rows reorders the groups but never changes which rows
    share a group (only the choice of representative follows the order)."""
    rng = np.random.default_rng(700 + seed)
    n, stride = 3000, 7
    base = rng.integers(0, 3, size=(400, stride)).astype(np.int32)
    pick = rng.integers(0, 400, size=n)
    tokens = base[pick]
    lens = rng.integers(4, stride + 1, size=400).astype(np.int32)[pick]
    perm = rng.permutation(n)
    _, inv = oracle.unique_inverse(tokens, lens)
    _, inv_p = oracle.unique_inverse(tokens[perm], lens[perm])
    # rows i and j share a group iff their permuted images share one
    pairs = rng.integers(0, n, size=(20000, 2))
    where = np.empty(n, dtype=np.int64)
    where[perm] = np.arange(n)
    same = inv[pairs[:, 0]] == inv[pairs[:, 1]]
    same_p = inv_p[where[pairs[:, 0]]] == inv_p[where[pairs[:, 1]]]
    assert (same == same_p).all()
    assert inv.max() == inv_p.max()
