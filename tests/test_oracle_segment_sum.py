"""Pins for the oracle's segment sum: the priority contribution of a fused
node is the sum of the contributions of the nodes merged into it (Section
3.3, "Reuse-Driven Priority Adjustment", Eq. 3)."""
import math
import os

import numpy as np
import pytest

import oracle
from synth import configs

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "segment_sum_hand.txt")
U = 2.0 ** -53


def gamma(m):
    """Bound on the relative error of any fp64 summation order of m terms
    (Higham, Accuracy and Stability of Numerical Algorithms, Section 4.2)."""
    h = max(m - 1, 0)
    return h * U / (1 - h * U)


def read_golden():
    vals = {}
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        key, rest = line.split(":", 1)
        vals[key.strip()] = rest.split()
    return (np.array(vals["phi"], float), np.array(vals["inverse"], np.int32),
            int(vals["groups"][0]), np.array(vals["expect"], float))


def test_hand_example():
    phi, inv, g, expect = read_golden()
    assert (oracle.segment_sum(phi, inv, g) == expect).all()


def test_identity_and_single_group():
    rng = np.random.default_rng(0)
    phi = rng.random(1000) * 100
    assert (oracle.segment_sum(phi, np.arange(1000), 1000) == phi).all()
    one = oracle.segment_sum(phi, np.zeros(1000, np.int32), 1)
    exact = math.fsum(phi.tolist())
    assert abs(one[0] - exact) <= gamma(1000) * np.abs(phi).sum()


def test_group_sums_against_exact_sums_and_bincount():
    """Every group against the correctly rounded sum of its members (fsum),
    and the integer case against numpy's bincount."""
    w = configs.build_dedup_heavy(scale=0.005)
    uidx, inv = oracle.unique_inverse(w["tokens"], w["lens"])
    rng = np.random.default_rng(1)
    phi = rng.standard_normal(len(inv)) * 10
    out = oracle.segment_sum(phi, inv, len(uidx))
    order = np.argsort(inv, kind="stable")
    bounds = np.searchsorted(inv[order], np.arange(len(uidx) + 1))
    for u in range(len(uidx)):
        members = phi[order[bounds[u]:bounds[u + 1]]]
        assert len(members) >= 1
        exact = math.fsum(members.tolist())
        assert abs(out[u] - exact) <= gamma(len(members)) * np.abs(members).sum()
    counts = oracle.segment_sum(np.ones(len(inv)), inv, len(uidx))
    assert (counts == np.bincount(inv, minlength=len(uidx))).all()
    ints = rng.integers(-1000, 1000, size=len(inv)).astype(np.float64)
    assert (oracle.segment_sum(ints, inv, len(uidx)) ==
            np.bincount(inv, weights=ints, minlength=len(uidx))).all()


def test_conservation_and_empty_groups():
    rng = np.random.default_rng(2)
    phi = rng.integers(0, 1 << 20, size=5000).astype(np.float64)
    inv = rng.integers(0, 300, size=5000).astype(np.int32)
    out = oracle.segment_sum(phi, inv, 400)
    assert out.sum() == phi.sum()                 # integers below 2^53: exact
    assert (out[300:] == 0).all()
    assert oracle.segment_sum(np.zeros(0), np.zeros(0, np.int32), 3).tolist() == [0, 0, 0]


def test_bad_inverse():
    with pytest.raises(IndexError):
        oracle.segment_sum(np.ones(3), np.array([0, 3, 1]), 3)
    with pytest.raises(IndexError):
        oracle.segment_sum(np.ones(2), np.array([-1, 0]), 3)


def test_row_order_does_not_change_integer_sums():
    """Permuting the rows (with their group ordinals) leaves every group's
    sum unchanged; with integer contributions below 2^53 every partial sum
    is exact, so the sums must agree bit for bit."""
    rng = np.random.default_rng(31)
    n, groups = 50_000, 700
    phi = rng.integers(-(1 << 20), 1 << 20, size=n).astype(np.float64)
    inv = rng.integers(0, groups, size=n).astype(np.int32)
    perm = rng.permutation(n)
    a = oracle.segment_sum(phi, inv, groups)
    b = oracle.segment_sum(phi[perm], inv[perm], groups)
    assert (a == b).all()
    # and a relabelling of the groups permutes the sums the same way
    relabel = rng.permutation(groups).astype(np.int32)
    c = oracle.segment_sum(phi, relabel[inv], groups)
    assert (c[relabel] == a).all()
