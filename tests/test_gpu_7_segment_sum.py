"""hs_segment_sum against the oracle: the priority contribution of a fused
node is the sum of the contributions of the rows merged into it (Section
3.3, "Reuse-Driven Priority Adjustment", Eq. 3).  Integer-valued and dyadic
contributions are compared bit-exactly (every partial sum is exact in
fp64); general values within the fp64 summation bound of the exact sum."""
import math
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
import synth
from hs_testutil import to_dev
from synth import configs

pytestmark = pytest.mark.gpu
U = 2.0 ** -53
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "segment_sum_hand.txt")


def gpu_sum(phi, inv, max_groups, count=None):
    c = None if count is None else to_dev(np.array([count], np.int32))
    out = hs.hs_segment_sum(to_dev(np.asarray(phi, np.float64)), to_dev(np.asarray(inv, np.int32)),
                            max_groups, n_groups_dev=c)
    hs.hs_get_device_error()
    return out.cpu().numpy()


def test_hand_example():
    vals = {}
    for line in open(GOLDEN):
        if line.strip() and not line.startswith("#"):
            k, v = line.split(":", 1)
            vals[k.strip()] = v.split()
    out = gpu_sum(np.array(vals["phi"], float), np.array(vals["inverse"], np.int32),
                  int(vals["groups"][0]))
    assert (out == np.array(vals["expect"], float)).all()


def dedup_inverse(scale):
    w = configs.build_dedup_heavy(scale=scale)
    t, L = to_dev(w["tokens"]), to_dev(w["lens"])
    nu, _, inv = hs.hs_unique_inverse(hs.hs_fingerprint(t, L), t, L)
    hs.hs_get_device_error()
    return int(nu.item()), inv


@pytest.mark.parametrize("scale", [0.01, 1.0])
def test_zipf_groups_exact_for_integers(scale):
    """Integer contributions over the dedup-heavy merge (a Zipf head of many
    thousands of copies in one group at full scale): bit-exact."""
    n_u, inv_d = dedup_inverse(scale)
    inv = inv_d.cpu().numpy()
    rng = np.random.default_rng(5)
    phi = rng.integers(0, 1 << 16, size=len(inv)).astype(np.float64)
    out = hs.hs_segment_sum(to_dev(phi), inv_d, len(inv),
                            n_groups_dev=torch.tensor([n_u], dtype=torch.int32, device="cuda"))
    hs.hs_get_device_error()
    out = out.cpu().numpy()
    assert (out[:n_u] == oracle.segment_sum(phi, inv, n_u)).all()
    assert (out[n_u:] == 0).all()
    ones = gpu_sum(np.ones(len(inv)), inv, n_u)
    assert (ones == np.bincount(inv, minlength=n_u)).all()


def test_real_values_within_summation_bound():
    n_u, inv_d = dedup_inverse(0.05)
    inv = inv_d.cpu().numpy()
    rng = np.random.default_rng(6)
    phi = rng.standard_normal(len(inv)) * 3 + 1
    out = gpu_sum(phi, inv, n_u)
    ref = oracle.segment_sum(phi, inv, n_u)
    order = np.argsort(inv, kind="stable")
    bounds = np.searchsorted(inv[order], np.arange(n_u + 1))
    for u in range(n_u):
        members = phi[order[bounds[u]:bounds[u + 1]]]
        h = len(members) - 1
        tol = (h * U / (1 - h * U)) * np.abs(members).sum()
        exact = math.fsum(members.tolist())
        assert abs(out[u] - exact) <= tol and abs(ref[u] - exact) <= tol


def test_one_hot_group_and_many_tiles():
    n = 3 * 2048 * 152 + 17                 # several tiles per CTA, ragged tail
    phi = np.arange(n, dtype=np.float64) % 1000
    inv = np.zeros(n, np.int32)
    inv[::7] = 1
    out = gpu_sum(phi, inv, 3)
    assert (out == oracle.segment_sum(phi, inv, 3)).all()
    assert out[2] == 0


def test_count_and_bad_entries():
    phi = np.ones(10)
    inv = np.array([0, 1, 2, 3, 4, 0, 1, 2, 3, 4], np.int32)
    out = gpu_sum(phi, inv, 8, count=5)
    assert out.tolist() == [2, 2, 2, 2, 2, 0, 0, 0]
    c = to_dev(np.array([3], np.int32))
    o = hs.hs_segment_sum(to_dev(phi), to_dev(inv), 8, n_groups_dev=c)
    with pytest.raises(hs.HsError):          # ordinals 3 and 4 are past the count
        hs.hs_get_device_error()
    assert o.cpu().numpy().tolist() == [2, 2, 2, 0, 0, 0, 0, 0]
    assert gpu_sum(np.zeros(0), np.zeros(0, np.int32), 4).tolist() == [0, 0, 0, 0]


@pytest.mark.parametrize("pattern", ["hot_high_ordinals", "cold_uniform", "identity",
                                     "late_hot", "adjacent_pairs", "dense_only"])
def test_group_patterns_exact(pattern):
    """Hot groups with large ordinals (merged in the per-CTA hash table),
    cold groups spread over many ordinals (added directly), one row per
    group, a hot group first seen after 10,000 others, pairs of adjacent
    rows (512 repeated groups per 1024-row tile: the hash table fills and
    the bounded probing sends the rest to the output), and every ordinal
    below the dense array's 256."""
    n = 300_000
    rng = np.random.default_rng(9)
    if pattern == "hot_high_ordinals":
        inv = (100_000 + rng.integers(0, 7, size=n)).astype(np.int32)
        G = 100_007
    elif pattern == "cold_uniform":
        inv = rng.integers(0, 200_000, size=n).astype(np.int32)
        G = 200_000
    elif pattern == "late_hot":
        inv = (np.arange(n) % 10_000).astype(np.int32)
        inv[10_000:] = np.where(rng.random(n - 10_000) < 0.5, 5_000,
                                rng.integers(0, 10_000, n - 10_000))
        G = 10_000
    elif pattern == "adjacent_pairs":
        inv = (1_000 + np.arange(n) // 2).astype(np.int32)
        G = 1_000 + n // 2
    elif pattern == "dense_only":
        inv = rng.integers(0, 256, size=n).astype(np.int32)
        G = 256
    else:
        inv = rng.permutation(n).astype(np.int32)
        G = n
    phi = rng.integers(-(1 << 20), 1 << 20, size=n).astype(np.float64)
    assert (gpu_sum(phi, inv, G) == oracle.segment_sum(phi, inv, G)).all()
