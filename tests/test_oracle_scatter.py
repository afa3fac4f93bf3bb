"""Pins for the oracle's scatter (result sharing: the output of the kept node
flows to every merged node, Section 3.3 (I) and Appendix A.2)."""
import numpy as np
import pytest

import oracle
from synth import configs


def test_identity_map():
    rng = np.random.default_rng(0)
    src = rng.integers(0, 255, size=(40, 24), dtype=np.uint8)
    assert (oracle.scatter(src, np.arange(40)) == src).all()


def test_matches_numpy_take():
    rng = np.random.default_rng(1)
    src = rng.integers(0, 255, size=(17, 80), dtype=np.uint8)
    m = rng.integers(0, 17, size=300)
    assert (oracle.scatter(src, m) == np.take(src, m, axis=0)).all()


def test_round_trip_through_unique():
    w = configs.build_dedup_heavy(scale=0.005)
    tok, lens = w["tokens"], w["lens"]
    uidx, inv = oracle.unique_inverse(tok, lens)
    back = oracle.scatter(tok[uidx], inv)
    assert (back == tok).all()            # the unique rows fan back out exactly


def test_empty_and_bad_maps():
    src = np.zeros((3, 16), np.uint8)
    assert oracle.scatter(src, np.zeros(0, np.int32)).shape == (0, 16)
    with pytest.raises(IndexError):
        oracle.scatter(src, np.array([0, 3]))
    with pytest.raises(IndexError):
        oracle.scatter(src, np.array([-1]))
