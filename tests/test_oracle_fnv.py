"""Pins for the oracle's fingerprint (the D_in part of Sig(v), Section 3.3 Eq. 2,
with H = 64-bit FNV-1a over octets).

The byte function is pinned to the published FNV-1a 64-bit test vectors; the
row function is pinned to the byte function through the little-endian octet
layout (numpy's explicit '<i4' encoding) and to the published vectors through
the continuation property of a seeded hash.
"""
import ast
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "fnv1a64_vectors.txt")


def _vectors():
    out = []
    with open(GOLDEN) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            lit, hx = line.rstrip("\n").split("\t")
            out.append((ast.literal_eval(lit), int(hx, 16)))
    return out


@pytest.mark.parametrize("data,expected", _vectors())
def test_published_vectors(data, expected):
    assert oracle.fnv1a64_bytes(data) == expected


def test_offset_basis():
    assert oracle.FNV64_OFFSET_BASIS == 0xCBF29CE484222325
    assert oracle.fnv1a64_bytes(b"") == oracle.FNV64_OFFSET_BASIS


def test_seed_continues_a_hash():
    # H(seed = H("foo"), "bar") must equal the published H("foobar"): a seeded
    # call continues the byte stream, which is how callers fold the operator
    # type, parameters and predecessor signatures of Eq. 2 into the seed.
    vec = dict(_vectors())
    h_foo = oracle.fnv1a64_bytes(b"foo")
    assert oracle.fnv1a64_bytes(b"bar", h_foo) == vec[b"foobar"]
    assert oracle.fnv1a64_bytes(b"ar\x00", oracle.fnv1a64_bytes(b"foob")) == vec[b"foobar\x00"]


def _le_word(b4: bytes) -> int:
    return int(np.frombuffer(b4, dtype="<i4")[0])


def test_row_is_little_endian_octets():
    vec = dict(_vectors())
    tok = np.array([[_le_word(b"foob")]], dtype=np.int32)
    assert int(oracle.fingerprint(tok)[0]) == vec[b"foob"]
    # Two tokens: "foob" + "ar\0\0" = octets of "foobar\0\0".
    tok2 = np.array([[_le_word(b"foob"), _le_word(b"ar\x00\x00")]], dtype=np.int32)
    h = oracle.fnv1a64_bytes(b"\x00", vec[b"foobar\x00"])
    assert int(oracle.fingerprint(tok2)[0]) == h


def test_rows_match_byte_function_on_random_rows():
    rng = np.random.default_rng(5)
    tokens = rng.integers(-2**31, 2**31 - 1, size=(40, 17), dtype=np.int64).astype(np.int32)
    lens = rng.integers(0, 18, size=40).astype(np.int32)
    seed = 0x1234_5678_9ABC_DEF0
    fp = oracle.fingerprint(tokens, lens, seed)
    for i in range(40):
        octets = tokens[i, : lens[i]].astype("<i4").tobytes()
        assert int(fp[i]) == oracle.fnv1a64_bytes(octets, seed)


def test_len_zero_row_is_the_seed():
    tok = np.arange(12, dtype=np.int32).reshape(3, 4)
    lens = np.zeros(3, dtype=np.int32)
    assert (oracle.fingerprint(tok, lens, 77) == 77).all()


def test_lens_none_means_full_rows():
    rng = np.random.default_rng(1)
    tok = rng.integers(0, 32000, size=(8, 9)).astype(np.int32)
    full = np.full(8, 9, dtype=np.int32)
    assert (oracle.fingerprint(tok) == oracle.fingerprint(tok, full)).all()


def test_padding_beyond_len_is_ignored():
    rng = np.random.default_rng(2)
    tok = rng.integers(0, 32000, size=(6, 10)).astype(np.int32)
    lens = np.array([0, 1, 3, 5, 9, 10], dtype=np.int32)
    tok2 = tok.copy()
    for i, L in enumerate(lens):
        tok2[i, L:] = rng.integers(0, 32000, size=10 - L)
    assert (oracle.fingerprint(tok, lens) == oracle.fingerprint(tok2, lens)).all()


def test_length_changes_the_hash():
    tok = np.zeros((2, 4), dtype=np.int32)
    lens = np.array([2, 3], dtype=np.int32)
    fp = oracle.fingerprint(tok, lens)
    assert fp[0] != fp[1]


def test_out_of_range_len_is_rejected():
    tok = np.zeros((2, 4), dtype=np.int32)
    with pytest.raises(ValueError):
        oracle.fingerprint(tok, np.array([1, 5], dtype=np.int32))
    with pytest.raises(ValueError):
        oracle.fingerprint(tok, np.array([-1, 0], dtype=np.int32))
