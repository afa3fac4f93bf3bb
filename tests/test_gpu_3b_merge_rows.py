"""hs_merge_rows (fingerprint + exact merge in one pass over the rows) vs the
oracle: fingerprints (Section 3.3, Eq. 2), unique sets and inverse maps
(Section 3.3 (I); Appendix A.2) bit-exact, and equal to hs_fingerprint
followed by hs_unique_inverse.  Forced fingerprint collisions (the table
keyed by a few bits of the fingerprint) must never merge unequal rows."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
from hs_testutil import to_dev
from synth import configs

pytestmark = pytest.mark.gpu


def merged(tokens, lens=None, seed=hs.HS_FNV64_OFFSET_BASIS):
    t = to_dev(tokens)
    L = None if lens is None else to_dev(lens)
    fp, nu, uidx, inv = hs.hs_merge_rows(t, L, seed)
    hs.hs_get_device_error()
    n = int(nu.item())
    return (fp.cpu().numpy().view(np.uint64), n, uidx.cpu().numpy(), inv.cpu().numpy())


def check(tokens, lens=None, seed=hs.HS_FNV64_OFFSET_BASIS):
    fp, n, uidx, inv = merged(tokens, lens, seed)
    assert (fp == oracle.fingerprint(tokens, lens, seed=seed)).all()
    ou, oi = oracle.unique_inverse(tokens, lens)
    assert n == len(ou)
    assert (uidx[:n] == ou).all() and (uidx[n:] == 0).all()
    assert (inv == oi).all()
    return n


def test_dedup_heavy_full():
    w = configs.build_dedup_heavy()
    n = check(w["tokens"], w["lens"])
    assert n == len(np.unique(w["chunk_root"]))


def test_rag_mix_chunks_and_tiny():
    w = configs.build_retrieval_mix(configs.RAG_MIX, corpus=False)
    assert check(w["tokens"]) == 65536 - 26214
    t = configs.build_retrieval_mix(configs.TINY, corpus=False)["tokens"]
    assert check(t) == 128                                   # the one-launch path


def random_rows(rng, n, stride, dup, big_tokens, zero_len_frac=0.05):
    base = rng.integers(0, 1 << 31 if big_tokens else 32000, size=(n, stride), dtype=np.int64)
    tokens = base.astype(np.int32)
    lens = rng.integers(0, stride + 1, size=n).astype(np.int32)
    lens[rng.random(n) < zero_len_frac] = 0
    src = rng.integers(0, n, size=n)
    copy = rng.random(n) < dup
    for i in np.flatnonzero(copy):
        j = src[i]
        tokens[i] = tokens[j]
        lens[i] = lens[j]
    # garbage past each row's length must be ignored
    tokens[:, :] = np.where(np.arange(stride)[None, :] < lens[:, None], tokens,
                            rng.integers(-5, 5, size=(n, stride)))
    return tokens, lens


@pytest.mark.parametrize("n,stride,dup,big", [
    (4097, 36, 0.5, False),       # just past the one-launch path, short rows
    (5000, 4, 0.7, True),         # one 16-byte piece per row, full-width tokens
    (33333, 128, 0.3, False),     # ragged last 32-row tile
    (70000, 1000, 0.6, True),     # long rows (32 chunk rounds), octet-wise rounds
    (100001, 64, 0.9, False),     # mostly duplicates, short rows
])
def test_random_shapes(n, stride, dup, big):
    rng = np.random.default_rng(n + stride)
    tokens, lens = random_rows(rng, n, stride, dup, big)
    check(tokens, lens)
    check(tokens, None, seed=0x0123456789ABCDEF)             # every row full length


def test_matches_the_two_calls_and_is_deterministic():
    w = configs.build_dedup_heavy(scale=0.3)
    t, L = to_dev(w["tokens"]), to_dev(w["lens"])
    fp2 = hs.hs_fingerprint(t, L)
    nu2, u2, i2 = hs.hs_unique_inverse(fp2, t, L)
    for _ in range(2):
        fp, nu, u, i = hs.hs_merge_rows(t, L)
        hs.hs_get_device_error()
        n = int(nu2.item())
        assert torch.equal(fp, fp2) and int(nu.item()) == n
        assert torch.equal(u[:n], u2[:n]) and torch.equal(i, i2)


@pytest.mark.parametrize("mask", [0xF, 0x1, 0xFFFF])
def test_forced_collisions_stay_exact(mask):
    """The table keyed by a few bits of the fingerprint: nearly every row
    collides with unequal rows; the full comparison and the regrouping of
    the collision list must still give the exact partition (the written
    fingerprints are the unmasked ones)."""
    w = configs.build_dedup_heavy(scale=0.05)
    try:
        hs.hs_debug_merge_key_mask(mask)
        check(w["tokens"], w["lens"])
        rng = np.random.default_rng(mask)
        tokens, lens = random_rows(rng, 9000, 32, 0.5, False)
        check(tokens, lens)
    finally:
        hs.hs_debug_merge_key_mask(0)


def test_invalid_lengths_are_reported():
    rng = np.random.default_rng(3)
    tokens, lens = random_rows(rng, 6000, 64, 0.5, False)
    bad = lens.copy()
    bad[[10, 4000]] = [-1, 65]
    t, L = to_dev(tokens), to_dev(bad)
    fp, nu, u, i = hs.hs_merge_rows(t, L)
    with pytest.raises(hs.HsError) as e:
        hs.hs_get_device_error()
    assert e.value.status == hs.HS_ERR_INVALID_ARG
    f = fp.cpu().numpy()
    assert f[10] == 0 and f[4000] == 0
    good = np.ones(6000, bool)
    good[[10, 4000]] = False
    assert (f.view(np.uint64)[good] == oracle.fingerprint(tokens, lens)[good]).all()
    # the rows with valid lengths keep their exact partition
    inv = i.cpu().numpy()
    _, oi = oracle.unique_inverse(tokens[good], lens[good])
    gi = inv[good]
    assert len(np.unique(gi)) == len(np.unique(oi))
    pairs = set(zip(gi.tolist(), oi.tolist()))
    assert len(pairs) == len(np.unique(oi))                  # the same partition


def test_unaligned_rows_take_the_two_calls():
    rng = np.random.default_rng(4)
    tokens, lens = random_rows(rng, 5000, 33, 0.5, False)    # row_stride % 4 != 0
    check(tokens, lens)


def test_workspace_errors():
    t = torch.zeros((5000, 16), dtype=torch.int32, device="cuda")
    with pytest.raises(hs.HsError) as e:
        hs.hs_merge_rows(t, workspace=torch.empty(256, dtype=torch.uint8, device="cuda"))
    assert e.value.status == hs.HS_ERR_WORKSPACE
    fp, nu, u, i = hs.hs_merge_rows(t[:0])
    hs.hs_get_device_error()
    assert int(nu.item()) == 0
