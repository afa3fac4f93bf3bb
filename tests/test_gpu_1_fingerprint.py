"""hs_fingerprint vs the oracle: bit-exact, on every workload shape and the
edge cases (Section 3.3 Eq. 2, D_in hashed with FNV-1a-64)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
from hs_testutil import fp_host, to_dev
from synth import configs

pytestmark = pytest.mark.gpu


def gpu_fp(tokens, lens=None, seed=hs.HS_FNV64_OFFSET_BASIS):
    t = to_dev(tokens)
    L = to_dev(lens) if lens is not None else None
    out = hs.hs_fingerprint(t, L, seed)
    hs.hs_get_device_error()
    return fp_host(out)


def test_tiny_chunks_and_queries():
    w = configs.build_retrieval_mix(configs.TINY, corpus=False)
    assert (gpu_fp(w["tokens"]) == oracle.fingerprint(w["tokens"])).all()
    q = w["queries"].view(np.int32)
    assert (gpu_fp(q) == oracle.fingerprint(q)).all()


def test_rag_mix_full_chunks_and_queries():
    w = configs.build_retrieval_mix(configs.RAG_MIX, corpus=False)
    assert w["tokens"].shape == (65536, 256)
    assert (gpu_fp(w["tokens"]) == oracle.fingerprint(w["tokens"])).all()
    q = w["queries"].view(np.int32)
    assert (gpu_fp(q) == oracle.fingerprint(q)).all()


def test_dedup_heavy_full_ragged_lengths():
    w = configs.build_dedup_heavy()
    assert w["tokens"].shape == (400000, 512)
    g = gpu_fp(w["tokens"], w["lens"])
    o = oracle.fingerprint(w["tokens"], w["lens"])
    assert (g == o).all()


@pytest.mark.parametrize("seed", [0, 1, 0xFFFFFFFFFFFFFFFF, 0x0123456789ABCDEF])
def test_seeds(seed):
    w = configs.build_retrieval_mix(configs.TINY, corpus=False)
    assert (gpu_fp(w["tokens"], seed=seed) == oracle.fingerprint(w["tokens"], seed=seed)).all()


def test_full_32bit_tokens_and_every_length():
    # Tokens >= 65536 and negative tokens take the octet-by-octet path; every
    # length 0..stride covers the 16-word blocks and the ragged tail.
    rng = np.random.default_rng(3)
    stride = 52
    n = 3 * (stride + 1)
    tok = rng.integers(-2**31, 2**31 - 1, size=(n, stride), dtype=np.int64).astype(np.int32)
    tok[::2, ::3] = rng.integers(0, 65536, size=tok[::2, ::3].shape)
    lens = (np.arange(n) % (stride + 1)).astype(np.int32)
    assert (gpu_fp(tok, lens) == oracle.fingerprint(tok, lens)).all()


@pytest.mark.parametrize("stride", [1, 3, 7, 13, 33])
def test_unaligned_rows_use_word_path(stride):
    rng = np.random.default_rng(stride)
    tok = rng.integers(0, 1 << 20, size=(301, stride)).astype(np.int32)
    lens = rng.integers(0, stride + 1, size=301).astype(np.int32)
    assert (gpu_fp(tok, lens) == oracle.fingerprint(tok, lens)).all()


def test_misaligned_base_pointer():
    rng = np.random.default_rng(9)
    big = rng.integers(0, 32000, size=(1 + 64 * 16,)).astype(np.int32)
    t = to_dev(big)[1:].view(64, 16)          # 4-byte aligned, not 16-byte aligned
    out = hs.hs_fingerprint(t)
    hs.hs_get_device_error()
    assert (fp_host(out) == oracle.fingerprint(big[1:].reshape(64, 16))).all()


def test_edge_sizes():
    assert hs.hs_fingerprint(torch.zeros((0, 8), dtype=torch.int32, device="cuda")).numel() == 0
    one = np.array([[5, 6, 7]], dtype=np.int32)
    assert (gpu_fp(one) == oracle.fingerprint(one)).all()
    zero_len = np.zeros((4, 8), dtype=np.int32)
    assert (gpu_fp(zero_len, np.zeros(4, np.int32), seed=42) == 42).all()
    empty_stride = np.zeros((3, 0), dtype=np.int32)
    assert (gpu_fp(empty_stride) == hs.HS_FNV64_OFFSET_BASIS).all()


def test_invalid_length_sets_device_error():
    tok = to_dev(np.zeros((4, 8), np.int32))
    lens = to_dev(np.array([1, 9, 2, -1], np.int32))
    out = hs.hs_fingerprint(tok, lens)
    with pytest.raises(hs.HsError) as e:
        hs.hs_get_device_error()
    assert e.value.status == hs.HS_ERR_INVALID_ARG
    got = fp_host(out)
    assert got[1] == 0 and got[3] == 0
    assert got[0] == oracle.fingerprint(np.zeros((1, 8), np.int32), np.array([1], np.int32))[0]
    hs.hs_get_device_error()      # cleared


def test_guard_band_untouched():
    w = configs.build_retrieval_mix(configs.TINY, corpus=False)
    n = w["tokens"].shape[0]
    buf = torch.full((n + 512,), 0x5A5A5A5A5A5A5A5A, dtype=torch.int64, device="cuda")
    hs.hs_fingerprint(to_dev(w["tokens"]), fp_out=buf[:n])
    hs.hs_get_device_error()
    assert (buf[n:] == 0x5A5A5A5A5A5A5A5A).all()
    assert (fp_host(buf[:n]) == oracle.fingerprint(w["tokens"])).all()


def test_deterministic():
    w = configs.build_dedup_heavy(scale=0.05)
    a = gpu_fp(w["tokens"], w["lens"])
    b = gpu_fp(w["tokens"], w["lens"])
    assert (a == b).all()


@pytest.mark.parametrize("stride,offset", [(200, 0), (200, 4), (100, 0)])
def test_chunk_paths_mixed_tokens(stride, offset):
    # Rows of several 32-token chunks plus a ragged tail.  offset 4 leaves the
    # base 16-byte (not 32-byte) aligned and stride 100 is not a multiple of
    # 8 tokens: both take 16-byte loads.  One large token in every third row
    # sends its chunk (and every other lane's chunk in that warp step) down
    # the octet-wise rounds.
    rng = np.random.default_rng(stride + offset)
    n = 2 * (stride + 1)
    tok = rng.integers(0, 32000, size=(n, stride)).astype(np.int32)
    rows = np.arange(0, n, 3)
    tok[rows, rng.integers(0, stride, size=len(rows))] = rng.integers(65536, 2**31 - 1,
                                                                      size=len(rows))
    lens = (np.arange(n) % (stride + 1)).astype(np.int32)
    flat = np.zeros(offset + n * stride, np.int32)
    flat[offset:] = tok.reshape(-1)
    t = to_dev(flat)[offset:].view(n, stride)
    out = hs.hs_fingerprint(t, to_dev(lens))
    hs.hs_get_device_error()
    assert (fp_host(out) == oracle.fingerprint(tok, lens)).all()


@pytest.mark.parametrize("pattern", [0, 1, 2])
def test_stream_rows_diagnostic_reads_exactly_the_valid_prefixes(pattern):
    """hs_debug_stream_rows (the read-ceiling diagnostic) folds the tokens it
    reads into an xor checksum: the valid prefixes for patterns 0 and 1,
    the whole padded rows for pattern 2."""
    rng = np.random.default_rng(pattern)
    n, stride = 3001, 72
    tokens = rng.integers(-2**31, 2**31 - 1, size=(n, stride), dtype=np.int64).astype(np.int32)
    lens = rng.integers(0, stride + 1, size=n).astype(np.int32)
    ck = torch.zeros(1, dtype=torch.int32, device="cuda")
    hs.hs_debug_stream_rows(to_dev(tokens), to_dev(lens), pattern, ck, 2)
    torch.cuda.synchronize()
    u = tokens.view(np.uint32)
    if pattern == 2:
        want = np.bitwise_xor.reduce(u.reshape(-1))
    else:
        mask = np.arange(stride)[None, :] < lens[:, None]
        want = np.bitwise_xor.reduce(np.where(mask, u, 0).reshape(-1))
    assert int(ck.cpu().numpy().view(np.uint32)[0]) == int(want)
