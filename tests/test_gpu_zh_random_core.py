"""Randomized parity sweeps over the four steps of the path: seeded draws of
row counts, strides, length patterns, token ranges, duplicate structure and
planted fingerprint collisions for the fingerprint (Section 3.3, Eq. 2) and
the exact merge (Section 3.3 (I), Appendix A.2); query counts, corpus sizes,
dimensions and k across every retrieval kernel regime (Section 4.1); row
widths, alignments and maps for the scatter.  Integer results are compared
bit-exactly, retrieval results with the top-k parity rule."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
import synth
from hs_testutil import check_topk, to_dev

pytestmark = pytest.mark.gpu


def token_case(rng):
    """Rows drawn from a pool (so that some repeat), with lengths, junk past
    each length, and tokens from a small, a 16-bit or the full int32 range."""
    stride = int(rng.choice([1, 2, 3, 4, 5, 8, 16, 31, 32, 33, 64, 100, 255, 256, 512]))
    n_max = max(1, min(300_000, 12_000_000 // stride))
    n = int(np.exp(rng.uniform(0.0, np.log(n_max))))
    pool = max(1, int(n * float(rng.choice([0.002, 0.05, 0.5, 1.0]))))
    vocab = int(rng.choice([2, 50, 65536, 2**31 - 1]))
    lo = -vocab if vocab == 2**31 - 1 else 0
    base = rng.integers(lo, vocab, size=(pool, stride), dtype=np.int64).astype(np.int32)
    pick = rng.integers(0, pool, size=n)
    tokens = base[pick]
    lens = None
    if rng.random() < 0.6:
        plens = rng.integers(0, stride + 1, size=pool).astype(np.int32)
        if rng.random() < 0.5:
            plens[:] = stride - rng.integers(0, min(stride, 3) + 1, size=pool)
        lens = plens[pick].copy()
        junk = rng.integers(-9, 9, size=tokens.shape).astype(np.int32)
        past = np.arange(stride)[None, :] >= lens[:, None]
        tokens[past] = junk[past]                  # ignored: past each row's length
    return np.ascontiguousarray(tokens), lens


@pytest.mark.parametrize("seed", range(40))
def test_fingerprint_and_unique_random(seed):
    rng = np.random.default_rng(5000 + seed)
    tokens, lens = token_case(rng)
    t = to_dev(tokens)
    L = to_dev(lens) if lens is not None else None
    fp = hs.hs_fingerprint(t, L)
    hs.hs_get_device_error()
    want_fp = oracle.fingerprint(tokens, lens)
    assert (fp.cpu().numpy().view(np.uint64) == want_fp).all()
    if seed % 3 == 2:                              # planted collisions: the contents decide
        mask = np.uint64(int(rng.choice([0x0, 0x1, 0xF, 0xFFFF])))
        fp = to_dev((want_fp & mask).astype(np.uint64))
    nu, uidx, inv = hs.hs_unique_inverse(fp, t, L)
    hs.hs_get_device_error()
    n_u = int(nu.item())
    ou, oi = oracle.unique_inverse(tokens, lens)
    assert n_u == len(ou)
    assert (uidx.cpu().numpy()[:n_u] == ou).all()
    assert (inv.cpu().numpy() == oi).all()


@pytest.mark.parametrize("seed", range(48))
def test_retrieve_random_shapes(seed):
    rng = np.random.default_rng(6000 + seed)
    regime = seed % 4
    nq = int(rng.integers(1, 17) if regime == 0 else
             rng.integers(17, 700) if regime == 1 else rng.integers(1, 300))
    N = max(1, int(np.exp(rng.uniform(0.0, np.log(70_000)))))
    d = int(rng.choice([8, 16, 24, 40, 64, 72, 128, 256, 384, 768, 1024, 1032, 2048]))
    k_max = min(N, hs.HS_TOPK_MAX_K)
    k = int(rng.choice([1, 2, 10, 16, 31, 32, 33, 100, 300, 1024, int(rng.integers(1, k_max + 1))]))
    k = min(k, k_max)
    Q = synth.unit_rows(nq, d, 7000 + seed, stream=903)
    C = synth.unit_rows(N, d, 7000 + seed, stream=904)
    Qd, Cd = to_dev(Q), to_dev(C)
    if regime == 3:                                # count in device memory, spare rows after it
        Qmax = nq + int(rng.integers(0, 40))
        Qpad = torch.zeros((Qmax, d), dtype=Qd.dtype, device="cuda")
        Qpad[:nq] = Qd
        s, i = hs.hs_retrieve_topk_n(Qpad, to_dev(np.array([nq], np.int32)), Cd, k)
        s, i = s[:nq], i[:nq]
    else:
        s, i = hs.hs_retrieve_topk(Qd, Cd, k)
    hs.hs_get_device_error()
    gs, gi = s.cpu().numpy(), i.cpu().numpy()
    assert (gi >= 0).all() and (gi < N).all()
    assert (np.diff(gs, axis=1) <= 0).all()
    assert (np.diff(np.sort(gi, axis=1), axis=1) > 0).all(), "an id twice in one query"
    rows = np.unique(rng.choice(nq, size=min(nq, 10), replace=False))
    os_, oi = oracle.topk(Q[rows], C, min(k + 1, N))
    exact = oracle.pair_scores(Q, C, np.repeat(rows, k), gi[rows].reshape(-1)).reshape(-1, k)
    for r, q in enumerate(rows):
        check_topk(gs[q], gi[q], os_[r], oi[r], exact[r], N, k)


@pytest.mark.parametrize("seed", range(24))
def test_scatter_random(seed):
    rng = np.random.default_rng(8000 + seed)
    row_bytes = int(rng.choice([1, 2, 3, 4, 12, 16, 40, 48, 80, 800, 1536, 4000, int(rng.integers(1, 3000))]))
    n_src = int(rng.integers(1, 5000))
    n = int(rng.integers(0, 60_000))
    off = int(rng.choice([0, 0, 1, 4, 8]))          # unaligned starts take the narrower paths
    flat = rng.integers(0, 256, size=n_src * row_bytes + off, dtype=np.uint8)
    src = flat[off:].reshape(n_src, row_bytes)
    m = rng.integers(0, n_src, size=n).astype(np.int32)
    d_src = to_dev(flat)[off:].view(n_src, row_bytes)
    out = hs.hs_scatter_results(d_src, to_dev(m))
    hs.hs_get_device_error()
    assert (out.cpu().numpy() == oracle.scatter(src, m)).all()
