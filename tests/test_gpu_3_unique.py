"""hs_unique_inverse vs the oracle: bit-exact unique sets and inverse maps
(topological fusion, Section 3.3 (I); merge sets, Appendix A.2), including
forced fingerprint collisions resolved by the full-row comparison."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
from hs_testutil import to_dev
from synth import configs

pytestmark = pytest.mark.gpu


def gpu_unique(tokens, lens=None, fp=None):
    t = to_dev(tokens)
    L = to_dev(lens) if lens is not None else None
    f = hs.hs_fingerprint(t, L) if fp is None else to_dev(fp.astype(np.uint64))
    nu, uidx, inv = hs.hs_unique_inverse(f, t, L)
    hs.hs_get_device_error()
    n = int(nu.item())
    return uidx[:n].cpu().numpy(), inv.cpu().numpy()


def same_as_oracle(tokens, lens=None, fp=None):
    gu, gi = gpu_unique(tokens, lens, fp)
    ou, oi = oracle.unique_inverse(tokens, lens)
    assert len(gu) == len(ou)
    assert (gu == ou).all() and (gi == oi).all()
    return len(gu)


def test_tiny():
    w = configs.build_retrieval_mix(configs.TINY, corpus=False)
    assert same_as_oracle(w["tokens"]) == 128
    assert same_as_oracle(w["queries"].view(np.int32)) == 24


def test_rag_mix_full():
    w = configs.build_retrieval_mix(configs.RAG_MIX, corpus=False)
    assert same_as_oracle(w["tokens"]) == 65536 - 26214
    assert same_as_oracle(w["queries"].view(np.int32)) == 2048 - 614


def test_dedup_heavy_full():
    w = configs.build_dedup_heavy()
    nu = same_as_oracle(w["tokens"], w["lens"])
    assert 20000 < nu < 100000


@pytest.mark.parametrize("mask", [0xF, 0x1, 0x0])
def test_forced_collisions(mask):
    # Fingerprints truncated to a few bits: distinct rows collide and must be
    # told apart by the full comparison.
    rng = np.random.default_rng(mask + 1)
    n, stride = 1500, 24
    base = rng.integers(0, 4, size=(60, stride)).astype(np.int32)
    tok = base[rng.integers(0, 60, size=n)]
    lens = rng.integers(20, 25, size=n).astype(np.int32)
    fp = oracle.fingerprint(tok, lens) & np.uint64(mask)
    same_as_oracle(tok, lens, fp)


def test_collisions_mixed_with_clean_segments():
    w = configs.build_dedup_heavy(scale=0.01)
    fp = oracle.fingerprint(w["tokens"], w["lens"])
    fp[fp % np.uint64(7) == 0] &= np.uint64(0x3)    # some segments collide, most do not
    same_as_oracle(w["tokens"], w["lens"], fp)


def test_edge_cases():
    one = np.array([[1, 2, 3]], np.int32)
    assert same_as_oracle(one) == 1
    assert same_as_oracle(np.tile(np.arange(7, dtype=np.int32), (3000, 1))) == 1
    assert same_as_oracle(np.arange(5000 * 3, dtype=np.int32).reshape(5000, 3)) == 5000
    tokens = np.array([[1, 2, 0, 0], [1, 2, 9, 9], [1, 2, 0, 0], [1, 2, 0, 5], [1, 2, 0, 6],
                       [1, 2, 0, 0]], np.int32)
    lens = np.array([2, 2, 3, 3, 4, 0], np.int32)
    gu, gi = gpu_unique(tokens, lens)
    assert gu.tolist() == [0, 2, 4, 5] and gi.tolist() == [0, 0, 1, 1, 2, 3]
    last = np.tile(np.arange(64, dtype=np.int32), (4, 1))
    last[1, -1] += 1
    last[3, -1] += 1
    gu, gi = gpu_unique(last)
    assert gu.tolist() == [0, 1] and gi.tolist() == [0, 1, 0, 1]


def test_empty_input():
    t = torch.zeros((0, 4), dtype=torch.int32, device="cuda")
    f = torch.zeros(0, dtype=torch.int64, device="cuda")
    nu, _, _ = hs.hs_unique_inverse(f, t)
    assert int(nu.item()) == 0


def test_unaligned_rows():
    rng = np.random.default_rng(4)
    base = rng.integers(0, 5, size=(30, 11)).astype(np.int32)
    tok = base[rng.integers(0, 30, size=700)]
    lens = rng.integers(8, 12, size=700).astype(np.int32)
    same_as_oracle(tok, lens)


def test_multi_tile_ragged_sizes():
    for n in [4095, 4096, 4097, 12289]:
        rng = np.random.default_rng(n)
        tok = rng.integers(0, 3, size=(n, 6)).astype(np.int32)
        same_as_oracle(tok)


def test_deterministic_and_workspace_reuse():
    w = configs.build_dedup_heavy(scale=0.05)
    t, L = to_dev(w["tokens"]), to_dev(w["lens"])
    f = hs.hs_fingerprint(t, L)
    ws = torch.empty(hs.hs_unique_inverse_workspace(t.shape[0]), dtype=torch.uint8, device="cuda")
    ws.fill_(0xAB)                                    # stale contents must not matter
    runs = []
    for _ in range(2):
        nu, uidx, inv = hs.hs_unique_inverse(f, t, L, workspace=ws)
        n = int(nu.item())
        runs.append((n, uidx[:n].clone(), inv.clone()))   # entries past n_unique are unspecified
    hs.hs_get_device_error()
    assert runs[0][0] == runs[1][0]
    assert torch.equal(runs[0][1], runs[1][1]) and torch.equal(runs[0][2], runs[1][2])


def test_workspace_too_small_is_rejected():
    t = torch.zeros((10, 4), dtype=torch.int32, device="cuda")
    f = torch.zeros(10, dtype=torch.int64, device="cuda")
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    with pytest.raises(hs.HsError) as e:
        hs.hs_unique_inverse(f, t, workspace=ws)
    assert e.value.status == hs.HS_ERR_WORKSPACE


def test_unique_idx_tail_is_a_valid_map():
    w = configs.build_retrieval_mix(configs.TINY, corpus=False)
    t = to_dev(w["tokens"])
    f = hs.hs_fingerprint(t)
    uidx = torch.full((t.shape[0],), 12345, dtype=torch.int32, device="cuda")
    nu = torch.empty(1, dtype=torch.int32, device="cuda")
    inv = torch.empty(t.shape[0], dtype=torch.int32, device="cuda")
    hs.hs_unique_inverse(f, t, out=(nu, uidx, inv))
    hs.hs_get_device_error()
    n = int(nu.item())
    assert n == 128 and (uidx[n:] == 0).all()


@pytest.mark.parametrize("n,distinct", [(4096, 4096), (200_000, 50_000)])
def test_constant_fingerprints_regroup_in_linear_work(n, distinct):
    """Every row given the same fingerprint (a caller's weak hash): each row
    that differs from row 0 is a collision.  The collision list is regrouped
    by a second key and compared in full — on the one-launch path (n <= 4096)
    and on the multi-kernel path — and the result is still exact."""
    rng = np.random.default_rng(n)
    base = rng.integers(-(1 << 30), 1 << 30, size=(distinct, 6)).astype(np.int32)
    tok = base[rng.integers(0, distinct, size=n)]
    same_as_oracle(tok, None, np.zeros(n, np.uint64))
    lens = rng.integers(0, 7, size=n).astype(np.int32)   # lengths in the key too
    same_as_oracle(tok, lens, np.full(n, 12345, np.uint64))


def test_lookback_wait_runs_out_and_reports_timeout():
    """Failure detection without a fault: the scan's look-back wait gets a
    1 ms limit and tile 1 withholds its status, so the later tiles wait for
    a status nobody publishes.  The call returns within the limit (not the
    default 2 s), hs_get_device_error reports HS_ERR_TIMEOUT and clears it,
    and the next call on the same stream is exact again."""
    import time
    w = configs.build_dedup_heavy(scale=0.2)
    tok, ln = w["tokens"][:70000], w["lens"][:70000]     # five scan tiles
    t, L = to_dev(tok), to_dev(ln)
    f = hs.hs_fingerprint(t, L)
    hs.hs_get_device_error()
    try:
        hs.hs_debug_scan_wait(1_000_000, 1)
        t0 = time.perf_counter()
        hs.hs_unique_inverse(f, t, L)
        with pytest.raises(hs.HsError) as e:
            hs.hs_get_device_error()
        elapsed = time.perf_counter() - t0
        assert e.value.status == hs.HS_ERR_TIMEOUT
        assert elapsed < 1.0, elapsed
    finally:
        hs.hs_debug_scan_wait()
    hs.hs_get_device_error()                              # the word was cleared
    nu, uidx, inv = hs.hs_unique_inverse(f, t, L)
    hs.hs_get_device_error()
    ou, oi = oracle.unique_inverse(tok, ln)
    n = int(nu.item())
    assert n == len(ou)
    assert (uidx[:n].cpu().numpy() == ou).all() and (inv.cpu().numpy() == oi).all()
