"""hs_unique_inverse_noalloc: the allocation-free variant of hs_unique_inverse,
for callers that may not allocate device memory where they merge rows (for
example code running during CUDA graph capture, plugins with a fixed memory
budget, or request paths that must not stall in an allocator).  Its scratch
is a fixed array inside the library, so it takes no workspace.

Called through the C ABI; each of two calls in a row must give exactly the
same outputs as hs_unique_inverse on the same input and as the oracle's
unique/inverse (unique sets and inverse maps are compared bit-exactly, as
everywhere in these tests).  Both of the variant's paths are covered: the
one-launch path of at most 4096 rows (which uses the scratch's counters and
collision list) and the multi-kernel path up to the 65,536-row limit.  This file is
collected last, so a run that stops at its first failure has already run every
other test."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
from hs_testutil import to_dev
from synth import configs

pytestmark = pytest.mark.gpu

LIMIT = 65536


def _lib():
    lib = hs.load()
    P, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    lib.hs_unique_inverse_noalloc.argtypes = [P, P, i64, i32, P, P, P, P, P]
    lib.hs_unique_inverse_noalloc.restype = ctypes.c_int
    return lib


def _noalloc(lib, fp, tokens, lens):
    n, stride = tokens.shape
    nu = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    uidx = torch.full((n,), -1, dtype=torch.int32, device="cuda")
    inv = torch.full((n,), -1, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    rc = lib.hs_unique_inverse_noalloc(fp.data_ptr(), tokens.data_ptr(), n, stride,
                                       None if lens is None else lens.data_ptr(),
                                       nu.data_ptr(), uidx.data_ptr(), inv.data_ptr(), stream)
    assert rc == hs.HS_OK, lib.hs_last_error()
    hs.hs_get_device_error()
    return nu, uidx, inv


def _check(lib, tokens_np, lens_np, mask=None):
    t = to_dev(tokens_np)
    L = None if lens_np is None else to_dev(lens_np)
    fp = hs.hs_fingerprint(t, L)
    if mask is not None:                     # forced fingerprint collisions
        fp = fp & mask
    nu_a, uidx_a, inv_a = _noalloc(lib, fp, t, L)
    nu_b, uidx_b, inv_b = hs.hs_unique_inverse(fp, t, L)
    hs.hs_get_device_error()
    n = int(nu_b.item())
    assert int(nu_a.item()) == n
    assert torch.equal(uidx_a[:n], uidx_b[:n])
    assert torch.equal(inv_a, inv_b)
    ou, oi = oracle.unique_inverse(tokens_np, lens_np)
    assert n == len(ou)
    assert (uidx_a[:n].cpu().numpy() == ou).all()
    assert (inv_a.cpu().numpy() == oi).all()


def test_noalloc_matches_workspace_entry_point_twice_in_a_row():
    lib = _lib()
    full = configs.build_retrieval_mix(configs.RAG_MIX, corpus=False)
    heavy = configs.build_dedup_heavy(scale=0.1)
    # Two different inputs one after the other: the second call must not be
    # affected by what the first left in the shared scratch.
    cases = [(full["tokens"], None), (heavy["tokens"][:50000], heavy["lens"][:50000])]
    assert full["tokens"].shape[0] == LIMIT
    for tokens_np, lens_np in cases:
        _check(lib, tokens_np, lens_np)


def test_noalloc_one_launch_path_with_collisions_twice_in_a_row():
    """At most 4096 rows take the one-launch path; keeping 4 bits of each
    fingerprint forces collisions, so the collision list in the scratch is
    used and must be cleared between the two calls."""
    lib = _lib()
    heavy = configs.build_dedup_heavy(scale=0.01)
    tok, ln = heavy["tokens"][:4096], heavy["lens"][:4096]
    for mask in (0xF, 0xF, None):
        _check(lib, tok, ln, mask)
    tiny = configs.build_retrieval_mix(configs.TINY, corpus=False)["tokens"]
    _check(lib, tiny, None, 0x1)
    _check(lib, tiny[:37], None)


def test_noalloc_rejects_rows_beyond_its_limit():
    lib = _lib()
    t = torch.zeros((LIMIT + 1, 4), dtype=torch.int32, device="cuda")
    fp = torch.zeros(LIMIT + 1, dtype=torch.int64, device="cuda")
    out = [torch.empty(LIMIT + 1, dtype=torch.int32, device="cuda") for _ in range(3)]
    rc = lib.hs_unique_inverse_noalloc(fp.data_ptr(), t.data_ptr(), LIMIT + 1, 4, None,
                                       out[0].data_ptr(), out[1].data_ptr(), out[2].data_ptr(),
                                       torch.cuda.current_stream().cuda_stream)
    assert rc == hs.HS_ERR_INVALID_ARG
    assert b"allocation-free limit" in lib.hs_last_error()
