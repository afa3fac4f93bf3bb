"""hs_scatter_results vs the oracle: bit-exact on every copy path (16-byte,
word, byte), with maps from unique/inverse and random maps (result sharing,
Section 3.3 (I); Appendix A.2)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_22578_gb300 as hs
from hs_testutil import to_dev
from synth import configs

pytestmark = pytest.mark.gpu


def run(src, m):
    out = hs.hs_scatter_results(to_dev(src), to_dev(m.astype(np.int32)))
    hs.hs_get_device_error()
    return out.cpu().numpy()


@pytest.mark.parametrize("row_bytes", [16, 80, 1536, 40, 12, 3, 7, 1])
def test_random_maps(row_bytes):
    rng = np.random.default_rng(row_bytes)
    src = rng.integers(0, 256, size=(97, row_bytes), dtype=np.uint8)
    m = rng.integers(0, 97, size=1000)
    assert (run(src, m) == oracle.scatter(src, m)).all()


def test_dedup_heavy_payload_fan_out():
    w = configs.build_dedup_heavy()
    uidx, inv = oracle.unique_inverse(w["tokens"], w["lens"])
    rng = np.random.default_rng(0)
    payload = rng.integers(0, 256, size=(len(uidx), 1536), dtype=np.uint8)
    got = run(payload, inv)
    assert got.shape == (400000, 1536)
    assert (got == oracle.scatter(payload, inv)).all()


def test_gather_unique_rows_and_round_trip():
    w = configs.build_retrieval_mix(configs.RAG_MIX, corpus=False)
    q = w["queries"]
    uidx, inv = oracle.unique_inverse(q.view(np.int32))
    qu = run(q.view(np.uint8).reshape(q.shape[0], -1), uidx)
    assert (qu.view(np.uint16).reshape(-1, q.shape[1]) == q[uidx]).all()
    back = run(qu, inv)
    assert (back.view(np.uint16).reshape(q.shape) == q).all()


def test_misaligned_pointers_take_byte_path():
    rng = np.random.default_rng(5)
    src = rng.integers(0, 256, size=(33 * 32 + 1,), dtype=np.uint8)
    d_src = to_dev(src)[1:].view(33, 32)
    m = rng.integers(0, 33, size=64).astype(np.int32)
    out = hs.hs_scatter_results(d_src, to_dev(m))
    hs.hs_get_device_error()
    assert (out.cpu().numpy() == oracle.scatter(src[1:].reshape(33, 32), m)).all()


def test_empty_map_and_bad_entries():
    src = to_dev(np.arange(64, dtype=np.uint8).reshape(4, 16))
    out = hs.hs_scatter_results(src, torch.zeros(0, dtype=torch.int32, device="cuda"))
    assert out.shape[0] == 0
    dst = torch.zeros((3, 16), dtype=torch.uint8, device="cuda")
    hs.hs_scatter_results(src, to_dev(np.array([1, 4, -2], np.int32)), dst=dst)
    with pytest.raises(hs.HsError) as e:
        hs.hs_get_device_error()
    assert e.value.status == hs.HS_ERR_INVALID_ARG
    d = dst.cpu().numpy()
    assert (d[0] == np.arange(16, 32)).all() and (d[1:] == 0).all()


def test_overlap_rejected():
    buf = torch.zeros(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(hs.HsError):
        hs.hs_scatter_results(buf[:32].view(2, 16), to_dev(np.array([0, 1], np.int32)),
                              dst=buf[16:48].view(2, 16))


def test_memcpy_async_round_trips_host_and_device():
    """hs_memcpy_async (the C ABI's copy between host buffers and the
    device): pinned host -> device -> device -> pageable host, bytes
    unchanged; zero bytes is a no-op."""
    import numpy as np
    import torch
    rng = np.random.default_rng(12)
    src = torch.from_numpy(rng.integers(0, 255, size=(1000, 1536), dtype=np.uint8)).pin_memory()
    d0 = torch.empty_like(src, device="cuda")
    d1 = torch.empty_like(d0)
    back = torch.empty_like(src)                     # pageable
    s = torch.cuda.Stream()
    hs.hs_memcpy_async(d0, src, s)
    hs.hs_memcpy_async(d1, d0, s)
    hs.hs_memcpy_async(back, d1, s)
    s.synchronize()
    assert torch.equal(back, src)
    empty = torch.empty(0, dtype=torch.uint8)
    hs.hs_memcpy_async(torch.empty(0, dtype=torch.uint8, device="cuda"), empty, s)
    with pytest.raises(ValueError):
        hs.hs_memcpy_async(d0[:10], src, s)
