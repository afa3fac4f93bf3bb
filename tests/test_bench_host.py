"""Host-side logic of bench.py on the CPU: the rank reduction (world_size 2,
gloo), clock-sample parsing and the profile-traffic lookup."""
import json
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out_q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = 10.0 + 5.0 * rank            # rank 1 is the slowest
        units = 100.0 * (rank + 1)
        t, u = bench.reduce_over_ranks(ms, units, world)
        bench.barrier(world)
        out_q.put((rank, t, u))
    finally:
        dist.destroy_process_group()


def test_reduce_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    for rank, t, u in got:
        assert t == 15.0          # max over ranks
        assert u == 300.0         # sum over ranks


def test_single_rank_is_identity():
    assert bench.reduce_over_ranks(3.5, 7.0, 1) == (3.5, 7.0)


def test_parse_clock_samples():
    lines = [
        "0, 1965, 2070, 900.1, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "0, 1980, 2070, 950.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "0, 345, 2070, 120.0, 0x0000000000000001, Not Active, Not Active, Not Active, Not Active",
        "garbage",
    ]
    c = bench.parse_clock_samples(lines)
    assert c["samples"] == 3
    assert c["sm_max_mhz"] == 2070
    assert c["reasons"] == ["sw_power_cap"]
    assert 1965 <= c["sm_mhz"] <= 1980          # idle sample excluded by power


def test_traffic_lookup_requires_matching_source(tmp_path, monkeypatch):
    src = tmp_path / "k.cu"
    src.write_text("kernel v1")
    prof = tmp_path / "profiles"
    prof.mkdir()
    (prof / "traffic.json").write_text(json.dumps(
        {"retrieve_kernel": {"bytes_per_launch": 123.0, "source_sha": bench.source_sha(str(src))}}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_from_profiles("retrieve_kernel", str(src)) == 123.0
    src.write_text("kernel v2")                 # kernel changed since the capture
    assert bench.traffic_from_profiles("retrieve_kernel", str(src)) is None
    assert bench.traffic_from_profiles("other", str(src)) is None


def test_peaks_fallback(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    peaks, kind = bench.load_peaks()
    assert kind == "fallback" and peaks["hbm_gbs"] == 6800.0


def test_warmup_floor():
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(bench.ROOT, "bench.py"), "--warmup", "1"],
                       capture_output=True, text=True)
    assert r.returncode != 0 and "warmup" in r.stderr


def test_oracle_baseline_is_measured_on_a_bounded_sample():
    """The CPU baseline and the reference arm time the oracle on a sample of
    the step and divide the merged queries they processed by the time they
    took (no extrapolation)."""
    from synth import configs
    w = configs.build_retrieval_mix(configs.TINY)
    r = bench.oracle_step(w, 5, 2)
    assert r["merged"] == 5 and r["merged_total"] == 24
    assert r["chunk_rows"] == round(256 * 5 / 24) and r["step_s"] > 0
    m = bench.oracle_measured(w, 0.2, 2, steps=2)
    assert m["steps"] == 2 and 2 <= m["S"] <= 24
    assert abs(m["value"] - m["S"] / (m["ms_per_step"] / 1e3)) < 1e-6 * m["value"]
    assert "measured" in bench.oracle_sample_desc(m)
    assert bench.cpu_model()
