#!/usr/bin/env python
"""Benchmark of the embed-and-retrieve stage (one JSON line on rank 0).

A step is one pass of the whole hot path over one batch of the concurrent
RAG mix (64 workflows x 32 queries with 30% cross-workflow duplicates, plus
65,536 chunk rows of 256 tokens with 40% cross-workflow copies, against a
resident 1,048,576 x 768 bf16 corpus, k = 10):
    chunk fingerprint + exact unique/inverse,
    query fingerprint + exact unique/inverse + gather of the unique queries,
    tcgen05 retrieval with fused top-10 of the merged queries,
    scatter of scores and ids back to all 2,048 workflow queries.
``value`` is merged (unique) queries retrieved per second over all GPUs,
with inputs resident in HBM; ``e2e`` is the same metric through the public
API with the step's inputs copied from pinned host memory and its results
copied back (``hs_memcpy_async`` of the C ABI) inside the timed region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gb300|reference]

N > 1 runs under torchrun, one independent replica of the stage per GPU
(the path has no exchange step); the slowest rank's time is reported.
``--impl reference`` times the CPU oracle (the plain reference
implementation of the method) on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = ("merged queries/sec for top-k retrieval + dedup rows/sec; "
          "% of HBM/tensor roofline")
UNIT = "merged queries/s"
WORKLOAD = ("rag_mix: 64 workflows x 32 queries (30% cross-workflow exact duplicates -> "
            "1434 merged) + 65,536 chunk rows x 256 int32 tokens (40% cross-workflow copies); "
            "corpus 1,048,576 x 768 bf16 unit-norm; top-10")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ---------------------------------------------------------------- host logic
def load_peaks() -> tuple[dict, str]:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f), "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def dist_env() -> tuple[int, int, int]:
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def reduce_over_ranks(ms: float, units: float, world: int) -> tuple[float, float]:
    """Max of the per-rank times and sum of the per-rank units (identity when
    world == 1)."""
    if world == 1:
        return ms, units
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([ms], dtype=torch.float64, device=dev)
    u = torch.tensor([units], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


def barrier(world: int) -> None:
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.gpu)],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.2)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        return parse_clock_samples(open(self.path).read().splitlines())


def parse_clock_samples(lines: list[str]) -> dict:
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    sm, mx, pw, reasons = [], [], [], set()
    for ln in lines:
        parts = [p.strip() for p in ln.split(",")]
        if len(parts) < 9:
            continue
        try:
            sm.append(float(parts[1]))
            mx.append(float(parts[2]))
            pw.append(float(parts[3]))
        except ValueError:
            continue
        for n, v in zip(names, parts[5:9]):
            if v.lower().startswith("active"):
                reasons.add(n)
    if not sm:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
    # Samples under load: the upper half by power draw.
    order = sorted(range(len(sm)), key=lambda i: pw[i])
    loaded = [sm[i] for i in order[len(order) // 2:]] or sm
    return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(mx),
            "reasons": sorted(reasons), "samples": len(sm),
            "power_w_max": max(pw)}


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo), for the
    CPU-baseline record."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().startswith("Model name:"):
                return ln.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        fields = {}
        for ln in open("/proc/cpuinfo"):
            if ":" in ln:
                k, v = ln.split(":", 1)
                fields.setdefault(k.strip().lower(), v.strip())
        if "model name" in fields:
            return fields["model name"]
        if "cpu part" in fields:
            return "implementer %s part %s" % (fields.get("cpu implementer", "?"),
                                               fields["cpu part"])
    except OSError:
        pass
    import platform
    return platform.machine() or "unknown"


def source_sha(path: str) -> str:
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def traffic_from_profiles(kernel: str, src: str) -> float | None:
    """Per-launch DRAM bytes of `kernel` from the committed ncu summary, or
    None if there is none or the kernel source changed since it was taken."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(kernel)
    except (OSError, ValueError):
        return None
    if not rec or rec.get("source_sha") != source_sha(src):
        return None
    return float(rec["bytes_per_launch"])


# ---------------------------------------------------------------- workload
def build_workload(seed: int):
    from synth import configs
    return configs.build_retrieval_mix(configs.RAG_MIX, seed=seed)


# ---------------------------------------------------------------- CPU oracle leg
def oracle_step(w: dict, S: int, nthreads: int) -> dict:
    """One bounded sample of the RAG-mix step through the oracle, timed as a
    whole: the query merge of all 2,048 queries, the fp64 top-k of the first
    S merged queries over the full corpus (nthreads host threads), the result
    fan-out to the queries merged into them, and the chunk merge of the same
    share of the chunk rows (S / merged-query count of them; one thread)."""
    import numpy as np

    import oracle
    t0 = time.perf_counter()
    q32 = w["queries"].view(np.int32)
    oracle.fingerprint(q32)
    quidx, qinv = oracle.unique_inverse(q32)
    nq = len(quidx)
    S = max(1, min(S, nq))
    rows = max(1, int(round(w["tokens"].shape[0] * S / nq)))
    t1 = time.perf_counter()
    oracle.fingerprint(w["tokens"][:rows])
    oracle.unique_inverse(w["tokens"][:rows])
    t2 = time.perf_counter()
    s, i = oracle.topk(w["queries"][quidx[:S]], w["corpus"], w["k"], nthreads=nthreads)
    t3 = time.perf_counter()
    fan = np.flatnonzero(qinv < S)
    oracle.scatter(s, qinv[fan])
    oracle.scatter(i, qinv[fan])
    t4 = time.perf_counter()
    return {"merged": S, "merged_total": nq, "chunk_rows": rows, "step_s": t4 - t0,
            "t_topk_s": t3 - t2, "t_dedup_s": (t1 - t0) + (t2 - t1), "threads": nthreads}


def oracle_measured(w: dict, budget_s: float, nthreads: int, steps: int = 1) -> dict:
    """The oracle as it stands, on bounded samples of the RAG-mix step: a
    one-thread-per-core calibration sizes the sample S so that `steps`
    samples take about budget_s seconds; value = merged queries processed /
    the measured time of those samples (no extrapolation)."""
    cal = oracle_step(w, nthreads, nthreads)
    per_q = cal["step_s"] / cal["merged"]
    S = max(nthreads, int(budget_s / max(steps, 1) / per_q))
    samples = [oracle_step(w, S, nthreads) for _ in range(steps)]
    t = sum(x["step_s"] for x in samples)
    m = sum(x["merged"] for x in samples)
    return {"value": m / t, "ms_per_step": 1e3 * t / len(samples), "S": samples[0]["merged"],
            "merged_total": samples[0]["merged_total"], "chunk_rows": samples[0]["chunk_rows"],
            "steps": len(samples), "wall_s": t + cal["step_s"], "threads": nthreads}


def oracle_sample_desc(r: dict) -> str:
    return ("oracle on a bounded sample of the rag_mix step, measured (not extrapolated): "
            "per sample the merge of all 2,048 queries, the fp64 top-10 of %d of the %d "
            "merged queries over the full 1,048,576 x 768 corpus (%d threads), their fan-out, "
            "and the merge of %d of the 65,536 chunk rows (the same share; 1 thread); %d "
            "sample(s), %.1f s of host time" % (r["S"], r["merged_total"], r["threads"],
                                                r["chunk_rows"], r["steps"], r["wall_s"]))


def reference_arm(args, rank: int, world: int) -> int:
    """The oracle, as it stands, timed on the host cores (reference arm)."""
    if rank != 0:
        return 0
    w = build_workload(args.seed)
    nthreads = os.cpu_count() or 1
    per_step = max(2.0, 150.0 / max(1, args.steps + args.warmup))
    cal = oracle_step(w, nthreads, nthreads)
    S = max(nthreads, int(per_step / (cal["step_s"] / cal["merged"])))
    for _ in range(args.warmup):
        oracle_step(w, S, nthreads)
    samples = [oracle_step(w, S, nthreads) for _ in range(args.steps)]
    t = sum(x["step_s"] for x in samples)
    value = sum(x["merged"] for x in samples) / t
    r = {"S": S, "merged_total": samples[0]["merged_total"], "threads": nthreads,
         "chunk_rows": samples[0]["chunk_rows"], "steps": len(samples), "wall_s": t}
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t / len(samples),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": WORKLOAD, "seed": args.seed,
                       "sample": "each step is one bounded sample of the rag_mix step"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": nthreads, "kind": "oracle",
                             "cpu": cpu_model(), "sample": oracle_sample_desc(r)},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- GPU arm
def gpu_arm(args, rank: int, local_rank: int, world: int) -> int:
    import numpy as np
    import torch

    import paper_2607_22578_gb300 as hs

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peaks_kind = load_peaks()
    w = build_workload(args.seed)

    def to_dev(a):
        a = np.ascontiguousarray(a)
        if a.dtype == np.uint16:
            return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)
        return torch.from_numpy(a).to(dev)

    corpus = to_dev(w["corpus"])
    tokens = to_dev(w["tokens"])
    queries = to_dev(w["queries"])
    N, d = corpus.shape
    k = w["k"]
    n_chunk, n_q = tokens.shape[0], queries.shape[0]
    stage = hs.EmbedRetrieveStage(corpus, k, max_queries=n_q, max_chunk_rows=n_chunk)

    def step(ev=None):
        return stage.step(tokens, queries, events=ev)[1]

    for _ in range(args.warmup):
        _, _, nu_dev = step()
    hs.hs_get_device_error()
    n_u = int(nu_dev.item())

    K = args.steps
    # (1) Eager steps, with events around each retrieval launch: the
    # dominant kernel's time for the roofline.
    rev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(K)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    start.record()
    for i in range(K):
        step(rev[i])
    end.record()
    torch.cuda.synchronize()
    barrier(world)
    hs.hs_get_device_error()
    eager_ms, _ = reduce_over_ranks(start.elapsed_time(end), float(n_u * K), world)
    ret_ms = statistics.mean(a.elapsed_time(b) for a, b in rev)

    # (2) The headline: the same step captured once as a CUDA graph and
    # replayed K times (every replay runs every kernel of the step).
    graph = stage.capture(tokens, queries)
    for _ in range(args.warmup):
        graph.replay()
    clocks = ClockSampler(local_rank)
    clocks.start()
    barrier(world)
    torch.cuda.synchronize()
    start.record()
    for i in range(K):
        graph.replay()
    end.record()
    torch.cuda.synchronize()
    barrier(world)
    launches = graph.launches * K
    clk = clocks.stop()
    hs.hs_get_device_error()
    ms_local = start.elapsed_time(end)
    ms, merged_total = reduce_over_ranks(ms_local, float(n_u * K), world)
    ms_step = ms / K
    value = merged_total / (ms / 1e3)
    rows_total = (n_chunk + n_q) * K * world

    breakdown = rag_mix_breakdown(stage, tokens, queries, min(K, 50)) if args.breakdown else None

    # End to end through the public API: every step copies its inputs from
    # pinned host memory and its scores and ids back, and the host reads
    # each step's results (HostFeed overlaps step i+1's input copy with
    # step i's kernels; the host reads step i's results after submitting
    # step i+1).
    h_tokens = torch.from_numpy(w["tokens"]).pin_memory()
    h_queries = torch.from_numpy(w["queries"].view(np.int16)).pin_memory()
    feed = hs.HostFeed(stage, n_chunk, tokens.shape[1], n_q)
    Ke = max(1, min(K, 100))

    def e2e_run(steps):
        prev, nu = None, 0
        for _ in range(steps):
            slot = feed.submit(h_tokens, h_queries)
            if prev is not None:
                nu += feed.fetch(prev)[2]
            prev = slot
        nu += feed.fetch(prev)[2]
        return nu

    e2e_run(3)
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    feed.copy_stream.wait_stream(torch.cuda.current_stream())   # no copy before e0
    nu_total = e2e_run(Ke)
    e1.record()
    torch.cuda.synchronize()
    barrier(world)
    ems, emerged = reduce_over_ranks(e0.elapsed_time(e1), float(nu_total), world)
    e2e_value = emerged / (ems / 1e3)
    h2d = h_tokens.numel() * 4 + h_queries.numel() * 2
    d2h = feed.h_s[0].numel() * 4 + feed.h_i[0].numel() * 4 + 4

    flops = 2.0 * n_u * N * d
    achieved = flops / (ret_ms / 1e3) / 1e12
    peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    peak_s = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    traffic = traffic_from_profiles(
        "retrieve_kernel", os.path.join(ROOT, "paper_2607_22578_gb300", "csrc", "retrieve.cu"))

    # The other workloads' figures, measured in the same process after the
    # headline (rank 0): the dedup-heavy merge (fingerprint, unique/inverse,
    # scatter against HBM), batch-sweep latencies and the large-corpus
    # retrieval (k = 100).
    extras = {}
    if rank == 0 and not args.no_extras:
        del graph, feed, stage, corpus, tokens, queries, h_tokens, h_queries
        import gc
        gc.collect()
        torch.cuda.empty_cache()
        extras["dedup_heavy"] = row_dedup_heavy(args, dev, peaks)
        extras["batch_sweep"] = row_batch_sweep(args, dev, peaks, batches=(1, 64, 512))
        torch.cuda.empty_cache()
        extras["large_corpus"] = row_large_corpus(args, dev, peaks)
        gc.collect()
        torch.cuda.empty_cache()

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {
                "workload": WORKLOAD, "seed": args.seed, "queries_per_step": n_q,
                "merged_queries_per_step": n_u, "chunk_rows_per_step": n_chunk,
                "corpus_rows": N, "dim": d, "k": k,
                "l2": "inputs larger than L2: the 1.61 GB corpus streamed by every step "
                      "evicts the 129 MB L2 between steps",
                "parallelism": "replicas: one independent stage per GPU (no exchange step)"},
            "queries_served_per_s": n_q * K * world / (ms / 1e3),
            "rows_merged_per_s": rows_total / (ms / 1e3),
            # Peak: the measured burst bf16 figure.  The timed region is short
            # (K steps of ~1.5 ms) and the sampled SM clock stays near its
            # maximum, so the burst peak is the bar; the fraction of the
            # sustained (power-capped) peak is given beside it.
            "roofline": {
                "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "traffic": traffic,
                "kernel": "hs_retrieve_topk (retrieve_kernel + merge_warp_kernel), %.3f ms/launch"
                          % ret_ms,
                "algorithmic": "2 * %d merged queries * %d rows * %d dims = %.4g FLOP/launch"
                               % (n_u, N, d, flops),
                "peak_source": ("%s bf16 burst (MEASURED_PEAKS.json)" % peaks_kind
                                if peaks_kind == "measured" else "fallback bf16 burst"),
                "frac_of_sustained": achieved / peak_s},
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "steps": Ke},
            "gpu_launches": int(launches),
            "eager_ms_per_step": eager_ms / K,
            "clocks": clk,
        }
        line.update(extras)
        if breakdown is not None:
            line["breakdown_ms"] = breakdown
        if world == 1 and not args.no_cpu_baseline:
            nthreads = os.cpu_count() or 1
            ob = oracle_measured(w, args.cpu_budget, nthreads)
            line["cpu_baseline"] = {
                "value": ob["value"], "unit": UNIT, "cores": nthreads, "kind": "oracle",
                "cpu": cpu_model(), "sample": oracle_sample_desc(ob)}
        print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- per-row measurements
# These print one JSON line per workload for the other rows of the hot-path
# table (dedup-heavy dedup + scatter, the batch sweep, the large corpus) and a
# per-phase breakdown of the RAG-mix step.  They are measurement aids beside
# the contract line above, not the headline.
def _dev_array(a, dev):
    import numpy as np
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)
    return torch.from_numpy(a).to(dev)


def _ev():
    import torch
    return torch.cuda.Event(enable_timing=True)


def _roof(bytes_=None, flops=None, ms=None, peaks=None):
    out = {"ms": ms}
    if bytes_ is not None:
        gbs = bytes_ / (ms / 1e3) / 1e9
        out.update(bytes=bytes_, gbs=gbs, frac_hbm=gbs / peaks["hbm_gbs"])
    if flops is not None:
        tf = flops / (ms / 1e3) / 1e12
        out.update(flops=flops, tflops=tf, frac_tensor=tf / peaks["bf16_tflops"])
    return out


def row_dedup_heavy(args, dev, peaks) -> dict:
    """Dedup-heavy: fingerprint + unique/inverse + scatter of a 1536-byte
    payload per unique row back to all 400,000 rows."""
    import numpy as np
    import torch

    import paper_2607_22578_gb300 as hs
    import synth
    from synth import configs
    w = configs.build_dedup_heavy(seed=args.seed)
    n = w["tokens"].shape[0]
    tokens, lens = _dev_array(w["tokens"], dev), _dev_array(w["lens"], dev)
    gu, gi = synth.partition_of(w["chunk_root"])
    n_u = len(gu)
    W = w["payload_bytes"]
    payload = torch.randint(0, 255, (n_u, W), dtype=torch.uint8, device=dev)
    fp = torch.empty(n, dtype=torch.int64, device=dev)
    ws = torch.empty(hs.hs_unique_inverse_workspace(n), dtype=torch.uint8, device=dev)
    outs = (torch.empty(1, dtype=torch.int32, device=dev),
            torch.empty(n, dtype=torch.int32, device=dev),
            torch.empty(n, dtype=torch.int32, device=dev))
    dst = torch.empty((n, W), dtype=torch.uint8, device=dev)
    # per-row priority contributions (Eq. 3), summed per merged node after the step
    phi = torch.rand(n, dtype=torch.float64, device=dev)
    phi_u = torch.empty(n, dtype=torch.float64, device=dev)
    K = max(1, args.steps)
    evs = [[_ev() for _ in range(5)] for _ in range(K)]

    def step(e=None):
        if e: e[0].record()
        hs.hs_fingerprint(tokens, lens, fp_out=fp)
        if e: e[1].record()
        hs.hs_unique_inverse(fp, tokens, lens, workspace=ws, out=outs)
        if e: e[2].record()
        hs.hs_scatter_results(payload, outs[2], dst=dst)
        if e: e[3].record()
        hs.hs_segment_sum(phi, outs[2], n, n_groups_dev=outs[0], out=phi_u)
        if e: e[4].record()

    for _ in range(args.warmup):
        step()
    hs.hs_get_device_error()
    torch.cuda.synchronize()
    for i in range(K):
        step(evs[i])
    torch.cuda.synchronize()
    hs.hs_get_device_error()
    assert int(outs[0].item()) == n_u
    t_fp = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    t_un = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    t_sc = statistics.mean(e[2].elapsed_time(e[3]) for e in evs)
    t_ss = statistics.mean(e[3].elapsed_time(e[4]) for e in evs)
    # The step's own time: the three calls back to back with no events
    # between them (events would keep each kernel from overlapping its
    # successor's launch), K steps between two events.
    def plain_step():
        hs.hs_fingerprint(tokens, lens, fp_out=fp)
        hs.hs_unique_inverse(fp, tokens, lens, workspace=ws, out=outs)
        hs.hs_scatter_results(payload, outs[2], dst=dst)

    e0, e1 = _ev(), _ev()
    e0.record()
    for _ in range(K):
        plain_step()
    e1.record()
    torch.cuda.synchronize()
    hs.hs_get_device_error()
    t_sep = e0.elapsed_time(e1) / K

    # The step as the stage runs it: hs_merge_rows (the fingerprint and the
    # merge in one call: chunk pass, tails fused with the table insert,
    # verify, resolve, scan, finalize) and the scatter after it.
    ws_m = torch.empty(hs.hs_merge_rows_workspace(n), dtype=torch.uint8, device=dev)
    mr_out = (fp, outs[0], outs[1], outs[2])

    def fused_step(e=None):
        if e: e[0].record()
        hs.hs_merge_rows(tokens, lens, workspace=ws_m, out=mr_out)
        if e: e[1].record()
        hs.hs_scatter_results(payload, outs[2], dst=dst)

    for _ in range(args.warmup):
        fused_step()
    torch.cuda.synchronize()
    hs.hs_get_device_error()
    mevs = [[_ev(), _ev()] for _ in range(K)]
    for i in range(K):
        fused_step(mevs[i])
    torch.cuda.synchronize()
    t_mr = statistics.mean(e[0].elapsed_time(e[1]) for e in mevs)
    e0.record()
    for _ in range(K):
        fused_step()
    e1.record()
    torch.cuda.synchronize()
    hs.hs_get_device_error()
    assert int(outs[0].item()) == n_u
    t_all = e0.elapsed_time(e1) / K
    cpu = None
    if not getattr(args, "no_cpu_baseline", False):
        # The oracle on the whole workload (a few seconds on one host core):
        # fingerprint, unique/inverse and the scatter of the 1536-byte rows.
        import oracle
        host_payload = payload.cpu().numpy()
        t0 = time.perf_counter()
        oracle.fingerprint(w["tokens"], w["lens"])
        _, oinv = oracle.unique_inverse(w["tokens"], w["lens"])
        oracle.scatter(host_payload, oinv)
        t_cpu = time.perf_counter() - t0
        cpu = {"value": n / t_cpu, "unit": "dedup rows/s", "cores": 1, "kind": "oracle",
               "cpu": cpu_model(),
               "sample": "all %d rows, measured: fingerprint + unique/inverse + scatter of "
                         "%d B rows, one host thread, %.2f s" % (n, W, t_cpu)}
    L = w["lens"].astype(np.int64)
    sizes = np.bincount(gi, minlength=n_u)
    multi = sizes[gi] > 1
    tok_bytes = 4 * int(L.sum())
    fp_bytes = tok_bytes + 4 * n + 8 * n
    un_bytes = 4 * int(L[multi].sum()) + 8 * n + 8 * n
    sc_bytes = n_u * W + n * W + 4 * n
    ss_bytes = 8 * n + 4 * n + 8 * n_u
    merge = _roof(fp_bytes + un_bytes, None, t_mr, peaks)
    # the lower bound: one pass over the valid tokens (+ lens, fp, outputs)
    merge["frac_hbm_one_pass"] = ((tok_bytes + 4 * n + 8 * n + 8 * n) / (t_mr / 1e3) / 1e9
                                  / peaks["hbm_gbs"])
    return {
        "workload": "dedup_heavy: 400,000 rows x 512 int32 (lens U[64,512], Zipf(1.1) over "
                    "100,000 distinct) -> %d unique; scatter %d B per row" % (n_u, W),
        "metric": "dedup rows/s (fingerprint + unique/inverse + scatter)",
        "value": n / (t_all / 1e3), "ms_per_step": t_all, "steps": K,
        "step": "hs_merge_rows + hs_scatter_results",
        "separate_calls_ms_per_step": t_sep,
        "separate_calls_ms_per_step_with_events": statistics.mean(e[0].elapsed_time(e[3])
                                                                  for e in evs),
        "kernels": {
            "hs_merge_rows": merge,
            "hs_fingerprint": _roof(fp_bytes, None, t_fp, peaks),
            "hs_unique_inverse": _roof(un_bytes, None, t_un, peaks),
            "hs_scatter_results": _roof(sc_bytes, None, t_sc, peaks),
            "hs_segment_sum": _roof(ss_bytes, None, t_ss, peaks)},
        "merge_bytes_note": "hs_merge_rows: the method bytes of the two calls it combines "
                            "(one pass over the valid tokens + the verify re-read of every row "
                            "in a group of size >= 2, + lens, fp, outputs); frac_hbm_one_pass "
                            "counts the lower bound, one pass over the valid tokens + lens, fp "
                            "and outputs",
        "segment_sum_note": "priority contribution per merged node (Eq. 3) over the same "
                            "inverse map, timed after the step and not part of its value; bytes: "
                            "phi (fp64) + inverse in, one fp64 per merged node out; the output "
                            "clear of the remaining %d entries is not counted" % (n - n_u),
        "bytes_note": "fingerprint: valid token bytes + lens + fp; unique: full-row verify "
                      "re-read of every row in a group of size >= 2 + fp in + unique_idx/inverse "
                      "out (sort scratch is L2-resident and not counted); scatter: unique rows "
                      "once + every destination row + map",
        "token_bytes_one_pass": tok_bytes,
        "cpu_baseline": cpu}


def row_read_ceiling(args, dev, peaks) -> dict:
    """What the dedup-heavy row layout costs to stream, with no hashing: the
    valid prefixes read by a warp per row (coalesced), by a lane per row (the
    fingerprint chunk kernel's pattern), and whole padded rows; beside them
    hs_fingerprint itself and a plain device copy of as many bytes."""
    import numpy as np
    import torch

    import paper_2607_22578_gb300 as hs
    from synth import configs
    w = configs.build_dedup_heavy(seed=args.seed)
    tokens, lens = _dev_array(w["tokens"], dev), _dev_array(w["lens"], dev)
    n, stride = w["tokens"].shape
    valid = 4 * int(w["lens"].astype(np.int64).sum())
    padded = 4 * n * stride
    ck = torch.zeros(1, dtype=torch.int32, device=dev)
    fp = torch.empty(n, dtype=torch.int64, device=dev)
    K = max(5, min(args.steps, 20))

    def timed(fn):
        for _ in range(3):
            fn()
        ts = []
        for _ in range(K):
            e0, e1 = _ev(), _ev()
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        return statistics.median(ts)

    out = {"workload": "read_ceiling: dedup_heavy rows, 400,000 x 512 int32, lens U[64,512] "
                       "(%.1f MB valid of %.1f MB padded)" % (valid / 1e6, padded / 1e6),
           "metric": "GB/s of the bytes each pattern must read", "steps": K, "patterns": {}}
    names = {0: "warp_per_row_16B", 1: "lane_per_row_32B", 2: "warp_per_row_full_padded_rows"}
    for pat in (0, 1, 2):
        for bps in (2, 4, 8):
            ms = timed(lambda: hs.hs_debug_stream_rows(tokens, lens, pat, ck, bps))
            out["patterns"]["%s/%d_blocks_per_sm" % (names[pat], bps)] = _roof(
                padded if pat == 2 else valid, None, ms, peaks)
    ms = timed(lambda: hs.hs_fingerprint(tokens, lens, fp_out=fp))
    out["hs_fingerprint"] = _roof(valid, None, ms, peaks)
    src = torch.empty(valid // 2, dtype=torch.uint8, device=dev)
    dst = torch.empty_like(src)
    ms = timed(lambda: dst.copy_(src))
    out["device_copy_same_bytes"] = _roof(valid, None, ms, peaks)
    out["note"] = ("rows are the dedup_heavy inputs (larger than L2); median of %d launches; "
                   "the copy reads and writes half the valid bytes each" % K)
    hs.hs_get_device_error()
    return out


def row_batch_sweep(args, dev, peaks, batches=None) -> dict:
    """Adaptive-batch sweep: latency p50/p99 and q/s per batch size against a
    2,097,152 x 768 corpus (every size of the sweep unless `batches` names
    some)."""
    import numpy as np
    import torch

    import paper_2607_22578_gb300 as hs
    from synth import configs
    cfg = configs.BATCH_SWEEP
    C = configs.sweep_corpus(seed=args.seed)
    corpus = _dev_array(C, dev)
    N, d = C.shape
    del C
    sizes = tuple(batches) if batches else cfg["batches"]
    stage = hs.EmbedRetrieveStage(corpus, cfg["k"], max_queries=max(sizes))
    out = {"workload": "batch_sweep: corpus 2,097,152 x 768 bf16, 20% in-batch duplicates, "
                       "k=10", "metric": "per-batch latency and queries/s", "batches": {}}
    for B in sizes:
        nb = 50 if B >= 4096 else 200
        batches = [_dev_array(configs.build_sweep_batch(B, seed=1000 + i)["queries"], dev)
                   for i in range(nb + 3)]
        lat, ret, nus = [], [], []
        for i, q in enumerate(batches):
            e0, e1, r0, r1 = _ev(), _ev(), _ev(), _ev()
            e0.record()
            _, _, nu_dev = stage.retrieve(q, (r0, r1))
            e1.record()
            torch.cuda.synchronize()
            nu = int(nu_dev.item())
            if i >= 3:
                lat.append(e0.elapsed_time(e1))
                ret.append(r0.elapsed_time(r1))
                nus.append(nu)
        # The same batches through the captured query path (one launch).
        graph = hs.RetrieveGraph(stage, B)
        glat = []
        for i, q in enumerate(batches):
            e0, e1 = _ev(), _ev()
            e0.record()
            graph.run(q)
            e1.record()
            torch.cuda.synchronize()
            if i >= 3:
                glat.append(e0.elapsed_time(e1))
        hs.hs_get_device_error()
        qu = float(np.mean(nus))
        t_ret = float(np.mean(ret))
        rb = 2.0 * N * d + 2.0 * qu * d + qu * cfg["k"] * 8
        out["batches"][str(B)] = {
            "merged_queries_mean": qu, "latency_ms_p50": float(np.percentile(lat, 50)),
            "latency_ms_p99": float(np.percentile(lat, 99)),
            "queries_per_s": B * len(lat) / (sum(lat) / 1e3),
            "graph_latency_ms_p50": float(np.percentile(glat, 50)),
            "graph_latency_ms_p99": float(np.percentile(glat, 99)),
            "graph_queries_per_s": B * len(glat) / (sum(glat) / 1e3),
            "retrieval": _roof(rb, 2.0 * qu * N * d, t_ret, peaks)}
        del batches
    return out


def row_large_corpus(args, dev, peaks) -> dict:
    """Large corpus: 4096 merged queries x 8,388,608 x 1024, k = 100."""
    import torch

    import paper_2607_22578_gb300 as hs
    from synth import configs
    cfg = dict(configs.LARGE_CORPUS)
    if args.k:
        cfg["k"] = args.k
    if args.corpus_rows:
        cfg["N"] = args.corpus_rows
    w = configs.build_large_corpus(cfg, seed=args.seed)
    corpus, queries = _dev_array(w["corpus"], dev), _dev_array(w["queries"], dev)
    N, d = corpus.shape
    Q, k = queries.shape[0], w["k"]
    del w
    ws = torch.empty(hs.hs_retrieve_topk_workspace(Q, N, d, k), dtype=torch.uint8, device=dev)
    outs = (torch.empty((Q, k), dtype=torch.float32, device=dev),
            torch.empty((Q, k), dtype=torch.int32, device=dev))
    for _ in range(2):
        hs.hs_retrieve_topk(queries, corpus, k, workspace=ws, out=outs)
    torch.cuda.synchronize()
    K = max(1, min(args.steps, 10))
    e0, e1 = _ev(), _ev()
    e0.record()
    for _ in range(K):
        hs.hs_retrieve_topk(queries, corpus, k, workspace=ws, out=outs)
    e1.record()
    torch.cuda.synchronize()
    hs.hs_get_device_error()
    ms = e0.elapsed_time(e1) / K
    return {"workload": "large_corpus: %d merged queries x %d x %d bf16 "
                        "(1024 planted clusters), k=%d" % (Q, N, d, k),
            "metric": "merged queries/s", "value": Q / (ms / 1e3), "steps": K,
            "retrieval": _roof(2.0 * N * d, 2.0 * Q * N * d, ms, peaks)}


def row_rerank(args, dev, peaks) -> dict:
    """RAG with rerank (Section 4.1): the merged RAG-mix queries retrieve
    their top-12 from the 1,048,576 x 768 corpus, then a second stage
    rescores those 12 with 1024-dim rerank vectors and keeps the top-8."""
    import torch

    import paper_2607_22578_gb300 as hs
    from synth import configs
    w = configs.build_retrieval_mix(configs.RAG_MIX, seed=args.seed)
    rows = args.corpus_rows or w["corpus"].shape[0]     # a smaller corpus for captures
    corpus = _dev_array(w["corpus"][:rows], dev)
    q = _dev_array(w["queries"], dev)
    N, d = corpus.shape
    Q = q.shape[0]
    del w
    d2, k1, k2 = 1024, 12, 8
    g = torch.Generator(device=dev).manual_seed(args.seed + 17)
    rc = torch.nn.functional.normalize(torch.randn(N, d2, device=dev, generator=g), dim=1)
    rc = rc.to(torch.bfloat16)
    rq_all = torch.nn.functional.normalize(torch.randn(Q, d2, device=dev, generator=g), dim=1)
    rq_all = rq_all.to(torch.bfloat16)
    _, nu, uidx, inv, uq = hs.hs_merge_queries(q) if Q <= hs.HS_MERGE_QUERIES_MAX else (None,) * 5
    if nu is None:
        fp = hs.hs_fingerprint(q.view(torch.int32))
        nu, uidx, inv = hs.hs_unique_inverse(fp, q.view(torch.int32))
        uq = hs.hs_scatter_results(q, uidx)
    rq = hs.hs_scatter_results(rq_all, uidx)            # rerank vectors of the merged queries
    s12, i12 = hs.hs_retrieve_topk_n(uq, nu, corpus, k1)
    torch.cuda.synchronize()
    Qu = int(nu.item())
    outs = (torch.empty((Q, k2), dtype=torch.float32, device=dev),
            torch.empty((Q, k2), dtype=torch.int32, device=dev))
    for _ in range(3):
        hs.hs_rerank_topk(rq, rc, i12, k2, n_queries_dev=nu, inverse=inv, out=outs)
    torch.cuda.synchronize()
    # the candidate rows of one launch (~50 MB) fit in L2: flush it between
    # the timed launches by reading 256 MB (clean lines: evicting them costs
    # the timed launch no write-back) so each launch reads from HBM
    flush = torch.ones(64 << 20, dtype=torch.float32, device=dev)
    K = max(3, min(args.steps, 50))
    times = []
    for _ in range(K):
        flush.max()
        e0, e1 = _ev(), _ev()
        e0.record()
        hs.hs_rerank_topk(rq, rc, i12, k2, n_queries_dev=nu, inverse=inv, out=outs)
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    hs.hs_get_device_error()
    ms = statistics.median(times)
    # every output row gathers its query's k1 candidate rows (merged
    # duplicates re-read rows that are then in L2)
    bytes_ = Q * (k1 * d2 * 2 + d2 * 2 + k1 * 4 + 4 + k2 * 8)
    return {"workload": "rerank: %d queries (%d merged), top-%d of a %d x %d corpus rescored "
                        "with %d-dim rerank vectors (%d x %d bf16), top-%d kept"
                        % (Q, Qu, k1, N, d, d2, N, d2, k2),
            "metric": "reranked queries/s", "value": Q / (ms / 1e3), "steps": K,
            "kernels": {"hs_rerank_topk": _roof(bytes_, None, ms, peaks)},
            "l2": "flushed before every timed launch by a 256 MB read (median of %d)" % K,
            "bytes_note": "per output row: k1 candidate rows + the rerank query row + "
                          "candidate ids + map entry + k2 results"}


def row_cache(args, dev, peaks) -> dict:
    """Cross-batch reuse (Section 3.3 (II)): a stream of RAG-mix-sized
    batches whose queries repeat across batches (Zipf(1.1) over a pool of
    distinct queries), retrieved against the 1,048,576 x 768 corpus with and
    without the result cache."""
    import numpy as np
    import torch

    import paper_2607_22578_gb300 as hs
    import synth
    from synth import configs
    cfg = configs.RAG_MIX
    corpus = _dev_array(configs.build_retrieval_mix(cfg, seed=args.seed)["corpus"], dev)
    N, d = corpus.shape
    B, pool_n, n_batches, k = 2048, 50_000, 24, cfg["k"]
    pool = synth.unit_rows(pool_n, d, args.seed + 31)
    rng = np.random.default_rng(args.seed + 32)
    p = np.arange(1, pool_n + 1, dtype=np.float64) ** -1.1
    p /= p.sum()
    batches = [_dev_array(pool[rng.choice(pool_n, B, p=p)], dev) for _ in range(n_batches)]
    out = {"workload": "cache: %d batches x %d queries drawn Zipf(1.1) from %d distinct, "
                       "corpus %d x %d, k=%d" % (n_batches, B, pool_n, N, d, k),
           "metric": "queries/s over the batch stream", "arms": {}}
    for name, cap in (("no_cache", 0), ("cache_65536", 65536)):
        stage = hs.EmbedRetrieveStage(corpus, k, max_queries=B, cache_capacity=cap)
        stage.retrieve(batches[0])                      # builds the kernels' state once
        torch.cuda.synchronize()
        if cap:
            stage.cache.mem.zero_()
            hs.hs_cache_init(stage.cache)
        e0, e1 = _ev(), _ev()
        e0.record()
        for qb in batches:
            stage.retrieve(qb)
        e1.record()
        torch.cuda.synchronize()
        hs.hs_get_device_error()
        ms = e0.elapsed_time(e1)
        arm = {"ms_total": ms, "queries_per_s": B * n_batches / (ms / 1e3)}
        if cap:
            h, m = stage.cache_stats()
            arm.update(hits=h, misses=m, hit_rate=h / max(h + m, 1))
        out["arms"][name] = arm
        del stage
    out["value"] = out["arms"]["cache_65536"]["queries_per_s"]
    out["speedup_vs_no_cache"] = (out["arms"]["cache_65536"]["queries_per_s"] /
                                  out["arms"]["no_cache"]["queries_per_s"])
    return out


def rag_mix_breakdown(stage, tokens, queries, K: int) -> dict:
    """Per-phase device time of the RAG-mix step (the same calls as the
    pipeline, with events between them)."""
    import torch

    import paper_2607_22578_gb300 as hs
    from paper_2607_22578_gb300 import _lib
    names = ["chunk_merge", "chunk_merge_", "query_fingerprint", "query_unique",
             "gather_unique_queries", "retrieve_topk_fanout"]
    acc = {n: 0.0 for n in names}
    Q = queries.shape[0]
    for _ in range(K):
        ev = [_ev() for _ in range(len(names) + 1)]
        ev[0].record()
        stage.dedup_chunks(tokens)
        ev[1].record()
        ev[2].record()
        qi32 = queries.view(torch.int32)
        qfp = _lib.hs_fingerprint(qi32, fp_out=stage.q_fp[:Q])
        ev[3].record()
        nu, uidx, inv = _lib.hs_unique_inverse(qfp, qi32, workspace=stage.ws_q, out=stage.q_out)
        ev[4].record()
        uq = _lib.hs_scatter_results(queries, uidx, dst=stage.uq[:Q])
        ev[5].record()
        _lib.hs_retrieve_topk_fanout(uq, nu, inv, stage.corpus, stage.k, workspace=stage.ws_r,
                                     out=(stage.scores[:Q], stage.ids[:Q]))
        ev[6].record()
        torch.cuda.synchronize()
        for i, n in enumerate(names):
            acc[n] += ev[i].elapsed_time(ev[i + 1])
    hs.hs_get_device_error()
    out = {n: v / K for n, v in acc.items()}
    out.pop("chunk_merge_")
    return out


def rows_arm(args) -> int:
    import torch
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    peaks, kind = load_peaks()
    fn = {"dedup_heavy": row_dedup_heavy, "batch_sweep": row_batch_sweep,
          "large_corpus": row_large_corpus, "rerank": row_rerank,
          "cache": row_cache, "read_ceiling": row_read_ceiling}[args.workload]
    line = fn(args, dev, peaks)
    line["peaks"] = {"hbm_gbs": peaks["hbm_gbs"], "bf16_tflops": peaks["bf16_tflops"],
                     "source": kind}
    print(json.dumps(line), flush=True)
    return 0


def main() -> int:
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-budget", type=float, default=20.0,
                    help="seconds of host time for the oracle baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the dedup-heavy and batch-sweep figures of the default line")
    ap.add_argument("--workload", default="rag_mix",
                    choices=["rag_mix", "dedup_heavy", "batch_sweep", "large_corpus", "rerank",
                             "cache", "read_ceiling"],
                    help="rag_mix is the headline step; the others measure the other "
                         "rows of the hot-path table (one GPU)")
    ap.add_argument("--k", type=int, default=0, help="override k (large_corpus only)")
    ap.add_argument("--corpus-rows", type=int, default=0,
                    help="override the corpus size (large_corpus and rerank; for profiling)")
    ap.add_argument("--breakdown", action="store_true",
                    help="add per-phase device times of the rag_mix step")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank, local_rank, world = dist_env()
    if world != args.gpus and world > 1:
        print("warning: WORLD_SIZE=%d differs from --gpus %d" % (world, args.gpus),
              file=sys.stderr)
    if args.gpus > 1 and world == 1:
        ap.error("--gpus > 1 runs under torchrun (one process per GPU)")
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if (args.impl == "gb300" and torch.cuda.is_available()) else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local_rank)
        dist.init_process_group(backend=backend)
    try:
        if args.impl == "reference":
            return reference_arm(args, rank, world)
        if args.workload != "rag_mix":
            return rows_arm(args) if rank == 0 else 0
        return gpu_arm(args, rank, local_rank, world)
    finally:
        if world > 1:
            import torch.distributed as dist
            if dist.is_initialized():
                dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
