"""The five workload shapes of the embed-and-retrieve benchmark.

Each builder returns a dict of host numpy arrays plus the ground truth it
planted.  Sizes follow the workload table; ``scale`` shrinks row counts (not
widths) for fast CPU tests.  The shapes stand in for the paper's MS MARCO /
TruthfulQA traffic with 5-15% Zipfian duplicates (Section 4.1, "Workloads"),
which is not reproduced here.
"""
from __future__ import annotations

import numpy as np

from . import (chunks_with_copies, chunks_zipf, clustered_corpus, queries_near_centres,
               queries_with_copies, unit_rows)

# Static description (sizes at scale 1).
TINY = dict(name="tiny", n_workflows=4, q_per_wf=8, q_dup=0.25, chunk_rows=256,
            chunk_len=128, chunk_copy=0.50, chunk_cross=False, N=4096, d=384, k=10)
RAG_MIX = dict(name="rag_mix", n_workflows=64, q_per_wf=32, q_dup=0.30, chunk_rows=65536,
               chunk_len=256, chunk_copy=0.40, chunk_cross=True, N=1048576, d=768, k=10)
DEDUP_HEAVY = dict(name="dedup_heavy", n_workflows=256, rows=400000, stride=512,
                   pool=100000, zipf_s=1.1, len_lo=64, len_hi=512, payload_bytes=1536)
LARGE_CORPUS = dict(name="large_corpus", N=8388608, d=1024, n_clusters=1024, members=128,
                    sigma=0.05, nq=4096, k=100)
BATCH_SWEEP = dict(name="batch_sweep", N=2097152, d=768, batches=(1, 8, 64, 512, 4096),
                   q_dup=0.20, k=10)

CONFIGS = {c["name"]: c for c in (TINY, RAG_MIX, DEDUP_HEAVY, LARGE_CORPUS, BATCH_SWEEP)}


def _scaled(n: int, scale: float, lo: int = 1) -> int:
    return max(lo, int(round(n * scale)))


def build_retrieval_mix(cfg: dict, seed: int = 0, scale: float = 1.0,
                        corpus: bool = True) -> dict:
    """Tiny / RAG-mix: chunk rows with copies, queries with cross-workflow
    duplicates, and a unit-norm corpus."""
    nwf = cfg["n_workflows"]
    qpw = cfg["q_per_wf"]
    nq = nwf * qpw
    q, qroot = queries_with_copies(nq, cfg["d"], cfg["q_dup"], seed, block=qpw)
    rows = _scaled(cfg["chunk_rows"], scale, lo=nwf * 2)
    rows -= rows % nwf
    block = rows // nwf if cfg["chunk_cross"] else None
    tokens, croot = chunks_with_copies(rows, cfg["chunk_len"], cfg["chunk_copy"], seed,
                                       block=block)
    out = dict(queries=q, query_root=qroot, tokens=tokens, lens=None, chunk_root=croot,
               k=cfg["k"], d=cfg["d"], n_workflows=nwf)
    if corpus:
        out["corpus"] = unit_rows(_scaled(cfg["N"], scale, lo=max(64, cfg["k"])), cfg["d"],
                                  seed)
    return out


def build_dedup_heavy(cfg: dict = DEDUP_HEAVY, seed: int = 0, scale: float = 1.0) -> dict:
    rows = _scaled(cfg["rows"], scale, lo=16)
    pool = _scaled(cfg["pool"], scale, lo=4)
    tokens, lens, pidx = chunks_zipf(rows, cfg["stride"], pool, cfg["zipf_s"],
                                     cfg["len_lo"], cfg["len_hi"], seed)
    return dict(tokens=tokens, lens=lens, chunk_root=pidx,
                payload_bytes=cfg["payload_bytes"], n_workflows=cfg["n_workflows"])


def build_large_corpus(cfg: dict = LARGE_CORPUS, seed: int = 0, scale: float = 1.0) -> dict:
    N = _scaled(cfg["N"], scale, lo=cfg["n_clusters"] * cfg["members"] * 2)
    corpus, centres, members = clustered_corpus(N, cfg["d"], cfg["n_clusters"],
                                                cfg["members"], cfg["sigma"], seed)
    nq = _scaled(cfg["nq"], scale, lo=8)
    q, cl = queries_near_centres(nq, centres, cfg["sigma"], seed)
    return dict(corpus=corpus, queries=q, query_cluster=cl, members=members, k=cfg["k"],
                d=cfg["d"])


def build_sweep_batch(B: int, cfg: dict = BATCH_SWEEP, seed: int = 0) -> dict:
    """One batch of the adaptive-batch sweep: B queries, round(0.2 B) in-batch
    copies (no workflow structure)."""
    q, root = queries_with_copies(B, cfg["d"], cfg["q_dup"], seed, block=None)
    return dict(queries=q, query_root=root, k=cfg["k"], d=cfg["d"])


def sweep_corpus(cfg: dict = BATCH_SWEEP, seed: int = 0, scale: float = 1.0) -> np.ndarray:
    return unit_rows(_scaled(cfg["N"], scale, lo=64), cfg["d"], seed)
