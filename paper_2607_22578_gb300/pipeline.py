"""The whole embed-and-retrieve stage for one batch of concurrent workflows.

Composition of the C-ABI calls only (no arithmetic here):
  chunks:  hs_merge_rows                            (fingerprint + merge of duplicate
                                                     chunk nodes)
  queries: hs_merge_queries                         (merge duplicate query nodes,
             (batches up to HS_MERGE_QUERIES_MAX;    Section 3.3 (I): fingerprint,
              larger ones: hs_merge_rows ->           unique and gather in one
              hs_scatter_results gathering the        launch)
              unique rows)
           -> hs_retrieve_topk_fanout               (one retrieval per merged node,
                                                     results written to every
                                                     originating query)
  cached:  hs_cache_lookup -> hs_retrieve_topk_n of the misses -> hs_cache_insert
           -> hs_scatter_results (results reused across batches, Section 3.3 (II))
  rerank:  hs_retrieve_topk_n -> hs_scatter_results (rerank vectors of the
           merged queries) -> hs_rerank_topk        (top-k rescored, best kept,
                                                     fanned out; Section 4.1)
Nothing here synchronises with the host: the merged-query count stays in
device memory (the retrieval reads it when its kernels run), and the
unique-index tail beyond that count is a valid row map, so the gather can
always cover the whole batch.  Buffers are allocated once per stage.
"""
from __future__ import annotations

import torch

from . import _lib


class EmbedRetrieveStage:
    """Holds the resident corpus and reusable buffers for repeated batches."""

    def __init__(self, corpus: torch.Tensor, k: int, max_queries: int,
                 max_chunk_rows: int = 0, rerank_corpus: torch.Tensor | None = None,
                 rerank_k: int = 0, cache_capacity: int = 0):
        if not corpus.is_cuda:
            raise TypeError("corpus must be resident on the GPU")
        self.corpus = corpus
        self.k = int(k)
        self.N, self.d = corpus.shape
        dev = corpus.device
        self.device = dev
        self.max_queries = int(max_queries)
        mq, mc = self.max_queries, max(int(max_chunk_rows), 1)
        i32 = dict(dtype=torch.int32, device=dev)
        self.ws_q = torch.empty(_lib.hs_merge_rows_workspace(mq), dtype=torch.uint8, device=dev)
        self.ws_r = torch.empty(_lib.hs_retrieve_topk_workspace(mq, self.N, self.d, k),
                                dtype=torch.uint8, device=dev)
        self.ws_c = torch.empty(_lib.hs_merge_rows_workspace(mc), dtype=torch.uint8, device=dev)
        self.q_out = (torch.empty(1, **i32), torch.empty(mq, **i32), torch.empty(mq, **i32))
        self.c_out = (torch.empty(1, **i32), torch.empty(mc, **i32), torch.empty(mc, **i32))
        self.q_fp = torch.empty(mq, dtype=torch.int64, device=dev)
        self.c_fp = torch.empty(mc, dtype=torch.int64, device=dev)
        self.uq = torch.empty((mq, self.d), dtype=corpus.dtype, device=dev)
        self.scores = torch.empty((mq, self.k), dtype=torch.float32, device=dev)
        self.ids = torch.empty((mq, self.k), **i32)
        # results reused across batches (Section 3.3 (II)): merged queries
        # found in the cache skip retrieval
        self.cache = None
        if cache_capacity > 0:
            self.cache = _lib.ResultCache(cache_capacity, self.d, self.k, device=dev)
            self.miss = (torch.empty(mq, **i32), torch.empty(1, **i32),
                         torch.empty((mq, self.d), dtype=corpus.dtype, device=dev))
            self.m_s = torch.empty((mq, self.k), dtype=torch.float32, device=dev)
            self.m_i = torch.empty((mq, self.k), **i32)
            self.c_s = torch.empty((mq, self.k), dtype=torch.float32, device=dev)
            self.c_i = torch.empty((mq, self.k), **i32)
        # second stage (RAG with rerank): k candidates rescored, rerank_k kept
        self.rerank_corpus, self.rerank_k = rerank_corpus, int(rerank_k)
        if rerank_corpus is not None:
            if not rerank_corpus.is_cuda or rerank_corpus.shape[0] != self.N:
                raise ValueError("rerank_corpus must be on the GPU, one row per corpus row")
            if not 1 <= self.rerank_k <= self.k:
                raise ValueError("need 1 <= rerank_k <= k")
            self.s_u = torch.empty((mq, self.k), dtype=torch.float32, device=dev)
            self.i_u = torch.empty((mq, self.k), **i32)
            self.rq_u = torch.empty((mq, rerank_corpus.shape[1]), dtype=rerank_corpus.dtype,
                                    device=dev)
            self.r_scores = torch.empty((mq, self.rerank_k), dtype=torch.float32, device=dev)
            self.r_ids = torch.empty((mq, self.rerank_k), **i32)

    def capture(self, tokens: torch.Tensor, queries: torch.Tensor,
                lens: torch.Tensor | None = None) -> "StepGraph":
        """Capture ``step`` on these device buffers as a replayable CUDA graph."""
        return StepGraph(self, tokens, queries, lens)

    def dedup_chunks(self, tokens: torch.Tensor, lens: torch.Tensor | None = None):
        """Fingerprint + exact unique of chunk rows.  Returns (n_unique_dev,
        unique_idx, inverse, fp) as device tensors."""
        n = tokens.shape[0]
        nu_b, uidx_b, inv_b = self.c_out
        fp, nu, uidx, inv = _lib.hs_merge_rows(
            tokens, lens, workspace=self.ws_c, out=(self.c_fp[:n], nu_b, uidx_b[:n], inv_b[:n]))
        return nu, uidx, inv, fp

    def retrieve(self, queries: torch.Tensor, events: tuple | None = None):
        """Merged retrieval of a query batch.  Returns (scores [Q, k],
        ids [Q, k], n_unique_dev) for every original query; n_unique_dev is
        a one-element device tensor.  If ``events`` is a pair of CUDA events
        they are recorded on the current stream around the retrieval launch
        (kernel timing for the roofline)."""
        Q, d = queries.shape
        if Q > self.max_queries:
            raise ValueError("batch larger than max_queries")
        nu, inv, uq = self._merge_queries(queries)
        return self._retrieve_merged(uq, nu, inv, events) + (nu,)

    def _retrieve_cached(self, uq, nu, inv, events):
        """Lookup of the merged queries, retrieval of the misses only, insert
        of their results, fan-out to every query."""
        Q = inv.shape[0]
        fp, uidx = self.q_fp[:Q], self.q_out[1][:Q]
        out = (self.c_s[:Q], self.c_i[:Q])
        miss = (self.miss[0][:Q], self.miss[1], self.miss[2][:Q])
        _lib.hs_cache_lookup(self.cache, uq, fp, fp_rows=uidx, n_queries_dev=nu, out=out,
                             miss=miss)
        if events is not None:
            events[0].record()
        _lib.hs_retrieve_topk_n(miss[2], miss[1], self.corpus, self.k, workspace=self.ws_r,
                                out=(self.m_s[:Q], self.m_i[:Q]))
        if events is not None:
            events[1].record()
        _lib.hs_cache_insert(self.cache, miss, fp, self.m_s[:Q], self.m_i[:Q], out,
                             fp_rows=uidx)
        scores = _lib.hs_scatter_results(out[0], inv, dst=self.scores[:Q])
        ids = _lib.hs_scatter_results(out[1], inv, dst=self.ids[:Q])
        return scores, ids

    def cache_stats(self):
        """(hits, misses) of the result cache since the stage was built."""
        return _lib.hs_cache_stats(self.cache)

    def retrieve_rerank(self, queries: torch.Tensor, rerank_queries: torch.Tensor):
        """RAG with rerank (Section 4.1): merged retrieval of the top-k, then
        the k candidates of each merged query rescored with its rerank
        vector (the representative's row of ``rerank_queries``) and the best
        rerank_k kept, fanned out to every query.  Returns (scores [Q,
        rerank_k], ids [Q, rerank_k], n_unique_dev)."""
        if self.rerank_corpus is None:
            raise ValueError("stage built without a rerank corpus")
        Q = queries.shape[0]
        if Q > self.max_queries or rerank_queries.shape[0] != Q:
            raise ValueError("batch larger than max_queries or rerank rows differ")
        nu, inv, uq = self._merge_queries(queries)
        uidx = self.q_out[1][:Q]
        _lib.hs_retrieve_topk_n(uq, nu, self.corpus, self.k, workspace=self.ws_r,
                                out=(self.s_u[:Q], self.i_u[:Q]))
        rq = _lib.hs_scatter_results(rerank_queries, uidx, dst=self.rq_u[:Q])
        scores, ids = _lib.hs_rerank_topk(rq, self.rerank_corpus, self.i_u[:Q], self.rerank_k,
                                          n_queries_dev=nu, inverse=inv,
                                          out=(self.r_scores[:Q], self.r_ids[:Q]))
        return scores, ids, nu

    def _merge_queries(self, queries: torch.Tensor):
        """Merged query nodes of a batch: (n_unique_dev, inverse, unique
        query rows)."""
        Q = queries.shape[0]
        nu_b, uidx_b, inv_b = self.q_out
        if Q <= _lib.HS_MERGE_QUERIES_MAX:
            _, nu, _, inv, uq = _lib.hs_merge_queries(
                queries, out=(self.q_fp[:Q], nu_b, uidx_b[:Q], inv_b[:Q], self.uq[:Q]))
            return nu, inv, uq
        qi32 = queries.view(torch.int32)
        _, nu, uidx, inv = _lib.hs_merge_rows(
            qi32, workspace=self.ws_q, out=(self.q_fp[:Q], nu_b, uidx_b[:Q], inv_b[:Q]))
        uq = _lib.hs_scatter_results(queries, uidx, dst=self.uq[:Q])
        return nu, inv, uq

    def _retrieve_merged(self, uq, nu, inv, events):
        Q = inv.shape[0]
        if self.cache is not None:
            return self._retrieve_cached(uq, nu, inv, events)
        if events is not None:
            events[0].record()
        scores, ids = _lib.hs_retrieve_topk_fanout(uq, nu, inv, self.corpus, self.k,
                                                   workspace=self.ws_r,
                                                   out=(self.scores[:Q], self.ids[:Q]))
        if events is not None:
            events[1].record()
        return scores, ids

    def step(self, tokens: torch.Tensor, queries: torch.Tensor,
             lens: torch.Tensor | None = None, events: tuple | None = None):
        """One batch of the whole stage.  The chunk merge and the query path
        are independent, so the chunk fingerprint + unique run on a side
        stream concurrently with the query fingerprint + unique, joined by an
        event before the retrieval.  Returns (chunk (n_unique_dev,
        unique_idx, inverse, fp), query (scores, ids, n_unique_dev))."""
        main = torch.cuda.current_stream(self.device)
        if not hasattr(self, "_side"):
            self._side = torch.cuda.Stream(device=self.device)
            self._fork = torch.cuda.Event()
            self._join = torch.cuda.Event()
        self._fork.record(main)
        self._side.wait_event(self._fork)
        with torch.cuda.stream(self._side):
            chunk = self.dedup_chunks(tokens, lens)
        self._join.record(self._side)
        if queries.shape[0] > self.max_queries:
            raise ValueError("batch larger than max_queries")
        nu, inv, uq = self._merge_queries(queries)
        main.wait_event(self._join)      # retrieval occupies every SM: chunk work first
        scores, ids = self._retrieve_merged(uq, nu, inv, events)
        return chunk, (scores, ids, nu)


class StepGraph:
    """One stage step captured as a CUDA graph on fixed device input buffers.

    ``replay()`` enqueues the whole step — both dedup paths, the gather, the
    retrieval and the result scatter, with the chunk path on its own branch —
    as one graph launch on the current stream, so the host issues one call
    instead of about twenty and the kernels follow each other without
    per-launch gaps.  Refill ``tokens``/``queries`` (the captured buffers) in
    place between replays; ``outputs`` are the stage's result buffers, which
    every replay overwrites."""

    def __init__(self, stage: "EmbedRetrieveStage", tokens: torch.Tensor,
                 queries: torch.Tensor, lens: torch.Tensor | None = None):
        self.tokens, self.queries, self.lens = tokens, queries, lens
        # One eager step first: one-time host work (kernel attributes,
        # occupancy queries) must not happen inside the capture.
        stage.step(tokens, queries, lens)
        torch.cuda.synchronize(stage.device)
        self.graph = torch.cuda.CUDAGraph()
        l0 = _lib.hs_launch_count()
        with torch.cuda.graph(self.graph):
            self.outputs = stage.step(tokens, queries, lens)
        self.launches = _lib.hs_launch_count() - l0   # kernels per replay

    def replay(self):
        self.graph.replay()
        return self.outputs


class RetrieveGraph:
    """The query path of a stage — fingerprint, unique, gather, retrieval,
    result scatter — captured as one CUDA graph for batches of exactly
    ``n_queries`` queries (serving pads batches to a few such sizes).

    ``run(queries)`` copies the batch into the captured input buffer and
    replays the graph: one launch for the whole path instead of one host
    call per kernel.  Returns the stage's (scores, ids, n_unique) buffers,
    which the next run overwrites."""

    def __init__(self, stage: "EmbedRetrieveStage", n_queries: int):
        if n_queries > stage.max_queries:
            raise ValueError("batch larger than the stage's max_queries")
        self.queries = torch.zeros((n_queries, stage.d), dtype=stage.corpus.dtype,
                                   device=stage.device)
        stage.retrieve(self.queries)           # one-time host work outside the capture
        torch.cuda.synchronize(stage.device)
        self.graph = torch.cuda.CUDAGraph()
        l0 = _lib.hs_launch_count()
        with torch.cuda.graph(self.graph):
            self.outputs = stage.retrieve(self.queries)
        self.launches = _lib.hs_launch_count() - l0

    def run(self, queries: torch.Tensor):
        self.queries.copy_(queries, non_blocking=True)
        self.graph.replay()
        return self.outputs


class HostFeed:
    """Runs batches that live in (pinned) host memory through a stage, with
    the next batch's host-to-device copy overlapping the current batch's
    kernels.

    Two device copies of the inputs alternate: batch i is copied on a copy
    stream into buffer i % 2 once batch i - 2 (the last user of that buffer)
    has finished, and the stage runs on the current stream after the copy.
    Each batch's scores and ids are copied back into their own pinned host
    buffers; ``fetch`` waits for that copy and returns them."""

    def __init__(self, stage: EmbedRetrieveStage, chunk_rows: int, chunk_stride: int,
                 n_queries: int, graphs: bool = True):
        dev = stage.device
        self.stage = stage
        self.copy_stream = torch.cuda.Stream(device=dev)
        self.d_tok = [torch.zeros((chunk_rows, chunk_stride), dtype=torch.int32, device=dev)
                      for _ in range(2)]
        self.d_q = [torch.zeros((n_queries, stage.d), dtype=stage.corpus.dtype, device=dev)
                    for _ in range(2)]
        # With graphs, each input buffer gets its captured step (nothing in a
        # step depends on the data on the host side, so replays serve any
        # contents of the buffers).
        self.graphs = ([stage.capture(self.d_tok[b], self.d_q[b]) for b in range(2)]
                       if graphs else None)
        self.h_s = [torch.empty((n_queries, stage.k), dtype=torch.float32).pin_memory()
                    for _ in range(2)]
        self.h_i = [torch.empty((n_queries, stage.k), dtype=torch.int32).pin_memory()
                    for _ in range(2)]
        self.h_nu = [torch.empty(1, dtype=torch.int32).pin_memory() for _ in range(2)]
        self.copied = [torch.cuda.Event() for _ in range(2)]
        self.freed = [torch.cuda.Event() for _ in range(2)]
        self.done = [torch.cuda.Event() for _ in range(2)]
        self.used = [False, False]
        self.count = 0

    def submit(self, h_tokens: torch.Tensor, h_queries: torch.Tensor) -> int:
        """Enqueue one batch (host tensors, pinned for an asynchronous copy).
        Returns its slot for ``fetch``.  The slot's previous results must
        have been fetched already."""
        b = self.count % 2
        self.count += 1
        main = torch.cuda.current_stream(self.stage.device)
        if self.used[b]:
            self.copy_stream.wait_event(self.freed[b])
        with torch.cuda.stream(self.copy_stream):
            _lib.hs_memcpy_async(self.d_tok[b], h_tokens, self.copy_stream)
            _lib.hs_memcpy_async(self.d_q[b], h_queries, self.copy_stream)
            self.copied[b].record(self.copy_stream)
        main.wait_event(self.copied[b])
        if self.graphs is not None:
            _, (s, i, nu) = self.graphs[b].replay()
        else:
            _, (s, i, nu) = self.stage.step(self.d_tok[b], self.d_q[b])
        self.freed[b].record(main)
        _lib.hs_memcpy_async(self.h_s[b], s, main)
        _lib.hs_memcpy_async(self.h_i[b], i, main)
        _lib.hs_memcpy_async(self.h_nu[b], nu, main)
        self.done[b].record(main)
        self.used[b] = True
        return b

    def fetch(self, slot: int):
        """Wait for a submitted batch; returns host (scores, ids, n_unique)."""
        self.done[slot].synchronize()
        return self.h_s[slot], self.h_i[slot], int(self.h_nu[slot][0])
