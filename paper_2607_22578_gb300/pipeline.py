"""The whole embed-and-retrieve stage for one batch of concurrent workflows.

Composition of the C-ABI calls only (no arithmetic here):
  chunks:  hs_fingerprint -> hs_unique_inverse      (merge duplicate chunk nodes)
  queries: hs_fingerprint -> hs_unique_inverse      (merge duplicate query nodes,
           -> hs_scatter_results (gather unique)     Section 3.3 (I))
           -> hs_retrieve_topk                      (one retrieval per merged node)
           -> hs_scatter_results (fan results back to every originating query)
The single host synchronisation is the read of the unique-query count, which
sizes the retrieval launch.
"""
from __future__ import annotations

import torch

from . import _lib


class EmbedRetrieveStage:
    """Holds the resident corpus and reusable workspaces for repeated batches."""

    def __init__(self, corpus: torch.Tensor, k: int, max_queries: int,
                 max_chunk_rows: int = 0):
        if not corpus.is_cuda:
            raise TypeError("corpus must be resident on the GPU")
        self.corpus = corpus
        self.k = int(k)
        self.N, self.d = corpus.shape
        dev = corpus.device
        self.device = dev
        self.max_queries = int(max_queries)
        self.ws_q = torch.empty(_lib.hs_unique_inverse_workspace(max_queries), dtype=torch.uint8,
                                device=dev)
        self.ws_r = torch.empty(_lib.hs_retrieve_topk_workspace(max_queries, self.N, self.d, k),
                                dtype=torch.uint8, device=dev)
        self.ws_c = torch.empty(_lib.hs_unique_inverse_workspace(max(max_chunk_rows, 1)),
                                dtype=torch.uint8, device=dev)
        self.q_out = (torch.empty(1, dtype=torch.int32, device=dev),
                      torch.empty(max_queries, dtype=torch.int32, device=dev),
                      torch.empty(max_queries, dtype=torch.int32, device=dev))
        self.c_out = (torch.empty(1, dtype=torch.int32, device=dev),
                      torch.empty(max(max_chunk_rows, 1), dtype=torch.int32, device=dev),
                      torch.empty(max(max_chunk_rows, 1), dtype=torch.int32, device=dev))
        self.launches = 0

    def dedup_chunks(self, tokens: torch.Tensor, lens: torch.Tensor | None = None):
        """Fingerprint + exact unique of chunk rows.  Returns (n_unique_dev,
        unique_idx, inverse, fp)."""
        fp = _lib.hs_fingerprint(tokens, lens)
        nu, uidx, inv = _lib.hs_unique_inverse(fp, tokens, lens, workspace=self.ws_c,
                                               out=self.c_out)
        return nu, uidx, inv, fp

    def retrieve(self, queries: torch.Tensor, events: tuple | None = None):
        """Merged retrieval of a query batch.  Returns (scores [Q, k],
        ids [Q, k], n_unique) for every original query.  If ``events`` is a
        pair of CUDA events they are recorded on the current stream around
        the hs_retrieve_topk launch (kernel timing for the roofline)."""
        Q, d = queries.shape
        if Q > self.max_queries:
            raise ValueError("batch larger than max_queries")
        qi32 = queries.view(torch.int32)
        fp = _lib.hs_fingerprint(qi32)
        nu, uidx, inv = _lib.hs_unique_inverse(fp, qi32, workspace=self.ws_q, out=self.q_out)
        n_unique = int(nu.item())                     # the one host synchronisation
        uq = _lib.hs_scatter_results(queries, uidx[:n_unique])
        if events is not None:
            events[0].record()
        s_u, i_u = _lib.hs_retrieve_topk(uq, self.corpus, self.k, workspace=self.ws_r)
        if events is not None:
            events[1].record()
        scores = _lib.hs_scatter_results(s_u, inv)
        ids = _lib.hs_scatter_results(i_u, inv)
        return scores, ids, n_unique
