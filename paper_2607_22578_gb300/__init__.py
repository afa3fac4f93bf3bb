"""GB300-native embed-and-retrieve hot path of HeraSys' cross-workflow node
merging: fingerprint, exact unique-with-inverse, tcgen05 retrieval with a
fused top-k, and result scatter — hand-written sm_103a CUDA behind the C ABI
in include/hs.h, called here through a thin ctypes binding."""
from ._lib import (HS_ERR_CUDA, HS_ERR_INVALID_ARG, HS_ERR_TIMEOUT, HS_ERR_UNSUPPORTED,
                   HS_ERR_WORKSPACE, HS_FNV64_OFFSET_BASIS, HS_MERGE_QUERIES_MAX, HS_OK,
                   HS_TOPK_MAX_K, HsError, hs_debug_merge_key_mask, hs_debug_retrieve_wait,
                   hs_debug_scan_wait,
                   hs_debug_stream_rows, hs_fingerprint, hs_merge_rows, hs_merge_rows_workspace, hs_get_device_error,
                   hs_launch_count, hs_memcpy_async, hs_merge_queries, hs_retrieve_topk, hs_retrieve_topk_fanout,
                   hs_retrieve_topk_n, hs_retrieve_topk_workspace, hs_scatter_results,
                   hs_rerank_topk, hs_segment_sum, ResultCache, hs_cache_bytes, hs_cache_init, hs_cache_insert,
                   hs_cache_lookup, hs_cache_stats,
                   hs_unique_inverse, hs_unique_inverse_noalloc, hs_unique_inverse_workspace,
                   hs_version, library_path, load)
from .pipeline import EmbedRetrieveStage, HostFeed, RetrieveGraph, StepGraph

__all__ = [
    "HS_OK", "HS_ERR_INVALID_ARG", "HS_ERR_UNSUPPORTED", "HS_ERR_CUDA", "HS_ERR_WORKSPACE",
    "HS_ERR_TIMEOUT", "HS_FNV64_OFFSET_BASIS", "HS_TOPK_MAX_K", "HS_MERGE_QUERIES_MAX",
    "HsError", "hs_fingerprint", "hs_unique_inverse", "hs_unique_inverse_noalloc",
    "hs_unique_inverse_workspace", "hs_retrieve_topk", "hs_retrieve_topk_n",
    "hs_retrieve_topk_fanout", "hs_merge_queries", "hs_retrieve_topk_workspace",
    "hs_scatter_results", "hs_rerank_topk", "hs_segment_sum", "ResultCache",
    "hs_cache_bytes", "hs_cache_init", "hs_cache_lookup", "hs_cache_insert", "hs_cache_stats", "hs_get_device_error", "hs_launch_count", "hs_memcpy_async",
    "hs_debug_scan_wait", "hs_debug_stream_rows", "hs_debug_merge_key_mask",
    "hs_debug_retrieve_wait", "hs_merge_rows",
    "hs_merge_rows_workspace", "hs_version",
    "library_path", "load", "EmbedRetrieveStage", "HostFeed", "RetrieveGraph", "StepGraph",
]
