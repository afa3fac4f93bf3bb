/*
 * hs.h — C ABI of the GB300 embed-and-retrieve hot path of HeraSys'
 * cross-workflow node merging.
 *
 * The stage has four steps, each one call:
 *   hs_fingerprint      hash every input row (chunk tokens or query vectors)
 *   hs_unique_inverse   merge exactly-equal rows into unique nodes + inverse map
 *   (hs_merge_rows      the two above in one pass over the rows)
 *   hs_retrieve_topk    score merged queries against a corpus, keep top-k
 *   hs_scatter_results  fan each kept result back out to every merged row
 * two fused forms for latency-bound batches:
 *   hs_merge_queries         fingerprint + merge + gather of a query batch
 *   hs_retrieve_topk_fanout  retrieval whose results go to every merged row
 * the second retrieval stage of the rerank workflow:
 *   hs_rerank_topk           rescore the retrieved candidates, keep the best
 * reuse of results across batches:
 *   hs_cache_lookup / hs_cache_insert   a device-resident result cache
 * and the scheduling weight of the merged nodes:
 *   hs_segment_sum           priority contribution of each fused node (Eq. 3)
 * and a batch's copies between host buffers and the device:
 *   hs_memcpy_async
 *
 * Conventions shared by every call
 *   - Pointers named *_dev or documented as device pointers must be device
 *     memory of the current CUDA device; the caller owns all of them
 *     (inputs, outputs and workspace).  The library allocates no device
 *     memory in any call.
 *   - Every call enqueues its kernels on `stream` (a cudaStream_t; NULL is
 *     the legacy default stream) and returns without synchronising.
 *   - Argument errors that the host can see are returned at once and nothing
 *     is enqueued; hs_last_error() then describes them.  Errors that only the
 *     device can see (a row length outside [0, row_stride], a map entry out
 *     of range, a bounded wait that ran out) set a per-device error word;
 *     hs_get_device_error() synchronises the stream and reports and clears it.
 *   - Unless stated otherwise, device pointers must be 16-byte aligned.
 *   - Calls on one stream run in order; calls on different streams that
 *     share an output or a workspace race.
 */
#ifndef HS_H_
#define HS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t / CUstream, without including CUDA headers. */
typedef struct CUstream_st* hs_stream_t;

typedef enum {
  HS_OK = 0,
  HS_ERR_INVALID_ARG = 1, /* bad size, pointer, alignment or (device) data  */
  HS_ERR_UNSUPPORTED = 2, /* valid request the library does not handle      */
  HS_ERR_CUDA = 3,        /* a CUDA runtime/driver call failed              */
  HS_ERR_WORKSPACE = 4,   /* workspace pointer NULL/misaligned or too small */
  HS_ERR_TIMEOUT = 5      /* a bounded device-side wait ran out             */
} hs_status;

/* FNV-1a 64-bit offset basis: the seed of a plain (unseeded) hash. */
#define HS_FNV64_OFFSET_BASIS 0xcbf29ce484222325ULL

/* Largest k accepted by hs_retrieve_topk. */
#define HS_TOPK_MAX_K 1024

/* Largest batch accepted by hs_merge_queries. */
#define HS_MERGE_QUERIES_MAX 256

/* Human-readable description of the last error returned on this host
 * thread ("" if none).  The string stays valid until the next hs_* call on
 * the same thread. */
const char* hs_last_error(void);

/* Library version string. */
const char* hs_version(void);

/*
 * hs_fingerprint — per-row node signature over the input data.
 *
 * Paper: Section 3.3, Eq. 2: Sig(v) = H(tau_v, Theta_p, D_in, ordered
 * combination of predecessor signatures).  This call computes the D_in part
 * with H = 64-bit FNV-1a over octets: for row i,
 *   fp[i] = FNV-1a(seed_state, little-endian octets of tokens[i, 0:len_i])
 * i.e. h = seed_state; for each octet b: h = (h xor b) * 1099511628211 mod 2^64.
 * tau_v, Theta_p and the predecessor signatures are folded in by the caller:
 * hash their canonical bytes first and pass the result as seed_state (FNV-1a
 * continues a byte stream exactly).  Pass HS_FNV64_OFFSET_BASIS for the
 * plain hash.
 *
 * tokens      device, int32 [n_rows, row_stride] row-major.  Query vectors are
 *             hashed by viewing their bf16 bits as int32 words (dim/2 words).
 * n_rows      >= 0 (0: nothing is enqueued).
 * row_stride  >= 0, words between consecutive rows.
 * lens        device int32 [n_rows] or NULL (every row has row_stride words).
 *             A length outside [0, row_stride] sets the device error word
 *             (HS_ERR_INVALID_ARG) and that row's fp is written as 0.
 * fp_out      device uint64 [n_rows], 8-byte aligned.
 * tokens needs only 4-byte alignment; 16-byte aligned tokens with
 * row_stride % 4 == 0 take the vector path.
 */
hs_status hs_fingerprint(const int32_t* tokens, int64_t n_rows, int32_t row_stride,
                         const int32_t* lens, uint64_t seed_state, uint64_t* fp_out,
                         hs_stream_t stream);

/*
 * hs_unique_inverse — exact merge of equal rows (node fusion).
 *
 * Paper: Section 3.3, "Dynamic Fusion and Reuse Mechanism" (I): a node that
 * matches a node already in the window is removed and its downstream edges
 * are redirected to the kept node; Appendix A.2, "Redundancy Elimination &
 * Result Sharing": merge sets M(v*) executed once.
 *
 * Rows i and j are equal iff len_i == len_j and tokens[i, 0:len] ==
 * tokens[j, 0:len] (words beyond len are ignored).  Outputs:
 *   *n_unique_dev      number of groups,
 *   unique_idx_out[u]  index of group u's first occurrence, ascending in u,
 *                      for u < *n_unique_dev; 0 for u >= *n_unique_dev, so
 *                      all n_rows entries form a valid row map,
 *   inverse_out[i]     group ordinal of row i (the redirected edge),
 * so rows[unique_idx[inverse[i]]] == rows[i].  fp must hold fingerprints of
 * these rows that are equal for equal rows (as hs_fingerprint produces with
 * one seed); different rows may share a fingerprint (a collision): they are
 * told apart by a full row comparison, never merged.  Cost is linear in the
 * row bytes of rows that have an equal-fingerprint predecessor, plus one hash
 * table insert and lookup per row.  Rows whose fingerprint equals an earlier
 * row's but whose contents differ (a collision) are regrouped by a second
 * hash of their contents and compared once more, in one thread block: linear
 * in their row bytes, so even a constant fp is exact at linear cost (slower
 * than distinct fingerprints, which spread the work over the whole GPU).
 * Only rows that collide in both hashes are compared pairwise.
 *
 * fp              device uint64 [n_rows], 8-byte aligned.
 * tokens, n_rows, row_stride, lens   as for hs_fingerprint;
 *                 1 <= ... n_rows <= 2^30 - 1 (0 writes *n_unique_dev = 0).
 * n_unique_dev    device int32 scalar.
 * unique_idx_out  device int32 [n_rows].
 * inverse_out     device int32 [n_rows].
 * workspace       device, >= hs_unique_inverse_workspace(n_rows) bytes,
 *                 256-byte aligned; contents on entry are ignored.
 */
size_t hs_unique_inverse_workspace(int64_t n_rows);
hs_status hs_unique_inverse(const uint64_t* fp, const int32_t* tokens, int64_t n_rows,
                            int32_t row_stride, const int32_t* lens, int32_t* n_unique_dev,
                            int32_t* unique_idx_out, int32_t* inverse_out, void* workspace,
                            size_t workspace_bytes, hs_stream_t stream);

/*
 * hs_merge_rows — hs_fingerprint and hs_unique_inverse in one pass over the
 * rows: node signatures and the exact merge of equal rows.
 *
 * Paper: Section 3.3, Eq. 2 (the signature of a node) and "Dynamic Fusion
 * and Reuse Mechanism" (I) (a node equal to one already in the window is
 * merged into it); Appendix A.2 (merge sets M(v*) executed once);
 * Appendix B.3, Phase 1 (duplicate detection by signature lookup).
 * The outputs are exactly those of
 *   hs_fingerprint(tokens, n_rows, row_stride, lens, seed_state, fp_out)
 *   hs_unique_inverse(fp_out, tokens, ..., n_unique_dev, unique_idx_out,
 *                     inverse_out)
 * (fingerprints, group count, first occurrences and inverse map, bit for
 * bit).  Each row is read from memory once: it is hashed, its fingerprint
 * is offered to the hash table, and the row is compared in full with the
 * smallest row holding the same fingerprint while both are still in L2.
 * Rows not 16-byte aligned (tokens or row_stride % 4 != 0) and batches of
 * at most 4096 rows take the two calls instead.
 *
 * tokens, n_rows, row_stride, lens, seed_state   as for hs_fingerprint;
 *                 0 <= n_rows <= 2^30 - 1 (0 writes *n_unique_dev = 0).
 *                 A length outside [0, row_stride] sets the device error
 *                 word, that row's fingerprint is 0 and it is compared with
 *                 its length clamped to [0, row_stride].
 * fp_out          device uint64 [n_rows], 8-byte aligned.
 * n_unique_dev, unique_idx_out, inverse_out   as for hs_unique_inverse.
 * workspace       device, >= hs_merge_rows_workspace(n_rows) bytes, 256-byte
 *                 aligned; contents on entry are ignored.
 */
size_t hs_merge_rows_workspace(int64_t n_rows);
hs_status hs_merge_rows(const int32_t* tokens, int64_t n_rows, int32_t row_stride,
                        const int32_t* lens, uint64_t seed_state, uint64_t* fp_out,
                        int32_t* n_unique_dev, int32_t* unique_idx_out, int32_t* inverse_out,
                        void* workspace, size_t workspace_bytes, hs_stream_t stream);

/*
 * hs_unique_inverse_noalloc — hs_unique_inverse for callers that cannot
 * allocate device memory.  The paper has no counterpart: this is a
 * convenience of this library.
 *
 * Some callers may not allocate at the point where they merge rows: code
 * running while a CUDA graph is being captured, plugins or embedded runtimes
 * that are given a fixed memory budget and no allocator, and latency-critical
 * request paths where an allocator call is an unbounded stall.  This entry
 * point takes no workspace: its scratch is a fixed array inside the
 * library's device memory (2,360,320 bytes, about 2.36 MB, present on every GPU
 * that loads the library until the process exits), so it calls no allocator at all.
 *
 * Same arguments, outputs and error behaviour as hs_unique_inverse, except:
 *   - n_rows must not exceed 65536 (larger n_rows returns
 *     HS_ERR_INVALID_ARG and enqueues nothing; use hs_unique_inverse);
 *   - every call on a device shares the one scratch array, so calls whose
 *     work overlaps on the GPU (different streams, or different host threads
 *     without ordering) race and give wrong results; calls on one stream are
 *     ordered and safe.  Each call clears whatever part of the scratch must
 *     start at zero, so leftovers of an earlier call do not matter;
 *   - the first call on each device looks up that device's copy of the
 *     scratch array (a host-side set-up step, done with the device current);
 *     make that first call before any stream capture begins.
 */
hs_status hs_unique_inverse_noalloc(const uint64_t* fp, const int32_t* tokens, int64_t n_rows,
                                    int32_t row_stride, const int32_t* lens,
                                    int32_t* n_unique_dev, int32_t* unique_idx_out,
                                    int32_t* inverse_out, hs_stream_t stream);

/*
 * hs_retrieve_topk — dense retrieval of the merged queries, fused top-k.
 *
 * Paper: Section 4.1, "Workloads": queries and documents are embedded and
 * the top-k (k = 12 in the paper) chunks are retrieved per query; the merged
 * queries of Section 3.3 share one retrieval.  Here:
 *   S[q, j] = sum_t queries[q, t] * corpus[j, t]   (bf16 inputs, fp32 sums)
 * and for each q the k pairs (S[q, j], j) that come first in the order
 * (score descending, ties to the lower j), written in that order.  The
 * Q x N score matrix is never stored.  For unit-norm rows S is the cosine.
 *
 * queries     device bf16 bits (uint16) [n_queries, dim] row-major.
 * corpus      device bf16 bits (uint16) [n_corpus, dim] row-major.
 * n_queries   >= 0 (0: nothing enqueued); n_corpus >= 1, < 2^31.
 * dim         >= 8, dim % 8 == 0.
 * k           1 <= k <= min(n_corpus, HS_TOPK_MAX_K).
 * scores_out  device float [n_queries, k]; ids_out device int32 [n_queries, k].
 * workspace   device, >= hs_retrieve_topk_workspace(...) bytes, 256-byte
 *             aligned; contents on entry are ignored.  The size returned for
 *             (n_queries, n_corpus, dim, k) suffices for every call with at
 *             most n_queries queries and the same n_corpus, dim and k.
 * Inputs must be finite; a NaN score is never selected.
 */
size_t hs_retrieve_topk_workspace(int64_t n_queries, int64_t n_corpus, int32_t dim, int32_t k);
hs_status hs_retrieve_topk(const uint16_t* queries, int64_t n_queries, const uint16_t* corpus,
                           int64_t n_corpus, int32_t dim, int32_t k, float* scores_out,
                           int32_t* ids_out, void* workspace, size_t workspace_bytes,
                           hs_stream_t stream);

/*
 * hs_retrieve_topk_n — hs_retrieve_topk with the query count in device
 * memory, so the merged queries of a batch can be retrieved without a host
 * synchronisation (Section 3.3: merged nodes execute once).
 *
 * Processes the first min(*n_queries_dev, max_queries) rows of `queries`
 * (rows up to max_queries must be addressable; the count is read on the
 * device when the kernels run) and writes that many rows of scores_out and
 * ids_out; later rows are left untouched.  Every other argument is as for
 * hs_retrieve_topk with n_queries = max_queries, including the workspace
 * size hs_retrieve_topk_workspace(max_queries, ...).
 */
hs_status hs_retrieve_topk_n(const uint16_t* queries, int64_t max_queries,
                             const int32_t* n_queries_dev, const uint16_t* corpus,
                             int64_t n_corpus, int32_t dim, int32_t k, float* scores_out,
                             int32_t* ids_out, void* workspace, size_t workspace_bytes,
                             hs_stream_t stream);

/*
 * hs_retrieve_topk_fanout — hs_retrieve_topk_n whose results go straight to
 * every row merged into each query: row o of scores_out / ids_out holds the
 * top-k of query inverse[o].
 *
 * Paper: Section 3.3 (I) and Appendix A.2: a merged node executes once and
 * its output flows to the downstream nodes of every node merged into it.
 * The result equals hs_retrieve_topk_n followed by hs_scatter_results of the
 * scores and of the ids with map = inverse, without the intermediate
 * per-query rows: the final merge of the retrieval writes the fanned-out
 * rows itself.
 *
 * n_queries_dev  device int32 scalar or NULL (NULL: max_queries queries).
 * inverse        device int32 [n_out]; an entry outside [0, query count)
 *                sets the device error word (HS_ERR_INVALID_ARG) and leaves
 *                that output row unwritten.
 * n_out          >= 0 (0: nothing enqueued); max_queries >= 1 if n_out > 0.
 * scores_out     device float [n_out, k]; ids_out device int32 [n_out, k].
 * Every other argument is as for hs_retrieve_topk_n (same workspace size).
 */
hs_status hs_retrieve_topk_fanout(const uint16_t* queries, int64_t max_queries,
                                  const int32_t* n_queries_dev, const int32_t* inverse,
                                  int64_t n_out, const uint16_t* corpus, int64_t n_corpus,
                                  int32_t dim, int32_t k, float* scores_out, int32_t* ids_out,
                                  void* workspace, size_t workspace_bytes, hs_stream_t stream);

/*
 * hs_merge_queries — the query side of a small batch in one launch:
 * fingerprint, exact merge and gather of the unique query vectors.
 *
 * Paper: Section 3.3, Eq. 2 (the signature of a node) and "Dynamic Fusion
 * and Reuse Mechanism" (I) (a node equal to one already in the window is
 * merged into it); Appendix A.2 (merge sets M(v*) executed once).
 * The outputs are exactly those of
 *   hs_fingerprint(queries as int32 words, n_queries, dim / 2, NULL,
 *                  seed_state, fp_out)
 *   hs_unique_inverse(fp, ..., n_unique_dev, unique_idx_out, inverse_out)
 *   hs_scatter_results(queries, unique_idx_out -> unique_queries_out)
 * with the gather limited to the first *n_unique_dev rows.  One kernel, no
 * workspace: meant for the latency-bound batches of an online stage.
 *
 * queries             device bf16 bits (uint16) [n_queries, dim] row-major,
 *                     16-byte aligned.
 * n_queries           0 <= n_queries <= HS_MERGE_QUERIES_MAX (0 writes
 *                     *n_unique_dev = 0 and nothing else).
 * dim                 8 <= dim <= 16384, dim % 8 == 0.
 * seed_state          FNV-1a seed, as for hs_fingerprint.
 * fp_in               device uint64 [n_queries] or NULL.  NULL: fingerprints
 *                     are computed here.  Otherwise these fingerprints are
 *                     used as given (they must be equal for equal rows, as
 *                     hs_unique_inverse requires; for instance fingerprints
 *                     carried from an earlier stage).
 * fp_out              device uint64 [n_queries] or NULL: the fingerprints used.
 * n_unique_dev, unique_idx_out, inverse_out   as for hs_unique_inverse.
 * unique_queries_out  device uint16 [n_queries, dim], 16-byte aligned, not
 *                     overlapping queries: row u < *n_unique_dev is
 *                     queries[unique_idx_out[u]]; later rows are untouched.
 */
hs_status hs_merge_queries(const uint16_t* queries, int64_t n_queries, int32_t dim,
                           uint64_t seed_state, const uint64_t* fp_in, uint64_t* fp_out,
                           int32_t* n_unique_dev, int32_t* unique_idx_out, int32_t* inverse_out,
                           uint16_t* unique_queries_out, hs_stream_t stream);

/*
 * hs_scatter_results — row gather/scatter: dst[i, :] = src[map[i], :].
 *
 * Paper: Section 3.3 (I): upon completion the output of the kept node flows
 * to the downstream nodes of all merged queries; Appendix A.2: nodes in
 * M(v*) depend on the output of v*.  With map = inverse from
 * hs_unique_inverse this fans results back to every originating row; with
 * map = unique_idx it gathers the unique rows.
 *
 * src        device [n_src, row_bytes] bytes; dst device [n_rows, row_bytes].
 * map        device int32 [n_rows]; an entry outside [0, n_src) sets the device
 *            error word (HS_ERR_INVALID_ARG) and leaves that dst row unwritten.
 * row_bytes  >= 1.  Any alignment is accepted; src/dst 16-byte aligned with
 *            row_bytes % 16 == 0 take the 16-byte vector path, 4-byte aligned
 *            with row_bytes % 4 == 0 the word path, otherwise bytes.
 * n_rows     >= 0 (0: nothing enqueued).  src and dst must not overlap.
 */
hs_status hs_scatter_results(const void* src, int64_t n_src, int64_t row_bytes,
                             const int32_t* map, int64_t n_rows, void* dst,
                             hs_stream_t stream);

/*
 * hs_rerank_topk — second retrieval stage: rescore each query's retrieved
 * candidates and keep the best k2.
 *
 * Paper: Section 4.1, "Workloads", RAG with rerank: a reranker scores the
 * initial top-12 chunks and the top-8 by those scores are kept.  The
 * reranker model is not part of this library; its score is the inner
 * product of bf16 rerank vectors accumulated in fp32:
 *   s[q, j] = sum_t rerank_queries[q, t] * rerank_corpus[candidates[q, j], t]
 * and query q keeps the k2 candidates first in (score descending, corpus
 * index ascending), written in that order.
 *
 * rerank_queries  device bf16 bits (uint16) [max_queries, dim], 16-byte
 *                 aligned rows.
 * n_queries_dev   device int32 scalar or NULL: queries processed =
 *                 min(*n_queries_dev, max_queries), or max_queries if NULL.
 * rerank_corpus   device bf16 bits [n_corpus, dim], 16-byte aligned.
 * dim             8 <= dim <= 65536, dim % 8 == 0.
 * candidates      device int32 [max_queries, k1] (e.g. the ids of
 *                 hs_retrieve_topk with k = k1).  A negative entry is an
 *                 absent candidate; an entry >= n_corpus sets the device
 *                 error word (HS_ERR_INVALID_ARG) and counts as absent.
 * k1, k2          1 <= k2 <= k1 <= 32.
 * inverse, n_out  NULL: one output row per query.  Otherwise n_out output
 *                 rows, row o holding the result of query inverse[o] (the
 *                 fan-out to every merged row, as hs_retrieve_topk_fanout);
 *                 an entry outside [0, query count) sets the device error
 *                 word and leaves that row unwritten.
 * scores_out      device float [rows, k2]; ids_out device int32 [rows, k2].
 *                 Entries past the number of present candidates are -inf / -1.
 */
hs_status hs_rerank_topk(const uint16_t* rerank_queries, int64_t max_queries,
                         const int32_t* n_queries_dev, const uint16_t* rerank_corpus,
                         int64_t n_corpus, int32_t dim, const int32_t* candidates, int32_t k1,
                         int32_t k2, const int32_t* inverse, int64_t n_out, float* scores_out,
                         int32_t* ids_out, hs_stream_t stream);

/*
 * Result cache — asynchronous cache reuse across batches.
 *
 * Paper: Section 3.3, "Dynamic Fusion and Reuse Mechanism" (II): a node
 * that matches a node completed earlier takes its result instead of being
 * executed.  Here the nodes are merged queries and the result is their
 * retrieval top-k.  The cache lives in device memory the caller provides
 * (hs_cache_bytes) and keeps `capacity` entries or more: sets of 8 entries,
 * chosen by the query's fingerprint; within a set a new entry takes an
 * empty way, else the least recently used one.  Every entry stores the
 * query vector, and a hit requires the whole vector to be equal: a
 * fingerprint collision never returns another query's result.
 *
 * A batch runs: hs_cache_lookup over its merged queries -> retrieval of the
 * misses (hs_retrieve_topk_n over miss_queries with count n_miss_dev) ->
 * hs_cache_insert of those results.  After the insert, row u of scores_out /
 * ids_out holds the top-k of query u, hit or miss.  Calls on one stream are
 * ordered, so each batch sees the inserts of the batches before it.  Streams
 * may share a cache: a query that equals one still being retrieved on
 * another stream misses and is retrieved again (no kernel waits for
 * another), and a lookup that overlaps an insert evicting the entry it reads
 * sees the slot's generation change and takes the miss path, so a hit never
 * returns a half-written or replaced entry.
 *
 * Arguments common to the cache calls:
 *   cache, cache_bytes   device memory, 256-byte aligned, at least
 *                        hs_cache_bytes(capacity, dim, k) bytes;
 *   capacity, dim, k     the values given to hs_cache_init (1 <= capacity
 *                        <= 2^30, 8 <= dim <= 65536 with dim % 8 == 0,
 *                        1 <= k <= HS_TOPK_MAX_K).  A cache whose header
 *                        does not match them sets the device error word
 *                        (HS_ERR_INVALID_ARG) and the call does nothing.
 */
size_t hs_cache_bytes(int64_t capacity, int32_t dim, int32_t k);  /* 0: invalid shape */
hs_status hs_cache_init(void* cache, size_t cache_bytes, int64_t capacity, int32_t dim,
                        int32_t k, hs_stream_t stream);

/*
 * hs_cache_lookup — look the merged queries of a batch up.
 *
 * queries        device bf16 bits [max_queries, dim], 16-byte aligned: the
 *                merged (unique) queries; the first count are looked up,
 *                count = min(*n_queries_dev, max_queries), or max_queries.
 * fp, fp_rows    query u's key is fp[fp_rows[u]] (fp_rows NULL: fp[u]);
 *                device uint64 / int32 (with hs_merge_queries: its fp_out
 *                and unique_idx_out).
 * scores_out     device float [max_queries, k], ids_out int32 [max_queries,
 *                k]: rows of hits are written here.
 * miss_list      device int32 [max_queries]: the ordinals u of the misses,
 *                in no particular order; *n_miss_dev their number (reset by
 *                this call); miss_queries device bf16 bits [max_queries,
 *                dim]: row i = queries[miss_list[i]].
 */
hs_status hs_cache_lookup(void* cache, size_t cache_bytes, int64_t capacity, int32_t dim,
                          int32_t k, const uint16_t* queries, const uint64_t* fp,
                          const int32_t* fp_rows, int64_t max_queries,
                          const int32_t* n_queries_dev, float* scores_out, int32_t* ids_out,
                          int32_t* miss_list, int32_t* n_miss_dev, uint16_t* miss_queries,
                          hs_stream_t stream);

/*
 * hs_cache_insert — store the retrieved results of a batch's misses.
 *
 * miss_list, n_miss_dev, miss_queries   as written by hs_cache_lookup.
 * max_queries    the max_queries of that lookup.
 * fp, fp_rows    as given to that lookup.
 * miss_scores, miss_ids   device float / int32 [max_queries, k]: row i is
 *                the top-k of miss_queries[i] (hs_retrieve_topk_n's output).
 * scores_out, ids_out     the lookup's outputs: row miss_list[i] receives
 *                row i of the results.  Entries are added to the cache; when
 *                every way of a set is being written by this batch the
 *                result is returned but not cached.
 */
hs_status hs_cache_insert(void* cache, size_t cache_bytes, int64_t capacity, int32_t dim,
                          int32_t k, const int32_t* miss_list, const int32_t* n_miss_dev,
                          int64_t max_queries, const uint16_t* miss_queries, const uint64_t* fp,
                          const int32_t* fp_rows, const float* miss_scores,
                          const int32_t* miss_ids, float* scores_out, int32_t* ids_out,
                          hs_stream_t stream);

/*
 * hs_cache_stats — hits and misses counted since hs_cache_init.
 * Synchronises `stream`; host pointers for the two counts.
 */
hs_status hs_cache_stats(const void* cache, uint64_t* hits, uint64_t* misses, hs_stream_t stream);

/*
 * hs_segment_sum — priority contribution of each fused node: the sum of the
 * contributions of the rows merged into it.
 *
 * Paper: Section 3.3, "Reuse-Driven Priority Adjustment", Eq. 3:
 * phi(v*) = sum over v in M(v*) of phi(v), so that a node shared by many
 * queries is scheduled with their combined weight.  With the inverse map of
 * hs_unique_inverse (or hs_merge_queries):
 *   out[u] = sum of phi[i] over the rows i with inverse[i] == u,
 * for u < count, count = min(*n_groups_dev, max_groups), or max_groups if
 * n_groups_dev is NULL; out[u] = 0 for count <= u < max_groups.
 *
 * Additions are fp64 in an unspecified order: for a group of m rows the
 * result is within (m-1)u/(1-(m-1)u) * sum|phi| of the exact sum
 * (u = 2^-53); sums whose partial sums are all representable (integers
 * below 2^53, for instance) are exact.
 *
 * phi           device double [n_rows], 8-byte aligned.
 * inverse       device int32 [n_rows]; an entry outside [0, count) sets the
 *               device error word (HS_ERR_INVALID_ARG) and that row is left
 *               out of every sum.
 * n_rows        >= 0.
 * n_groups_dev  device int32 scalar or NULL.
 * max_groups    0 <= max_groups < 2^31 (>= 1 when n_rows > 0).
 * out           device double [max_groups], 8-byte aligned; every entry is
 *               written.
 */
hs_status hs_segment_sum(const double* phi, const int32_t* inverse, int64_t n_rows,
                         const int32_t* n_groups_dev, int64_t max_groups, double* out,
                         hs_stream_t stream);

/*
 * hs_get_device_error — synchronise `stream`, then read and clear the
 * current device's error word.  Returns HS_OK if no kernel reported a
 * problem since the last call, else the recorded status (HS_ERR_TIMEOUT
 * takes precedence over HS_ERR_INVALID_ARG).
 */
hs_status hs_get_device_error(hs_stream_t stream);

/*
 * hs_memcpy_async — copy `bytes` bytes from src to dst on `stream`: host
 * to device, device to host or device to device, the direction taken from
 * the pointers (unified addressing).  This is how a caller moves a batch's
 * inputs from host buffers into the device buffers the other calls take,
 * and its results back; with pinned host memory the copy is asynchronous
 * and overlaps kernels on other streams.  The caller owns both buffers and
 * keeps them alive until the copy has run.  bytes == 0 does nothing.
 * Returns HS_ERR_INVALID_ARG for a NULL pointer with bytes > 0, and
 * HS_ERR_CUDA if the runtime rejects the copy.
 */
hs_status hs_memcpy_async(void* dst, const void* src, size_t bytes, hs_stream_t stream);

/*
 * hs_launch_count — diagnostics: number of kernels this library has launched
 * in this process (all devices, all threads) since it was loaded.  Takes no
 * part in the method; callers use it to count device work per call.
 */
uint64_t hs_launch_count(void);

/*
 * hs_debug_scan_wait — test hook of the bounded device waits (failure
 * detection); takes no part in the method.
 *
 * Every device-side wait of the library gives up after a limit (2 s by
 * default) and then sets HS_ERR_TIMEOUT in the device error word instead of
 * spinning on.  hs_unique_inverse's scan waits for the status each earlier
 * tile of 16,384 rows publishes (decoupled look-back).  This hook, for tests
 * only, lowers that wait's limit and can stop one tile from publishing, so
 * that a test can make the wait run out and check that the call returns,
 * that hs_get_device_error reports HS_ERR_TIMEOUT, and that the next call
 * is correct again.  While a tile is withheld, the outputs of
 * hs_unique_inverse calls with more than withhold_tile + 1 tiles are
 * unspecified (every write stays inside the outputs and the workspace).
 *
 * limit_ns       wait limit in ns, 1 <= limit_ns <= 2e9; 0 restores 2 s.
 * withhold_tile  index of the scan tile that does not publish; -1: none.
 * Settings are process-wide and take effect at the next launch.
 * Returns HS_ERR_INVALID_ARG for a limit above 2 s or withhold_tile < -1.
 */
hs_status hs_debug_scan_wait(uint64_t limit_ns, int64_t withhold_tile);

/*
 * hs_debug_merge_key_mask — test hook of hs_merge_rows; takes no part in
 * the method.  hs_merge_rows keys its hash table by fingerprint & mask
 * (the fingerprints it writes are not masked), so a narrow mask forces
 * fingerprint collisions and exercises the full-row comparison that keeps
 * the merge exact.  mask 0 restores all ones.  Process-wide; takes effect
 * at the next launch; affects only batches of more than 4096 aligned rows.
 */
hs_status hs_debug_merge_key_mask(uint64_t mask);

/*
 * hs_debug_retrieve_wait — test hook of the retrieval's bounded waits
 * (failure detection); takes no part in the method.  Both retrieval kernels
 * (the main one and, for at most 16 addressable queries, the small-batch
 * one) give up a pipeline wait (shared-memory stage, query load,
 * tensor-memory accumulator) after limit_ns, set HS_ERR_TIMEOUT in the
 * device error word and return: before tensor memory is freed, the CTA
 * whose barriers count the copies (the even CTA of a pair) waits, with the
 * same limit, for every copy it armed and every MMA it issued.  With
 * withhold_first = 1 every CTA skips the copies of its first corpus stage,
 * so that stage never fills and the waits run out; the outputs of such a
 * call are unspecified (every write stays inside the outputs and the
 * workspace).
 *
 * limit_ns        wait limit in ns, at most 2e9; 0 restores 2 s.
 * withhold_first  0 or 1.
 * Settings are process-wide and take effect at the next launch.
 * Returns HS_ERR_INVALID_ARG for a limit above 2 s or withhold_first
 * outside {0, 1}.
 */
hs_status hs_debug_retrieve_wait(uint64_t limit_ns, int32_t withhold_first);

/*
 * hs_debug_stream_rows — diagnostics: stream the rows' valid prefixes with
 * no hashing, to measure what the row layout itself costs to read; takes no
 * part in the method.
 *
 * Reads tokens[i, 0:len_i] of every row (the bytes hs_fingerprint hashes)
 * with access pattern `pattern`, folds them into *checksum_dev (xor; the
 * caller zeroes it first), and enqueues one kernel on num_SMs *
 * blocks_per_sm blocks of 256 threads:
 *   0  a warp per row, 16 bytes per lane (coalesced 512-byte reads);
 *   1  a lane per row, 32-byte loads (hs_fingerprint's chunk pattern);
 *   2  a warp per row over the whole padded row (row_stride tokens).
 * tokens        device int32 [n_rows, row_stride], 32-byte aligned,
 *               row_stride % 8 == 0.
 * lens          device int32 [n_rows] or NULL; lengths are clamped to
 *               [0, row_stride] (no error is recorded).
 * checksum_dev  device uint32 scalar.
 * blocks_per_sm 1 ... 8.
 */
hs_status hs_debug_stream_rows(const int32_t* tokens, int64_t n_rows, int32_t row_stride,
                               const int32_t* lens, int32_t pattern, uint32_t* checksum_dev,
                               int32_t blocks_per_sm, hs_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* HS_H_ */
