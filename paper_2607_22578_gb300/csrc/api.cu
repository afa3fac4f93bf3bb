// C-ABI entry points (include/hs.h): argument validation, workspace checks,
// the per-device error word, and dispatch to the kernels.
#include <stdarg.h>
#include <stdio.h>

#include <atomic>
#include <mutex>

#include "hs_internal.cuh"

namespace hs {

hs_status launch_fingerprint(const int32_t*, int64_t, int32_t, const int32_t*, uint64_t,
                             uint64_t*, cudaStream_t);
size_t unique_inverse_workspace(int64_t);
hs_status launch_unique_inverse(const uint64_t*, const int32_t*, int64_t, int32_t,
                                const int32_t*, int32_t*, int32_t*, int32_t*, void*,
                                cudaStream_t);
size_t merge_rows_workspace(int64_t);
hs_status launch_merge_rows(const int32_t*, int64_t, int32_t, const int32_t*, uint64_t, uint64_t*,
                            int32_t*, int32_t*, int32_t*, void*, cudaStream_t);
size_t retrieve_topk_workspace(int64_t, int64_t, int32_t, int32_t);
hs_status launch_retrieve_topk(const uint16_t*, int64_t, const int32_t*, const int32_t*, int64_t,
                               const uint16_t*, int64_t, int32_t, int32_t, float*, int32_t*,
                               void*, size_t, cudaStream_t);
hs_status launch_segment_sum(const double*, const int32_t*, int64_t, const int32_t*, int64_t,
                             double*, cudaStream_t);
hs_status launch_rerank(const uint16_t*, int64_t, const int32_t*, const uint16_t*, int64_t, int32_t,
                        const int32_t*, int32_t, int32_t, const int32_t*, int64_t, float*,
                        int32_t*, cudaStream_t);
size_t cache_bytes(int64_t, int32_t, int32_t);
hs_status launch_cache_init(void*, int64_t, int32_t, int32_t, cudaStream_t);
hs_status launch_cache_lookup(void*, int64_t, int32_t, int32_t, const uint16_t*, const uint64_t*,
                              const int32_t*, int64_t, const int32_t*, float*, int32_t*, int32_t*,
                              int32_t*, uint16_t*, cudaStream_t);
hs_status launch_cache_insert(void*, int64_t, int32_t, int32_t, const int32_t*, const int32_t*,
                              int64_t, const uint16_t*, const uint64_t*, const int32_t*,
                              const float*, const int32_t*, float*, int32_t*, cudaStream_t);
hs_status cache_stats(const void*, unsigned long long*, unsigned long long*, cudaStream_t);
hs_status launch_merge_queries(const uint16_t*, int64_t, int32_t, uint64_t, const uint64_t*,
                               uint64_t*, int32_t*, int32_t*, int32_t*, uint16_t*, cudaStream_t);
hs_status launch_scatter(const void*, int64_t, int64_t, const int32_t*, int64_t, void*,
                         cudaStream_t);

namespace {
thread_local char g_msg[512] = "";
constexpr int kMaxDevices = 64;
__device__ unsigned g_device_error;  // one word per device (module-scope variable)
unsigned* g_err_addr[kMaxDevices] = {};
int g_sms[kMaxDevices] = {};
std::mutex g_mu;
std::atomic<uint64_t> g_launches{0};

int current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return -1;
  return dev;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

void clear_msg() { g_msg[0] = '\0'; }
}  // namespace

hs_status fail(hs_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_msg, sizeof g_msg, fmt, ap);
  va_end(ap);
  return s;
}

hs_status cuda_fail(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return HS_OK;
  return fail(HS_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

unsigned* device_error_word() {
  const int dev = current_device();
  if (dev < 0) return nullptr;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_err_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_device_error) != cudaSuccess) return nullptr;
    g_err_addr[dev] = static_cast<unsigned*>(p);
  }
  return g_err_addr[dev];
}

void clear_last_error() { clear_msg(); }

void count_launches(unsigned n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

int num_sms() {
  const int dev = current_device();
  if (dev < 0) return 1;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_sms[dev]) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v < 1)
      v = 1;
    g_sms[dev] = v;
  }
  return g_sms[dev];
}

}  // namespace hs

using namespace hs;

extern "C" {

const char* hs_last_error(void) { return g_msg; }

const char* hs_version(void) { return "hs 0.2 (sm_103a)"; }

uint64_t hs_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

hs_status hs_fingerprint(const int32_t* tokens, int64_t n_rows, int32_t row_stride,
                         const int32_t* lens, uint64_t seed_state, uint64_t* fp_out,
                         hs_stream_t stream) {
  clear_msg();
  if (n_rows < 0) return fail(HS_ERR_INVALID_ARG, "n_rows < 0");
  if (row_stride < 0) return fail(HS_ERR_INVALID_ARG, "row_stride < 0");
  if (n_rows == 0) return HS_OK;
  if (!tokens && row_stride > 0) return fail(HS_ERR_INVALID_ARG, "tokens is NULL");
  if (!fp_out) return fail(HS_ERR_INVALID_ARG, "fp_out is NULL");
  if (!aligned(tokens, 4) || !aligned(fp_out, 8) || (lens && !aligned(lens, 4)))
    return fail(HS_ERR_INVALID_ARG, "misaligned pointer (tokens/lens 4 B, fp_out 8 B)");
  return launch_fingerprint(tokens, n_rows, row_stride, lens, seed_state, fp_out,
                            reinterpret_cast<cudaStream_t>(stream));
}

size_t hs_unique_inverse_workspace(int64_t n_rows) { return unique_inverse_workspace(n_rows); }

hs_status hs_unique_inverse(const uint64_t* fp, const int32_t* tokens, int64_t n_rows,
                            int32_t row_stride, const int32_t* lens, int32_t* n_unique_dev,
                            int32_t* unique_idx_out, int32_t* inverse_out, void* workspace,
                            size_t workspace_bytes, hs_stream_t stream) {
  clear_msg();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (n_rows < 0 || n_rows > (int64_t)((1u << 30) - 1))
    return fail(HS_ERR_INVALID_ARG, "n_rows outside [0, 2^30 - 1]");
  if (row_stride < 0) return fail(HS_ERR_INVALID_ARG, "row_stride < 0");
  if (!n_unique_dev) return fail(HS_ERR_INVALID_ARG, "n_unique_dev is NULL");
  if (!aligned(n_unique_dev, 4)) return fail(HS_ERR_INVALID_ARG, "n_unique_dev misaligned");
  if (n_rows == 0) return cuda_fail(cudaMemsetAsync(n_unique_dev, 0, sizeof(int32_t), s),
                                    "n_unique clear");
  if (!fp || !unique_idx_out || !inverse_out || (!tokens && row_stride > 0))
    return fail(HS_ERR_INVALID_ARG, "NULL input or output pointer");
  if (!aligned(fp, 8) || !aligned(tokens, 4) || (lens && !aligned(lens, 4)) ||
      !aligned(unique_idx_out, 4) || !aligned(inverse_out, 4))
    return fail(HS_ERR_INVALID_ARG, "misaligned pointer");
  const size_t need = unique_inverse_workspace(n_rows);
  if (!workspace || !aligned(workspace, 256))
    return fail(HS_ERR_WORKSPACE, "workspace NULL or not 256-byte aligned");
  if (workspace_bytes < need)
    return fail(HS_ERR_WORKSPACE, "unique workspace too small: %zu < %zu", workspace_bytes, need);
  return launch_unique_inverse(fp, tokens, n_rows, row_stride, lens, n_unique_dev,
                               unique_idx_out, inverse_out, workspace, s);
}

size_t hs_merge_rows_workspace(int64_t n_rows) { return merge_rows_workspace(n_rows); }

hs_status hs_merge_rows(const int32_t* tokens, int64_t n_rows, int32_t row_stride,
                        const int32_t* lens, uint64_t seed_state, uint64_t* fp_out,
                        int32_t* n_unique_dev, int32_t* unique_idx_out, int32_t* inverse_out,
                        void* workspace, size_t workspace_bytes, hs_stream_t stream) {
  clear_msg();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (n_rows < 0 || n_rows > (int64_t)((1u << 30) - 1))
    return fail(HS_ERR_INVALID_ARG, "n_rows outside [0, 2^30 - 1]");
  if (row_stride < 0) return fail(HS_ERR_INVALID_ARG, "row_stride < 0");
  if (!n_unique_dev) return fail(HS_ERR_INVALID_ARG, "n_unique_dev is NULL");
  if (!aligned(n_unique_dev, 4)) return fail(HS_ERR_INVALID_ARG, "n_unique_dev misaligned");
  if (n_rows == 0) return cuda_fail(cudaMemsetAsync(n_unique_dev, 0, sizeof(int32_t), s),
                                    "n_unique clear");
  if (!fp_out || !unique_idx_out || !inverse_out || (!tokens && row_stride > 0))
    return fail(HS_ERR_INVALID_ARG, "NULL input or output pointer");
  if (!aligned(fp_out, 8) || !aligned(tokens, 4) || (lens && !aligned(lens, 4)) ||
      !aligned(unique_idx_out, 4) || !aligned(inverse_out, 4))
    return fail(HS_ERR_INVALID_ARG, "misaligned pointer");
  const size_t need = merge_rows_workspace(n_rows);
  if (!workspace || !aligned(workspace, 256))
    return fail(HS_ERR_WORKSPACE, "workspace NULL or not 256-byte aligned");
  if (workspace_bytes < need)
    return fail(HS_ERR_WORKSPACE, "merge workspace too small: %zu < %zu", workspace_bytes, need);
  return launch_merge_rows(tokens, n_rows, row_stride, lens, seed_state, fp_out, n_unique_dev,
                           unique_idx_out, inverse_out, workspace, s);
}

size_t hs_retrieve_topk_workspace(int64_t n_queries, int64_t n_corpus, int32_t dim, int32_t k) {
  return retrieve_topk_workspace(n_queries, n_corpus, dim, k);
}

static hs_status retrieve_common(const uint16_t* queries, int64_t n_queries,
                                 const int32_t* n_queries_dev, const int32_t* inverse,
                                 int64_t n_out, const uint16_t* corpus, int64_t n_corpus,
                                 int32_t dim, int32_t k, float* scores_out, int32_t* ids_out,
                                 void* workspace, size_t workspace_bytes, hs_stream_t stream) {
  if (n_queries < 0) return fail(HS_ERR_INVALID_ARG, "n_queries < 0");
  if (n_corpus < 1 || n_corpus > 0x7fffffffLL)
    return fail(HS_ERR_INVALID_ARG, "n_corpus outside [1, 2^31 - 1]");
  if (dim < 8 || dim % 8 != 0) return fail(HS_ERR_INVALID_ARG, "dim must be >= 8 and a multiple of 8");
  if (k < 1 || (int64_t)k > n_corpus || k > HS_TOPK_MAX_K)
    return fail(HS_ERR_INVALID_ARG, "k outside [1, min(n_corpus, %d)]", HS_TOPK_MAX_K);
  if (inverse) {
    if (n_out < 0 || n_out > 0x7fffffffLL)
      return fail(HS_ERR_INVALID_ARG, "n_out outside [0, 2^31 - 1]");
    if (n_out == 0) return HS_OK;
    if (n_queries == 0) return fail(HS_ERR_INVALID_ARG, "n_out > 0 rows but no queries");
    if (!aligned(inverse, 4)) return fail(HS_ERR_INVALID_ARG, "inverse misaligned");
  }
  if (n_queries == 0) return HS_OK;
  if (n_queries > 0x7fffffffLL) return fail(HS_ERR_INVALID_ARG, "n_queries >= 2^31");
  if (!queries || !corpus || !scores_out || !ids_out)
    return fail(HS_ERR_INVALID_ARG, "NULL input or output pointer");
  if (!aligned(queries, 16) || !aligned(corpus, 16))
    return fail(HS_ERR_INVALID_ARG, "queries/corpus must be 16-byte aligned");
  if (!aligned(scores_out, 4) || !aligned(ids_out, 4))
    return fail(HS_ERR_INVALID_ARG, "scores_out/ids_out misaligned");
  if (!workspace || !aligned(workspace, 256))
    return fail(HS_ERR_WORKSPACE, "workspace NULL or not 256-byte aligned");
  if (n_queries_dev && !aligned(n_queries_dev, 4))
    return fail(HS_ERR_INVALID_ARG, "n_queries_dev misaligned");
  return launch_retrieve_topk(queries, n_queries, n_queries_dev, inverse, n_out, corpus,
                              n_corpus, dim, k, scores_out, ids_out, workspace, workspace_bytes,
                              reinterpret_cast<cudaStream_t>(stream));
}

hs_status hs_retrieve_topk(const uint16_t* queries, int64_t n_queries, const uint16_t* corpus,
                           int64_t n_corpus, int32_t dim, int32_t k, float* scores_out,
                           int32_t* ids_out, void* workspace, size_t workspace_bytes,
                           hs_stream_t stream) {
  clear_msg();
  return retrieve_common(queries, n_queries, nullptr, nullptr, 0, corpus, n_corpus, dim, k,
                         scores_out, ids_out, workspace, workspace_bytes, stream);
}

hs_status hs_retrieve_topk_n(const uint16_t* queries, int64_t max_queries,
                             const int32_t* n_queries_dev, const uint16_t* corpus,
                             int64_t n_corpus, int32_t dim, int32_t k, float* scores_out,
                             int32_t* ids_out, void* workspace, size_t workspace_bytes,
                             hs_stream_t stream) {
  clear_msg();
  if (!n_queries_dev) return fail(HS_ERR_INVALID_ARG, "n_queries_dev is NULL");
  return retrieve_common(queries, max_queries, n_queries_dev, nullptr, 0, corpus, n_corpus, dim,
                         k, scores_out, ids_out, workspace, workspace_bytes, stream);
}

hs_status hs_retrieve_topk_fanout(const uint16_t* queries, int64_t max_queries,
                                  const int32_t* n_queries_dev, const int32_t* inverse,
                                  int64_t n_out, const uint16_t* corpus, int64_t n_corpus,
                                  int32_t dim, int32_t k, float* scores_out, int32_t* ids_out,
                                  void* workspace, size_t workspace_bytes, hs_stream_t stream) {
  clear_msg();
  if (n_out < 0 || n_out > 0x7fffffffLL)
    return fail(HS_ERR_INVALID_ARG, "n_out outside [0, 2^31 - 1]");
  if (n_out == 0) return HS_OK;
  if (!inverse) return fail(HS_ERR_INVALID_ARG, "inverse is NULL");
  return retrieve_common(queries, max_queries, n_queries_dev, inverse, n_out, corpus, n_corpus,
                         dim, k, scores_out, ids_out, workspace, workspace_bytes, stream);
}

hs_status hs_merge_queries(const uint16_t* queries, int64_t n_queries, int32_t dim,
                           uint64_t seed_state, const uint64_t* fp_in, uint64_t* fp_out,
                           int32_t* n_unique_dev, int32_t* unique_idx_out, int32_t* inverse_out,
                           uint16_t* unique_queries_out, hs_stream_t stream) {
  clear_msg();
  if (n_queries < 0 || n_queries > HS_MERGE_QUERIES_MAX)
    return fail(HS_ERR_INVALID_ARG, "n_queries outside [0, %d]", HS_MERGE_QUERIES_MAX);
  if (dim < 8 || dim % 8 != 0 || dim > 16384)
    return fail(HS_ERR_INVALID_ARG, "dim must be a multiple of 8 in [8, 16384]");
  if (!n_unique_dev || !aligned(n_unique_dev, 4))
    return fail(HS_ERR_INVALID_ARG, "n_unique_dev NULL or misaligned");
  if (n_queries > 0) {
    if (!queries || !unique_idx_out || !inverse_out || !unique_queries_out)
      return fail(HS_ERR_INVALID_ARG, "NULL input or output pointer");
    if (!aligned(queries, 16) || !aligned(unique_queries_out, 16))
      return fail(HS_ERR_INVALID_ARG, "queries/unique_queries_out must be 16-byte aligned");
    if (!aligned(unique_idx_out, 4) || !aligned(inverse_out, 4) || (fp_in && !aligned(fp_in, 8)) ||
        (fp_out && !aligned(fp_out, 8)))
      return fail(HS_ERR_INVALID_ARG, "misaligned pointer");
    const uintptr_t q0 = reinterpret_cast<uintptr_t>(queries);
    const uintptr_t u0 = reinterpret_cast<uintptr_t>(unique_queries_out);
    const uintptr_t bytes = (uintptr_t)n_queries * (uintptr_t)dim * 2u;
    if (q0 < u0 + bytes && u0 < q0 + bytes)
      return fail(HS_ERR_INVALID_ARG, "queries and unique_queries_out overlap");
  }
  return launch_merge_queries(queries, n_queries, dim, seed_state, fp_in, fp_out, n_unique_dev,
                              unique_idx_out, inverse_out, unique_queries_out,
                              reinterpret_cast<cudaStream_t>(stream));
}

hs_status hs_scatter_results(const void* src, int64_t n_src, int64_t row_bytes,
                             const int32_t* map, int64_t n_rows, void* dst, hs_stream_t stream) {
  clear_msg();
  if (n_rows < 0 || n_src < 0) return fail(HS_ERR_INVALID_ARG, "negative row count");
  if (row_bytes < 1 || row_bytes > 0x7fffffffLL)
    return fail(HS_ERR_INVALID_ARG, "row_bytes outside [1, 2^31 - 1]");
  if (n_rows == 0) return HS_OK;
  if (!src || !map || !dst) return fail(HS_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned(map, 4)) return fail(HS_ERR_INVALID_ARG, "map misaligned");
  const uintptr_t s0 = reinterpret_cast<uintptr_t>(src), d0 = reinterpret_cast<uintptr_t>(dst);
  const uintptr_t s1 = s0 + (uintptr_t)(n_src * row_bytes), d1 = d0 + (uintptr_t)(n_rows * row_bytes);
  if (s0 < d1 && d0 < s1) return fail(HS_ERR_INVALID_ARG, "src and dst overlap");
  return launch_scatter(src, n_src, row_bytes, map, n_rows, dst,
                        reinterpret_cast<cudaStream_t>(stream));
}

hs_status hs_rerank_topk(const uint16_t* rerank_queries, int64_t max_queries,
                         const int32_t* n_queries_dev, const uint16_t* rerank_corpus,
                         int64_t n_corpus, int32_t dim, const int32_t* candidates, int32_t k1,
                         int32_t k2, const int32_t* inverse, int64_t n_out, float* scores_out,
                         int32_t* ids_out, hs_stream_t stream) {
  clear_msg();
  if (max_queries < 0 || max_queries > 0x7fffffffLL)
    return fail(HS_ERR_INVALID_ARG, "max_queries outside [0, 2^31 - 1]");
  if (n_corpus < 1 || n_corpus > 0x7fffffffLL)
    return fail(HS_ERR_INVALID_ARG, "n_corpus outside [1, 2^31 - 1]");
  if (dim < 8 || dim % 8 != 0 || dim > 65536)
    return fail(HS_ERR_INVALID_ARG, "dim must be a multiple of 8 in [8, 65536]");
  if (k1 < 1 || k1 > 32 || k2 < 1 || k2 > k1)
    return fail(HS_ERR_INVALID_ARG, "need 1 <= k2 <= k1 <= 32");
  if (inverse && (n_out < 0 || n_out > 0x7fffffffLL))
    return fail(HS_ERR_INVALID_ARG, "n_out outside [0, 2^31 - 1]");
  const int64_t rows = inverse ? n_out : max_queries;
  if (rows == 0) return HS_OK;
  if (max_queries == 0) return fail(HS_ERR_INVALID_ARG, "output rows but no queries");
  if (!rerank_queries || !rerank_corpus || !candidates || !scores_out || !ids_out)
    return fail(HS_ERR_INVALID_ARG, "NULL input or output pointer");
  if (!aligned(rerank_queries, 16) || !aligned(rerank_corpus, 16))
    return fail(HS_ERR_INVALID_ARG, "rerank vectors must be 16-byte aligned");
  if (!aligned(candidates, 4) || !aligned(scores_out, 4) || !aligned(ids_out, 4) ||
      (inverse && !aligned(inverse, 4)) || (n_queries_dev && !aligned(n_queries_dev, 4)))
    return fail(HS_ERR_INVALID_ARG, "misaligned pointer");
  return launch_rerank(rerank_queries, max_queries, n_queries_dev, rerank_corpus, n_corpus, dim,
                       candidates, k1, k2, inverse, n_out, scores_out, ids_out,
                       reinterpret_cast<cudaStream_t>(stream));
}

size_t hs_cache_bytes(int64_t capacity, int32_t dim, int32_t k) {
  if (capacity < 1 || capacity > (1LL << 30) || dim < 8 || dim % 8 != 0 || dim > 65536 || k < 1 ||
      k > HS_TOPK_MAX_K)
    return 0;
  return cache_bytes(capacity, dim, k);
}

static hs_status cache_check(const void* cache, size_t bytes, int64_t capacity, int32_t dim,
                             int32_t k) {
  const size_t need = hs_cache_bytes(capacity, dim, k);
  if (need == 0)
    return fail(HS_ERR_INVALID_ARG, "cache shape: capacity in [1, 2^30], dim %% 8 == 0 in "
                                    "[8, 65536], k in [1, %d]", HS_TOPK_MAX_K);
  if (!cache || !aligned(cache, 256))
    return fail(HS_ERR_WORKSPACE, "cache NULL or not 256-byte aligned");
  if (bytes < need) return fail(HS_ERR_WORKSPACE, "cache too small: %zu < %zu", bytes, need);
  return HS_OK;
}

hs_status hs_cache_init(void* cache, size_t cache_bytes_, int64_t capacity, int32_t dim, int32_t k,
                        hs_stream_t stream) {
  clear_msg();
  const hs_status st = cache_check(cache, cache_bytes_, capacity, dim, k);
  if (st != HS_OK) return st;
  return launch_cache_init(cache, capacity, dim, k, reinterpret_cast<cudaStream_t>(stream));
}

hs_status hs_cache_lookup(void* cache, size_t cache_bytes_, int64_t capacity, int32_t dim,
                          int32_t k, const uint16_t* queries, const uint64_t* fp,
                          const int32_t* fp_rows, int64_t max_queries,
                          const int32_t* n_queries_dev, float* scores_out, int32_t* ids_out,
                          int32_t* miss_list, int32_t* n_miss_dev, uint16_t* miss_queries,
                          hs_stream_t stream) {
  clear_msg();
  const hs_status st = cache_check(cache, cache_bytes_, capacity, dim, k);
  if (st != HS_OK) return st;
  if (max_queries < 0 || max_queries > 0x7fffffffLL)
    return fail(HS_ERR_INVALID_ARG, "max_queries outside [0, 2^31 - 1]");
  if (!n_miss_dev || !aligned(n_miss_dev, 4))
    return fail(HS_ERR_INVALID_ARG, "n_miss_dev NULL or misaligned");
  if (max_queries > 0) {
    if (!queries || !fp || !scores_out || !ids_out || !miss_list || !miss_queries)
      return fail(HS_ERR_INVALID_ARG, "NULL input or output pointer");
    if (!aligned(queries, 16) || !aligned(miss_queries, 16) || !aligned(fp, 8) ||
        !aligned(scores_out, 4) || !aligned(ids_out, 4) || !aligned(miss_list, 4) ||
        (fp_rows && !aligned(fp_rows, 4)) || (n_queries_dev && !aligned(n_queries_dev, 4)))
      return fail(HS_ERR_INVALID_ARG, "misaligned pointer");
  }
  return launch_cache_lookup(cache, capacity, dim, k, queries, fp, fp_rows, max_queries,
                             n_queries_dev, scores_out, ids_out, miss_list, n_miss_dev,
                             miss_queries, reinterpret_cast<cudaStream_t>(stream));
}

hs_status hs_cache_insert(void* cache, size_t cache_bytes_, int64_t capacity, int32_t dim,
                          int32_t k, const int32_t* miss_list, const int32_t* n_miss_dev,
                          int64_t max_queries, const uint16_t* miss_queries, const uint64_t* fp,
                          const int32_t* fp_rows, const float* miss_scores,
                          const int32_t* miss_ids, float* scores_out, int32_t* ids_out,
                          hs_stream_t stream) {
  clear_msg();
  const hs_status st = cache_check(cache, cache_bytes_, capacity, dim, k);
  if (st != HS_OK) return st;
  if (max_queries < 0 || max_queries > 0x7fffffffLL)
    return fail(HS_ERR_INVALID_ARG, "max_queries outside [0, 2^31 - 1]");
  if (max_queries == 0) return HS_OK;
  if (!miss_list || !n_miss_dev || !miss_queries || !fp || !miss_scores || !miss_ids ||
      !scores_out || !ids_out)
    return fail(HS_ERR_INVALID_ARG, "NULL input or output pointer");
  if (!aligned(miss_queries, 16) || !aligned(fp, 8) || !aligned(miss_list, 4) ||
      !aligned(n_miss_dev, 4) || !aligned(miss_scores, 4) || !aligned(miss_ids, 4) ||
      !aligned(scores_out, 4) || !aligned(ids_out, 4) || (fp_rows && !aligned(fp_rows, 4)))
    return fail(HS_ERR_INVALID_ARG, "misaligned pointer");
  return launch_cache_insert(cache, capacity, dim, k, miss_list, n_miss_dev, max_queries,
                             miss_queries, fp, fp_rows, miss_scores, miss_ids, scores_out,
                             ids_out, reinterpret_cast<cudaStream_t>(stream));
}

hs_status hs_cache_stats(const void* cache, uint64_t* hits, uint64_t* misses,
                         hs_stream_t stream) {
  clear_msg();
  if (!cache || !hits || !misses) return fail(HS_ERR_INVALID_ARG, "NULL pointer");
  unsigned long long h = 0, m = 0;
  const hs_status st = cache_stats(cache, &h, &m, reinterpret_cast<cudaStream_t>(stream));
  if (st != HS_OK) return st;
  *hits = h;
  *misses = m;
  return HS_OK;
}

hs_status hs_segment_sum(const double* phi, const int32_t* inverse, int64_t n_rows,
                         const int32_t* n_groups_dev, int64_t max_groups, double* out,
                         hs_stream_t stream) {
  clear_msg();
  if (n_rows < 0) return fail(HS_ERR_INVALID_ARG, "n_rows < 0");
  if (max_groups < 0 || max_groups > 0x7fffffffLL)
    return fail(HS_ERR_INVALID_ARG, "max_groups outside [0, 2^31 - 1]");
  if (max_groups > 0 && !out) return fail(HS_ERR_INVALID_ARG, "out is NULL");
  if (n_rows > 0 && (!phi || !inverse)) return fail(HS_ERR_INVALID_ARG, "NULL input pointer");
  if (!aligned(phi, 8) || !aligned(out, 8) || !aligned(inverse, 4) ||
      (n_groups_dev && !aligned(n_groups_dev, 4)))
    return fail(HS_ERR_INVALID_ARG, "misaligned pointer (phi/out 8 B, inverse/count 4 B)");
  if (n_rows > 0 && max_groups == 0)
    return fail(HS_ERR_INVALID_ARG, "rows given but max_groups is 0");
  return launch_segment_sum(phi, inverse, n_rows, n_groups_dev, max_groups, out,
                            reinterpret_cast<cudaStream_t>(stream));
}

hs_status hs_get_device_error(hs_stream_t stream) {
  clear_msg();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
  unsigned* addr = device_error_word();
  if (!addr) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  unsigned v = 0;
  e = cudaMemcpy(&v, addr, sizeof v, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "error word read");
  if (v) {
    const unsigned zero = 0;
    e = cudaMemcpy(addr, &zero, sizeof zero, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "error word clear");
  }
  if (v & kErrTimeout) return fail(HS_ERR_TIMEOUT, "a bounded device wait ran out");
  if (v & kErrInvalidArg)
    return fail(HS_ERR_INVALID_ARG, "a kernel saw invalid data (row length or map entry)");
  return HS_OK;
}

hs_status hs_memcpy_async(void* dst, const void* src, size_t bytes, hs_stream_t stream) {
  clear_msg();
  if (bytes == 0) return HS_OK;
  if (!dst || !src) return fail(HS_ERR_INVALID_ARG, "NULL pointer");
  // One copy, its direction from unified addressing (pinned or pageable
  // host memory, or device memory, on either side).
  return cuda_fail(cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDefault,
                                   reinterpret_cast<cudaStream_t>(stream)),
                   "copy");
}

}  // extern "C"
