// Asynchronous cache reuse across batches (Section 3.3, "Dynamic Fusion and
// Reuse Mechanism" (II)): a node that equals a node completed earlier takes
// its result instead of executing.  Here the nodes are merged queries and
// the result is their retrieval top-k; the cache lives in device memory the
// caller provides and persists across batches.
//
// Layout (hs_cache_bytes): a header, then S slots (S a power of two, at
// least 8) grouped into sets of kWays consecutive slots.  A slot holds the
// query's fingerprint, state, last-use epoch, the query vector itself (so a
// hit is confirmed by a full comparison: a fingerprint collision can never
// return another query's result) and its k scores and ids.
//
// Per batch:
//   lookup  one warp per merged query: the ways of the fingerprint's set
//           whose key matches are compared in full; a hit copies the
//           cached result to the query's output row and refreshes the
//           slot's epoch; a miss appends the query to a miss list and
//           copies its vector to a compact buffer for retrieval;
//   insert  one warp per miss, after the retrieval of the compact buffer:
//           claims the set's empty way, else its least recently used way,
//           with a compare-and-swap on the slot state, writes key, vector
//           and result, then publishes the slot; the result also goes to
//           the query's output row.
// Calls on one stream are ordered, so a batch sees every insert of the
// batches before it.  A query that equals one still being retrieved by a
// concurrent stream is not waited for: it misses and is retrieved again (a
// kernel never waits for another kernel here).
//
// Concurrent streams.  A slot's state word carries, above its two state
// bits, a generation count that every claim advances.  A lookup reads the
// state, then the slot's key, vector and result (from L2, never from a
// stale L1 line), then the state again: a hit needs both reads to show the
// same ready generation.  An insert that claimed the slot in between (to
// evict it) changes the word, and the lookup takes the miss path, so a hit
// never returns a half-written or replaced entry.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kWays = 8;
constexpr uint32_t kEmptyState = 0, kBusy = 1, kReady = 2;   // state word: generation << 2 | state
constexpr uint32_t kStateMask = 3u;
constexpr uint32_t kMagic = 0x48534331u;   // "HSC1"

struct CacheHeader {
  uint32_t magic, slots, dim, k;
  uint32_t epoch, pad0;
  unsigned long long hits, misses;
};

struct CacheView {
  CacheHeader* hdr;
  uint64_t* keys;
  uint32_t* state;
  uint32_t* used;
  uint16_t* vec;
  float* scores;
  int32_t* ids;
  uint32_t slots;
  int dim, k;
};

constexpr size_t a256(size_t x) { return (x + 255) & ~(size_t)255; }

CacheView view_of(void* base, uint32_t S, int dim, int k) {
  char* p = static_cast<char*>(base);
  CacheView v{};
  v.hdr = reinterpret_cast<CacheHeader*>(p);
  size_t o = a256(sizeof(CacheHeader));
  v.keys = reinterpret_cast<uint64_t*>(p + o);   o += a256((size_t)S * 8);
  v.state = reinterpret_cast<uint32_t*>(p + o);  o += a256((size_t)S * 4);
  v.used = reinterpret_cast<uint32_t*>(p + o);   o += a256((size_t)S * 4);
  v.vec = reinterpret_cast<uint16_t*>(p + o);    o += a256((size_t)S * dim * 2);
  v.scores = reinterpret_cast<float*>(p + o);    o += a256((size_t)S * k * 4);
  v.ids = reinterpret_cast<int32_t*>(p + o);
  v.slots = S;
  v.dim = dim;
  v.k = k;
  return v;
}

size_t bytes_of(uint32_t S, int dim, int k) {
  return a256(sizeof(CacheHeader)) + a256((size_t)S * 8) + 2 * a256((size_t)S * 4) +
         a256((size_t)S * dim * 2) + 2 * a256((size_t)S * k * 4);
}

uint32_t slots_for(int64_t capacity) {
  uint64_t S = kWays;
  while ((int64_t)S < capacity) S <<= 1;
  return (uint32_t)S;
}

__device__ __forceinline__ uint32_t set_of(uint64_t f, uint32_t S) {
  const uint32_t sets = S / kWays;
  return (uint32_t)((f * 0x9E3779B97F4A7C15ull) >> 32) & (sets - 1u);
}

// Warp-wide equality of two rows of nv 16-byte pieces.
__device__ __forceinline__ bool rows_equal(const uint4* a, const uint4* b, int nv, int lane) {
  bool eq = true;
#pragma unroll 1
  for (int v = lane; v < nv; v += 32) {
    const uint4 x = __ldg(a + v), y = __ldcg(b + v);
    eq &= x.x == y.x && x.y == y.y && x.z == y.z && x.w == y.w;
  }
  return __all_sync(0xffffffffu, eq);
}

__global__ void cache_init_kernel(CacheView c) {
  pdl_wait();
  pdl_trigger();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; s < c.slots; s += stride) {
    c.state[s] = kEmptyState;
    c.used[s] = 0;
    c.keys[s] = 0;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    c.hdr->magic = kMagic;
    c.hdr->slots = c.slots;
    c.hdr->dim = (uint32_t)c.dim;
    c.hdr->k = (uint32_t)c.k;
    c.hdr->epoch = 1;
    c.hdr->hits = 0;
    c.hdr->misses = 0;
  }
}

__device__ __forceinline__ bool header_ok(const CacheView& c, unsigned* err) {
  const CacheHeader* h = c.hdr;
  const bool ok = h->magic == kMagic && h->slots == c.slots && h->dim == (uint32_t)c.dim &&
                  h->k == (uint32_t)c.k;
  if (!ok && threadIdx.x == 0 && blockIdx.x == 0) set_error(err, kErrInvalidArg);
  return ok;
}

__global__ void __launch_bounds__(256) cache_lookup_kernel(
    CacheView c, const uint4* __restrict__ queries, const uint64_t* __restrict__ fp,
    const int32_t* __restrict__ rows, int64_t Qmax, const int32_t* __restrict__ count_dev,
    float* __restrict__ out_s, int32_t* __restrict__ out_i, int32_t* __restrict__ miss_list,
    int32_t* __restrict__ n_miss, uint4* __restrict__ miss_q, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  if (!header_ok(c, err)) return;
  const int lane = threadIdx.x & 31;
  const int nv = c.dim / 8, k = c.k;
  int64_t Q = Qmax;
  if (count_dev) {
    const int64_t n = __ldg(count_dev);
    Q = n < 0 ? 0 : (n > Qmax ? Qmax : n);
  }
  const uint32_t epoch = *reinterpret_cast<volatile uint32_t*>(&c.hdr->epoch);
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t u = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; u < Q; u += nwarps) {
    const uint64_t f = __ldg(fp + (rows ? (int64_t)__ldg(rows + u) : u));
    const uint32_t base = set_of(f, c.slots) * kWays;
    const uint4* qrow = queries + u * nv;
    bool match = false;
    uint32_t st = 0;
    if (lane < kWays) {
      st = *reinterpret_cast<volatile uint32_t*>(c.state + base + lane);
      __threadfence();   // order the state read before the key
      match = (st & kStateMask) == kReady && __ldcg(c.keys + base + lane) == f;
    }
    unsigned cand = __ballot_sync(0xffffffffu, match);
    int hit = -1;
    while (cand && hit < 0) {
      const int w = __ffs(cand) - 1;
      cand &= cand - 1;
      const uint32_t seen = __shfl_sync(0xffffffffu, st, w);
      const uint32_t s = base + w;
      __threadfence();   // order the state read before the slot contents
      if (!rows_equal(qrow, reinterpret_cast<const uint4*>(c.vec) + (int64_t)s * nv, nv, lane))
        continue;
      // copy the result, then confirm that no insert claimed the slot meanwhile;
      // a row copied from a changed slot is overwritten by the miss path
      for (int j = lane; j < k; j += 32) {
        out_s[u * k + j] = __ldcg(c.scores + (int64_t)s * k + j);
        out_i[u * k + j] = __ldcg(c.ids + (int64_t)s * k + j);
      }
      __syncwarp();
      __threadfence();
      uint32_t again = 0;
      if (lane == 0) again = *reinterpret_cast<volatile uint32_t*>(c.state + s);
      if (__shfl_sync(0xffffffffu, again, 0) == seen) hit = w;
    }
    if (hit >= 0) {
      const uint32_t s = base + hit;
      if (lane == 0) {
        c.used[s] = epoch;
        atomicAdd(&c.hdr->hits, 1ull);
      }
    } else {
      int32_t pos = 0;
      if (lane == 0) {
        pos = atomicAdd(n_miss, 1);
        miss_list[pos] = (int32_t)u;
        atomicAdd(&c.hdr->misses, 1ull);
      }
      pos = __shfl_sync(0xffffffffu, pos, 0);
#pragma unroll 1
      for (int v = lane; v < nv; v += 32) miss_q[(int64_t)pos * nv + v] = __ldg(qrow + v);
    }
  }
}

__global__ void __launch_bounds__(256) cache_insert_kernel(
    CacheView c, const int32_t* __restrict__ miss_list, const int32_t* __restrict__ n_miss_dev,
    int64_t Qmax, const uint4* __restrict__ miss_q, const uint64_t* __restrict__ fp,
    const int32_t* __restrict__ rows, const float* __restrict__ miss_s,
    const int32_t* __restrict__ miss_i, float* __restrict__ out_s, int32_t* __restrict__ out_i,
    unsigned* err) {
  pdl_wait();
  pdl_trigger();
  if (!header_ok(c, err)) return;
  const int lane = threadIdx.x & 31;
  const int nv = c.dim / 8, k = c.k;
  int64_t M = __ldg(n_miss_dev);
  M = M < 0 ? 0 : (M > Qmax ? Qmax : M);
  const uint32_t epoch = *reinterpret_cast<volatile uint32_t*>(&c.hdr->epoch);
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < M; i += nwarps) {
    const int64_t u = __ldg(miss_list + i);
    for (int j = lane; j < k; j += 32) {                 // the result for this batch
      out_s[u * k + j] = miss_s[i * k + j];
      out_i[u * k + j] = miss_i[i * k + j];
    }
    const uint64_t f = __ldg(fp + (rows ? (int64_t)__ldg(rows + u) : u));
    const uint32_t base = set_of(f, c.slots) * kWays;
    // claim a way: empty first, then least recently used; a way another
    // miss of this batch claimed first is skipped
    int claimed = -1;
    uint32_t gen_busy = 0;
    for (int attempt = 0; attempt < kWays && claimed < 0; ++attempt) {
      uint32_t st = kBusy, age = 0xffffffffu;
      if (lane < kWays) {
        st = *reinterpret_cast<volatile uint32_t*>(c.state + base + lane) & kStateMask;
        age = st == kEmptyState ? 0u : (st == kReady ? c.used[base + lane] + 1u : 0xffffffffu);
      }
      // lowest (age, way) over the ways that are not busy
      uint64_t key = ((uint64_t)age << 8) | (uint64_t)(lane < kWays ? lane : 255);
      if (st == kBusy) key = ~0ull;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const uint64_t y = __shfl_xor_sync(0xffffffffu, key, o);
        key = y < key ? y : key;
      }
      if (key == ~0ull) break;                            // every way busy: not cached
      const int w = (int)(key & 0xff);
      uint32_t ok = 0;
      if (lane == w) {
        const uint32_t seen = *reinterpret_cast<volatile uint32_t*>(c.state + base + w);
        const uint32_t busy = (((seen >> 2) + 1u) << 2) | kBusy;   // next generation
        ok = (seen & kStateMask) != kBusy && atomicCAS(c.state + base + w, seen, busy) == seen
                 ? busy : 0u;
        __threadfence();   // the claim is visible before any write to the slot
      }
      ok = __shfl_sync(0xffffffffu, ok, w);
      if (ok) {
        claimed = w;
        gen_busy = ok;
      }
    }
    if (claimed < 0) continue;
    const uint32_t s = base + claimed;
    uint4* dst = reinterpret_cast<uint4*>(c.vec) + (int64_t)s * nv;
    for (int v = lane; v < nv; v += 32) dst[v] = __ldg(miss_q + i * nv + v);
    for (int j = lane; j < k; j += 32) {
      c.scores[(int64_t)s * k + j] = miss_s[i * k + j];
      c.ids[(int64_t)s * k + j] = miss_i[i * k + j];
    }
    if (lane == 0) {
      c.keys[s] = f;
      c.used[s] = epoch;
    }
    __threadfence();
    __syncwarp();
    if (lane == 0) atomicExch(c.state + s, (gen_busy & ~kStateMask) | kReady);   // publish
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) atomicAdd(&c.hdr->epoch, 1u);
}

}  // namespace

size_t cache_bytes(int64_t capacity, int32_t dim, int32_t k) {
  if (capacity < 1 || dim < 8 || k < 1) return 0;
  return bytes_of(slots_for(capacity), dim, k);
}

hs_status launch_cache_init(void* cache, int64_t capacity, int32_t dim, int32_t k,
                            cudaStream_t stream) {
  const CacheView c = view_of(cache, slots_for(capacity), dim, k);
  const int64_t blocks = ((int64_t)c.slots + 255) / 256;
  launch_pdl(cache_init_kernel, dim3((unsigned)(blocks < 4096 ? blocks : 4096)), dim3(256), 0,
             stream, c);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "cache init launch");
}

hs_status launch_cache_lookup(void* cache, int64_t capacity, int32_t dim, int32_t k,
                              const uint16_t* queries, const uint64_t* fp, const int32_t* rows,
                              int64_t Qmax, const int32_t* count_dev, float* out_s,
                              int32_t* out_i, int32_t* miss_list, int32_t* n_miss,
                              uint16_t* miss_q, cudaStream_t stream) {
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const CacheView c = view_of(cache, slots_for(capacity), dim, k);
  cudaError_t e = cudaMemsetAsync(n_miss, 0, sizeof(int32_t), stream);
  if (e != cudaSuccess) return cuda_fail(e, "miss count clear");
  if (Qmax == 0) return HS_OK;
  int64_t grid = (Qmax + 7) / 8;
  const int64_t cap = (int64_t)num_sms() * 8;
  if (grid > cap) grid = cap;
  launch_pdl(cache_lookup_kernel, dim3((unsigned)grid), dim3(256), 0, stream, c,
             reinterpret_cast<const uint4*>(queries), fp, rows, Qmax, count_dev, out_s, out_i,
             miss_list, n_miss, reinterpret_cast<uint4*>(miss_q), err);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "cache lookup launch");
}

hs_status launch_cache_insert(void* cache, int64_t capacity, int32_t dim, int32_t k,
                              const int32_t* miss_list, const int32_t* n_miss, int64_t Qmax,
                              const uint16_t* miss_q, const uint64_t* fp, const int32_t* rows,
                              const float* miss_s, const int32_t* miss_i, float* out_s,
                              int32_t* out_i, cudaStream_t stream) {
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const CacheView c = view_of(cache, slots_for(capacity), dim, k);
  int64_t grid = (Qmax + 7) / 8;
  const int64_t cap = (int64_t)num_sms() * 8;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  launch_pdl(cache_insert_kernel, dim3((unsigned)grid), dim3(256), 0, stream, c, miss_list, n_miss,
             Qmax, reinterpret_cast<const uint4*>(miss_q), fp, rows, miss_s, miss_i, out_s, out_i,
             err);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "cache insert launch");
}

hs_status cache_stats(const void* cache, unsigned long long* hits, unsigned long long* misses,
                      cudaStream_t stream) {
  CacheHeader h{};
  cudaError_t e = cudaMemcpyAsync(&h, cache, sizeof h, cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "cache header read");
  if (h.magic != kMagic) return fail(HS_ERR_INVALID_ARG, "not an initialised cache");
  *hits = h.hits;
  *misses = h.misses;
  return HS_OK;
}

}  // namespace hs
