// K1 + K2 + K5 fused for a small query batch: fingerprint every query row,
// merge exactly-equal rows into unique queries with an inverse map, and
// gather the unique rows for retrieval — one launch.
//
// Paper: the signature of a node (Section 3.3, Eq. 2), the merge of a node
// into an equal node already in the window (Section 3.3, "Dynamic Fusion and
// Reuse Mechanism" (I)) and the merge sets M(v*) executed once (Appendix A.2).
// The results are those of hs_fingerprint, hs_unique_inverse and
// hs_scatter_results(queries, unique_idx) called in turn.
//
// Small batches are latency-bound: each of those calls is a few microseconds
// of launch and dependency latency around very little work.  Here every CTA
// runs the whole merge on its own — the fingerprints of all rows (one thread
// per row), the hash table in shared memory, the verification, the scan —
// so the CTAs never wait for one another, and they split only the final
// gather.  The redundant work is cheap at these sizes: at most 256 rows,
// read from L2.  CTA 0 alone writes fingerprints, unique_idx, inverse and the
// unique count.
//
// Exactness: rows are grouped by fingerprint (the table keeps the smallest
// row index per fingerprint), then every row whose group leader is another
// row is compared with it in full.  A row that differs from its leader (a
// fingerprint collision) is re-grouped by a warp in ascending row order:
// its leader is the first earlier row with the same fingerprint that leads
// its own group and has equal contents, else itself.
#include "fnv.cuh"
#include "hs_internal.cuh"
#include "row_table.cuh"

namespace hs {
namespace {

using namespace table;

constexpr int kQmThreads = 256;             // one thread per query row
constexpr int kQmMaxRows = kQmThreads;
constexpr int kQmLog2 = table_log2(kQmMaxRows);
constexpr int kQmSlots = (1 << kQmLog2) + 1;
constexpr int kQmMaxCtas = 32;
constexpr int kQmChunk = 8;                 // 16-byte vectors per register chunk (32 words)
constexpr int kQmUnroll = 4;                // independent 16-byte copies in flight per thread

__device__ __forceinline__ bool same4(const uint4& a, const uint4& b) {
  return a.x == b.x && a.y == b.y && a.z == b.z && a.w == b.w;
}

__global__ void __launch_bounds__(kQmThreads) merge_queries_kernel(
    const uint4* __restrict__ q, int n, int nv, uint64_t seed, const uint64_t* __restrict__ fp_in,
    uint64_t* __restrict__ fp_out, int32_t* __restrict__ n_unique,
    int32_t* __restrict__ unique_idx, int32_t* __restrict__ inverse, uint4* __restrict__ uq) {
  pdl_wait();
  pdl_trigger();
  __shared__ uint64_t s_fp[kQmMaxRows];
  __shared__ uint64_t s_keys[kQmSlots];
  __shared__ uint32_t s_idx[kQmSlots];
  __shared__ int32_t s_rep[kQmMaxRows];
  __shared__ int32_t s_uid[kQmMaxRows];
  __shared__ int32_t s_uidx[kQmMaxRows];
  __shared__ int32_t s_list[kQmMaxRows];
  __shared__ uint8_t s_diff[kQmMaxRows];
  __shared__ int32_t s_warp[kQmThreads / 32];
  __shared__ int32_t s_nlist, s_ncoll;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int log2T = table_log2(n);
  const int T1 = (1 << log2T) + 1;
  const bool row = tid < n;

  for (int s = tid; s < T1; s += kQmThreads) {
    s_keys[s] = kEmpty;
    s_idx[s] = kNoRow;
  }
  s_diff[tid] = 0;
  if (tid == 0) s_nlist = s_ncoll = 0;

  // 1. fingerprint of row tid: FNV-1a over its octets, one chunk of 32 words
  //    loaded ahead of the chunk being hashed
  uint64_t f = 0;
  if (row) {
    if (fp_in) {
      f = __ldg(fp_in + tid);
    } else {
      const uint4* r = q + (size_t)tid * nv;
      uint32_t lo = (uint32_t)seed, hi = (uint32_t)(seed >> 32);
      uint4 cur[kQmChunk], nxt[kQmChunk];
#pragma unroll
      for (int j = 0; j < kQmChunk; ++j) cur[j] = j < nv ? __ldg(r + j) : make_uint4(0, 0, 0, 0);
      for (int c0 = 0; c0 < nv; c0 += kQmChunk) {
#pragma unroll
        for (int j = 0; j < kQmChunk; ++j)
          nxt[j] = c0 + kQmChunk + j < nv ? __ldg(r + c0 + kQmChunk + j) : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int j = 0; j < kQmChunk; ++j) {
          if (c0 + j < nv) {
            fnv::hash_word_full(lo, hi, cur[j].x);
            fnv::hash_word_full(lo, hi, cur[j].y);
            fnv::hash_word_full(lo, hi, cur[j].z);
            fnv::hash_word_full(lo, hi, cur[j].w);
          }
        }
#pragma unroll
        for (int j = 0; j < kQmChunk; ++j) cur[j] = nxt[j];
      }
      f = ((uint64_t)hi << 32) | lo;
    }
    s_fp[tid] = f;
    if (blockIdx.x == 0 && fp_out) fp_out[tid] = f;
  }
  __syncthreads();

  // 2. table: each fingerprint's smallest row index; rep = that row
  insert_row(s_keys, s_idx, log2T, row, f, (uint32_t)tid);
  __syncthreads();
  int32_t rep = tid;
  if (row) {
    const uint32_t v = s_idx[find_key(s_keys, f, log2T)];
    rep = v < (uint32_t)n ? (int32_t)v : tid;
    s_rep[tid] = rep;
    if (rep != tid) s_list[atomicAdd(&s_nlist, 1)] = tid;
  }
  __syncthreads();

  // 3. verify every listed row against its leader, all 16-byte pairs in flight
  const int m = s_nlist;
  const int items = m * nv;
  for (int b = tid; b < items; b += kQmThreads * kQmUnroll) {
    uint4 x[kQmUnroll], y[kQmUnroll];
    int ra[kQmUnroll];
#pragma unroll
    for (int u = 0; u < kQmUnroll; ++u) {
      const int it = b + u * kQmThreads;
      ra[u] = -1;
      if (it < items) {
        const int li = it / nv, v = it - li * nv;
        ra[u] = s_list[li];
        x[u] = __ldg(q + (size_t)ra[u] * nv + v);
        y[u] = __ldg(q + (size_t)s_rep[ra[u]] * nv + v);
      }
    }
#pragma unroll
    for (int u = 0; u < kQmUnroll; ++u)
      if (ra[u] >= 0 && !same4(x[u], y[u])) s_diff[ra[u]] = 1;
  }
  __syncthreads();
  if (row && s_diff[tid]) atomicAdd(&s_ncoll, 1);
  __syncthreads();

  // 4. collisions (rows that differ from their leader): warp 0, ascending
  if (s_ncoll > 0 && warp == 0) {
    for (int a0 = 0; a0 < n; a0 += 32) {
      unsigned cm = __ballot_sync(0xffffffffu, a0 + lane < n && s_diff[a0 + lane]);
      while (cm) {
        const int a = a0 + __ffs(cm) - 1;
        cm &= cm - 1;
        const uint64_t fa = s_fp[a];
        int found = a;
        for (int j0 = 0; j0 < a && found == a; j0 += 32) {
          const int j = j0 + lane;
          unsigned cand = __ballot_sync(0xffffffffu, j < a && s_fp[j] == fa && s_rep[j] == j);
          while (cand && found == a) {
            const int jj = j0 + __ffs(cand) - 1;
            cand &= cand - 1;
            bool eq = true;
            for (int v = lane; v < nv; v += 32)
              eq &= same4(__ldg(q + (size_t)jj * nv + v), __ldg(q + (size_t)a * nv + v));
            if (__all_sync(0xffffffffu, eq)) found = jj;
          }
        }
        if (lane == 0) s_rep[a] = found;
        __syncwarp();
      }
    }
  }
  __syncthreads();

  // 5. ordinals in first-occurrence order
  if (row) rep = s_rep[tid];
  const bool lead = row && rep == tid;
  const unsigned bal = __ballot_sync(0xffffffffu, lead);
  if (lane == 0) s_warp[warp] = __popc(bal);
  __syncthreads();
  int32_t off = 0, total = 0;
#pragma unroll
  for (int w = 0; w < kQmThreads / 32; ++w) {
    off += w < warp ? s_warp[w] : 0;
    total += s_warp[w];
  }
  if (lead) {
    const int32_t u = off + __popc(bal & ((1u << lane) - 1u));
    s_uid[tid] = u;
    s_uidx[u] = tid;
  }
  __syncthreads();
  if (blockIdx.x == 0 && row) {
    inverse[tid] = s_uid[rep];
    unique_idx[tid] = tid < total ? s_uidx[tid] : 0;
    if (tid == 0) *n_unique = total;
  }

  // 6. gather the unique rows, split over the CTAs
  const int gitems = total * nv;
  const int gstride = gridDim.x * kQmThreads;
  for (int b = blockIdx.x * kQmThreads + tid; b < gitems; b += gstride * kQmUnroll) {
    uint4 x[kQmUnroll];
    int dst[kQmUnroll];
#pragma unroll
    for (int u = 0; u < kQmUnroll; ++u) {
      const int it = b + u * gstride;
      dst[u] = -1;
      if (it < gitems) {
        const int g = it / nv, v = it - g * nv;
        x[u] = __ldg(q + (size_t)s_uidx[g] * nv + v);
        dst[u] = it;
      }
    }
#pragma unroll
    for (int u = 0; u < kQmUnroll; ++u)
      if (dst[u] >= 0) uq[dst[u]] = x[u];
  }
}

}  // namespace

hs_status launch_merge_queries(const uint16_t* queries, int64_t n, int32_t dim, uint64_t seed,
                               const uint64_t* fp_in, uint64_t* fp_out, int32_t* n_unique,
                               int32_t* unique_idx, int32_t* inverse, uint16_t* uq,
                               cudaStream_t stream) {
  if (n == 0)
    return cuda_fail(cudaMemsetAsync(n_unique, 0, sizeof(int32_t), stream), "n_unique clear");
  const int nv = dim / 8;                     // 16-byte vectors per row
  const int64_t work = n * (int64_t)nv;
  int64_t grid = (work + kQmThreads * kQmUnroll - 1) / (kQmThreads * kQmUnroll);
  grid = grid < 1 ? 1 : (grid > kQmMaxCtas ? kQmMaxCtas : grid);
  launch_pdl(merge_queries_kernel, dim3((unsigned)grid), dim3(kQmThreads), 0, stream,
             reinterpret_cast<const uint4*>(queries), (int)n, nv, seed, fp_in, fp_out, n_unique,
             unique_idx, inverse, reinterpret_cast<uint4*>(uq));
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "merge_queries launch");
}

}  // namespace hs
