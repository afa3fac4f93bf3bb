// Second retrieval stage of the RAG-with-rerank workflow (Section 4.1,
// "Workloads": a reranker scores the initial top-12 chunks and the top-8 by
// those scores are kept).  The reranker's model is not part of this library;
// its score is taken as the inner product of bf16 rerank vectors (a query
// vector and one vector per corpus chunk), accumulated in fp32:
//   s[q, j] = sum_t rq[q, t] * rc[cand[q, j], t],   j < k1,
// and each query keeps the k2 candidates first in (score descending, corpus
// index ascending).
//
// One warp per output row.  The work is a gather of k1 corpus rows per
// query, and with a few thousand output rows every row is resident at once:
// the kernel's time is the chain of dependent memory round trips of one row,
// not bandwidth.  So the chain is kept short: the map entry, the candidate
// ids, then per group of four candidates one round trip in which each lane
// requests all of its 16-byte pieces (l, l + 32, l + 64, l + 96) of the
// query row and the four candidate rows before the first product (d <= 1024;
// longer rows take one round trip per 1024 dimensions).  The four partial
// dot products are reduced with shuffles.  Lane c then holds candidate c's
// score; its rank is the number of candidates ahead of it in the order
// (ties between equal keys by lane), and the lanes of rank < k2 write their
// entry.  CTAs of two warps spread the rows evenly over the SMs.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kRrThreads = 64;
constexpr int kRrGroup = 4;                  // candidate rows in flight per warp
constexpr int kRrPieces = 4;                 // 16-byte pieces per lane and row in flight

__device__ __forceinline__ uint64_t rr_key(float s, int32_t id) {
  uint32_t u = __float_as_uint(s);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((uint64_t)u << 32) | (uint64_t)(0xffffffffu - (uint32_t)id);
}

// Eight bf16 products of two 16-byte pieces, added to acc in fp32.
__device__ __forceinline__ float dot8(const uint4& a, const uint4& b, float acc) {
  const uint32_t x[4] = {a.x, a.y, a.z, a.w}, y[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    acc = fmaf(__uint_as_float(x[i] << 16), __uint_as_float(y[i] << 16), acc);
    acc = fmaf(__uint_as_float(x[i] & 0xffff0000u), __uint_as_float(y[i] & 0xffff0000u), acc);
  }
  return acc;
}

__global__ void __launch_bounds__(kRrThreads) rerank_kernel(
    const uint4* __restrict__ rq, int64_t Qmax, const int32_t* __restrict__ count_dev,
    const uint4* __restrict__ rc, int64_t n_rc, int nv, const int32_t* __restrict__ cand, int k1,
    int k2, const int32_t* __restrict__ inv, int64_t n_out, float* __restrict__ out_s,
    int32_t* __restrict__ out_i, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  int64_t Q = Qmax;
  if (count_dev) {
    const int64_t c = __ldg(count_dev);
    Q = c < 0 ? 0 : (c > Qmax ? Qmax : c);
  }
  const int64_t R = inv ? n_out : Q;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t o = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; o < R; o += nwarps) {
    const int64_t q = inv ? (int64_t)__ldg(inv + o) : o;
    if (q < 0 || q >= Q) {                                   // warp-uniform
      if (lane == 0) set_error(err, kErrInvalidArg);
      continue;
    }
    int32_t id = -1;
    if (lane < k1) {
      id = __ldg(cand + q * k1 + lane);
      if (id >= n_rc) {
        set_error(err, kErrInvalidArg);
        id = -1;
      }
      if (id < 0) id = -1;                                  // absent: written as -1
    }
    const uint4* qrow = rq + q * nv;
    float score = 0.0f;
    for (int c0 = 0; c0 < k1; c0 += kRrGroup) {
      int32_t cid[kRrGroup];
      float acc[kRrGroup];
#pragma unroll
      for (int g = 0; g < kRrGroup; ++g) {
        cid[g] = __shfl_sync(0xffffffffu, id, (c0 + g) & 31);
        if (c0 + g >= k1) cid[g] = -1;
        acc[g] = 0.0f;
      }
      // Every piece of the group's rows that this lane reads in a round of
      // kRrPieces pieces is requested before the first product, so a round
      // costs one memory round trip (one per group for d <= 1024).
      for (int v0 = 0; v0 < nv; v0 += 32 * kRrPieces) {
        uint4 a[kRrPieces], b[kRrGroup][kRrPieces];
#pragma unroll
        for (int pc = 0; pc < kRrPieces; ++pc) {
          const int v = v0 + pc * 32 + lane;
          a[pc] = v < nv ? __ldg(qrow + v) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
          for (int g = 0; g < kRrGroup; ++g)
            b[g][pc] = (cid[g] >= 0 && v < nv) ? __ldg(rc + (int64_t)cid[g] * nv + v)
                                               : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int pc = 0; pc < kRrPieces; ++pc) {
          if (v0 + pc * 32 + lane < nv) {
#pragma unroll
            for (int g = 0; g < kRrGroup; ++g)
              if (cid[g] >= 0) acc[g] = dot8(a[pc], b[g][pc], acc[g]);
          }
        }
      }
#pragma unroll
      for (int g = 0; g < kRrGroup; ++g) {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) acc[g] += __shfl_xor_sync(0xffffffffu, acc[g], off);
        if (lane == c0 + g) score = acc[g];
      }
    }
    // rank of this lane's candidate; absent candidates (key 0) come last
    const uint64_t key = id >= 0 ? rr_key(score, id) : 0ull;
    int rank = 0;
    for (int j = 0; j < 32; ++j) {
      const uint64_t kj = __shfl_sync(0xffffffffu, key, j);
      rank += (kj > key) || (kj == key && j < lane);
    }
    if (lane < k1 && rank < k2) {
      out_s[o * k2 + rank] = id >= 0 ? score : __int_as_float(0xff800000);  // -inf
      out_i[o * k2 + rank] = id;
    }
  }
}

}  // namespace

hs_status launch_rerank(const uint16_t* rq, int64_t Qmax, const int32_t* count_dev,
                        const uint16_t* rc, int64_t n_rc, int32_t d, const int32_t* cand,
                        int32_t k1, int32_t k2, const int32_t* inv, int64_t n_out,
                        float* out_s, int32_t* out_i, cudaStream_t stream) {
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const int64_t rows = inv ? n_out : Qmax;
  if (rows == 0) return HS_OK;
  const int64_t warps_per_cta = kRrThreads / 32;
  int64_t grid = (rows + warps_per_cta - 1) / warps_per_cta;
  const int64_t cap = (int64_t)num_sms() * 16;
  if (grid > cap) grid = cap;
  launch_pdl(rerank_kernel, dim3((unsigned)grid), dim3(kRrThreads), 0, stream,
             reinterpret_cast<const uint4*>(rq), Qmax, count_dev,
             reinterpret_cast<const uint4*>(rc), n_rc, d / 8, cand, k1, k2, inv, n_out, out_s,
             out_i, err);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "rerank launch");
}

}  // namespace hs
