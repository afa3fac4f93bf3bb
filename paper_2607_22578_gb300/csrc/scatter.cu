// K8: row scatter / gather, dst[i, :] = src[map[i], :] — result sharing: the
// output of the kept node flows to every merged node (Section 3.3 (I);
// Appendix A.2).  Used with map = inverse to fan results back to workflows,
// and with map = unique_idx to gather the unique rows.
//
// HBM-bound copy.  The flat index space is (row, chunk) with chunks of 16, 4
// or 1 bytes; consecutive threads write consecutive chunks of dst (coalesced
// stores, streamed past L1/L2 with evict-first) and read consecutive chunks
// of one src row.  Each thread moves 2 chunks per iteration: on the
// dedup-heavy scatter (1536-byte rows, 614 MB written) that took 110 µs
// against 127 µs for 4 chunks and 125 µs for 1.
#include "hs_internal.cuh"

namespace hs {
namespace {

template <class T>
__device__ __forceinline__ T ld_chunk(const T* p) { return __ldg(p); }

template <class T>
__device__ __forceinline__ void st_chunk(T* p, const T& v) { __stcs(p, v); }

template <>
__device__ __forceinline__ void st_chunk<uint8_t>(uint8_t* p, const uint8_t& v) { *p = v; }

template <>
__device__ __forceinline__ uint8_t ld_chunk<uint8_t>(const uint8_t* p) { return *p; }

// row = g / cpr as one 64x64 high multiply: with magic = floor((2^64 - 1) / cpr)
// + 1 (the reciprocal rounded up), the quotient is exact for every g with
// g * cpr < 2^64, which the host checks for the largest g.
template <class T, int U>
__global__ void __launch_bounds__(256) scatter_kernel(const T* __restrict__ src, int64_t n_src,
                                                      const int32_t* __restrict__ map,
                                                      int64_t n_rows, uint32_t cpr,
                                                      uint64_t magic, T* __restrict__ dst,
                                                      unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int64_t total = n_rows * (int64_t)cpr;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t g0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g0 < total; g0 += stride * U) {
    T v[U];
    int64_t dsti[U];
    bool ok[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t g = g0 + (int64_t)u * stride;
      ok[u] = false;
      if (g < total) {
        const int64_t row = magic ? (int64_t)__umul64hi((uint64_t)g, magic) : g / cpr;
        const int64_t c = g - row * cpr;
        const int32_t m = __ldg(map + row);
        if (m < 0 || (int64_t)m >= n_src) {
          if (c == 0) set_error(err, kErrInvalidArg);
        } else {
          v[u] = ld_chunk(src + (int64_t)m * cpr + c);
          dsti[u] = g;
          ok[u] = true;
        }
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (ok[u]) st_chunk(dst + dsti[u], v[u]);
  }
}

template <class T>
hs_status launch_typed(const void* src, int64_t n_src, int64_t row_bytes, const int32_t* map,
                       int64_t n_rows, void* dst, cudaStream_t stream, unsigned* err) {
  constexpr int U = 2;
  const int64_t cpr = row_bytes / (int64_t)sizeof(T);
  const int64_t total = n_rows * cpr;
  int64_t blocks = (total + 256 * U - 1) / (256 * U);
  const int64_t cap = (int64_t)num_sms() * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  // Reciprocal multiply when (total - 1) * cpr fits in 64 bits (else divide).
  uint64_t magic = 0;
  const unsigned __int128 span = (unsigned __int128)(uint64_t)(total > 0 ? total - 1 : 0) * (uint64_t)cpr;
  if (cpr > 0 && (span >> 64) == 0) magic = ~0ull / (uint64_t)cpr + 1ull;
  launch_pdl(scatter_kernel<T, U>, dim3((unsigned)blocks), dim3(256), 0, stream,
             static_cast<const T*>(src), n_src, map, n_rows, (uint32_t)cpr, magic,
             static_cast<T*>(dst), err);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "scatter launch");
}

}  // namespace

hs_status launch_scatter(const void* src, int64_t n_src, int64_t row_bytes, const int32_t* map,
                         int64_t n_rows, void* dst, cudaStream_t stream) {
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const uintptr_t a = reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst);
  if ((a & 15u) == 0 && row_bytes % 16 == 0)
    return launch_typed<uint4>(src, n_src, row_bytes, map, n_rows, dst, stream, err);
  if ((a & 3u) == 0 && row_bytes % 4 == 0)
    return launch_typed<uint32_t>(src, n_src, row_bytes, map, n_rows, dst, stream, err);
  return launch_typed<uint8_t>(src, n_src, row_bytes, map, n_rows, dst, stream, err);
}

}  // namespace hs
