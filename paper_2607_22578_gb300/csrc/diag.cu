// Diagnostics: what streaming the valid prefixes of a row layout costs, with
// no hashing.  The merge (Section 3.3 (I)) reads every row's first len
// tokens once to fingerprint it; rows are zero-padded to a stride, so the
// bytes read are scattered prefixes of fixed-stride rows.  This kernel reads
// exactly those bytes with one of several access patterns and folds them
// into a checksum (so no load is dropped), giving the achievable DRAM rate
// for the layout that the fingerprint and verify kernels can be measured
// against.  It takes no part in the method.
//
// Patterns:
//   0  warp per row, 16 bytes per lane: each warp instruction reads 512
//      consecutive bytes of one row (coalesced); four instructions in flight
//   1  lane per row, 32-byte loads: each warp instruction reads one 32-byte
//      piece of 32 different rows (the fingerprint chunk kernel's pattern)
//   2  warp per row over the whole padded row (stride tokens), 16 bytes per
//      lane: the padding is read too
#include "hs_internal.cuh"

namespace hs {
namespace {

__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void ld_stream32(const void* p, uint32_t* x) {
  asm volatile("ld.global.nc.L1::no_allocate.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(x[0]), "=r"(x[1]), "=r"(x[2]), "=r"(x[3]), "=r"(x[4]), "=r"(x[5]),
                 "=r"(x[6]), "=r"(x[7])
               : "l"(p));
}

__device__ __forceinline__ int32_t row_len(const int32_t* lens, int64_t r, int32_t stride) {
  const int32_t L = lens ? __ldg(lens + r) : stride;
  return L < 0 ? 0 : (L > stride ? stride : L);
}

// Pattern 0 (full = false) and 2 (full = true): warp per row.
template <bool FULL>
__global__ void __launch_bounds__(256) stream_rows_warp_kernel(const int32_t* __restrict__ tokens,
                                                               int64_t n, int32_t stride,
                                                               const int32_t* __restrict__ lens,
                                                               unsigned* checksum) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  uint32_t acc = 0;
  for (int64_t r = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < n; r += warps) {
    const int32_t L = FULL ? stride : row_len(lens, r, stride);
    const int32_t pieces = L >> 2;                       // whole 16-byte pieces
    const uint4* p = reinterpret_cast<const uint4*>(tokens + r * (int64_t)stride);
    for (int32_t j0 = 0; j0 < pieces; j0 += 128) {
      uint4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int32_t j = j0 + u * 32 + lane;
        v[u] = j < pieces ? ld_stream16(p + j) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) acc ^= v[u].x ^ v[u].y ^ v[u].z ^ v[u].w;
    }
    const int32_t t = (pieces << 2) + lane;               // the last L mod 4 tokens
    if (t < L) acc ^= (uint32_t)__ldg(tokens + r * (int64_t)stride + t);
  }
  acc = __reduce_xor_sync(0xffffffffu, acc);
  if (lane == 0) atomicXor(checksum, acc);
}

// Pattern 1: lane per row, 32-byte pieces (rows are 32-byte aligned).
__global__ void __launch_bounds__(256) stream_rows_lane_kernel(const int32_t* __restrict__ tokens,
                                                               int64_t n, int32_t stride,
                                                               const int32_t* __restrict__ lens,
                                                               unsigned* checksum) {
  const int64_t threads = (int64_t)gridDim.x * blockDim.x;
  uint32_t acc = 0;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n; r += threads) {
    const int32_t L = row_len(lens, r, stride);
    const int32_t* row = tokens + r * (int64_t)stride;
    int32_t t = 0;
    for (; t + 32 <= L; t += 32) {
      uint32_t x[32];
#pragma unroll
      for (int u = 0; u < 4; ++u) ld_stream32(row + t + 8 * u, x + 8 * u);
#pragma unroll
      for (int u = 0; u < 32; ++u) acc ^= x[u];
    }
    for (; t < L; ++t) acc ^= (uint32_t)__ldg(row + t);
  }
  acc = __reduce_xor_sync(0xffffffffu, acc);
  if ((threadIdx.x & 31) == 0) atomicXor(checksum, acc);
}

}  // namespace
}  // namespace hs

/*
 * Diagnostics only (declared in hs.h as hs_debug_stream_rows).
 */
extern "C" hs_status hs_debug_stream_rows(const int32_t* tokens, int64_t n_rows, int32_t row_stride,
                                          const int32_t* lens, int32_t pattern,
                                          uint32_t* checksum_dev, int32_t blocks_per_sm,
                                          hs_stream_t stream) {
  using namespace hs;
  clear_last_error();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (n_rows < 0 || row_stride < 0) return fail(HS_ERR_INVALID_ARG, "negative size");
  if (pattern < 0 || pattern > 2) return fail(HS_ERR_INVALID_ARG, "pattern outside [0, 2]");
  if (blocks_per_sm < 1 || blocks_per_sm > 8)
    return fail(HS_ERR_INVALID_ARG, "blocks_per_sm outside [1, 8]");
  if (n_rows == 0) return HS_OK;
  if (!tokens || !checksum_dev) return fail(HS_ERR_INVALID_ARG, "NULL pointer");
  if ((reinterpret_cast<uintptr_t>(tokens) & 31u) || row_stride % 8)
    return fail(HS_ERR_INVALID_ARG, "tokens must be 32-byte aligned with row_stride %% 8 == 0");
  if ((lens && reinterpret_cast<uintptr_t>(lens) % 4) || reinterpret_cast<uintptr_t>(checksum_dev) % 4)
    return fail(HS_ERR_INVALID_ARG, "misaligned pointer");
  const unsigned grid = (unsigned)(num_sms() * blocks_per_sm);
  if (pattern == 0)
    stream_rows_warp_kernel<false><<<grid, 256, 0, s>>>(tokens, n_rows, row_stride, lens,
                                                         checksum_dev);
  else if (pattern == 1)
    stream_rows_lane_kernel<<<grid, 256, 0, s>>>(tokens, n_rows, row_stride, lens, checksum_dev);
  else
    stream_rows_warp_kernel<true><<<grid, 256, 0, s>>>(tokens, n_rows, row_stride, lens,
                                                        checksum_dev);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "stream_rows launch");
}
