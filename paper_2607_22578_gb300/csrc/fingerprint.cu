// K1: per-row 64-bit FNV-1a fingerprints over int32 token rows — the D_in
// part of the node semantic signature Sig(v) (Section 3.3, Eq. 2).
//
// FNV-1a is a serial chain over the octets of one row, so parallelism comes
// from rows: each lane of a warp owns one row at a time and streams it in
// 128-byte blocks of 16-byte loads, the next block in flight while the current
// one is hashed.  Rows have
// different lengths; a lane that finishes its row claims the next unclaimed
// row of its warp's range (warp-synchronous ballot, no atomics), so the
// lanes of a warp stay busy until the range is drained.
//
// Arithmetic: h = (hi:lo) as two 32-bit words; a multiply by the prime
// 2^40 + 0x1b3 is one wide 32x32 multiply, one multiply-add and one
// shift-add.  When a token's two high octets are zero (every token below
// 65536), the last two rounds "xor 0, multiply by prime" collapse exactly into
// one multiply by prime^3 mod 2^64 — xor with zero is the identity — so the
// result is bit-identical to the octet-wise definition.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr uint64_t kPrime = 1099511628211ull;  // 2^40 + 0x1b3
constexpr uint64_t kPrime3 = kPrime * kPrime * kPrime;  // mod 2^64
constexpr uint32_t kP3Lo = (uint32_t)(kPrime3 & 0xffffffffull);
constexpr uint32_t kP3Hi = (uint32_t)(kPrime3 >> 32);

__device__ __forceinline__ void mul_prime(uint32_t& lo, uint32_t& hi) {
  // (hi * 2^32 + lo) * (2^40 + 0x1b3) mod 2^64
  const uint64_t t = (uint64_t)lo * 0x1b3u;
  hi = (uint32_t)(t >> 32) + hi * 0x1b3u + (lo << 8);
  lo = (uint32_t)t;
}

__device__ __forceinline__ void mul_prime3(uint32_t& lo, uint32_t& hi) {
  const uint64_t t = (uint64_t)lo * kP3Lo;
  hi = (uint32_t)(t >> 32) + lo * kP3Hi + hi * kP3Lo;
  lo = (uint32_t)t;
}

// Octet-wise rounds for one token, little-endian octet order.
__device__ __forceinline__ void hash_word_full(uint32_t& lo, uint32_t& hi, uint32_t w) {
  lo ^= (w & 0xffu);
  mul_prime(lo, hi);
  lo ^= ((w >> 8) & 0xffu);
  mul_prime(lo, hi);
  lo ^= ((w >> 16) & 0xffu);
  mul_prime(lo, hi);
  lo ^= (w >> 24);
  mul_prime(lo, hi);
}

// Same result for a token below 65536.
__device__ __forceinline__ void hash_word_small(uint32_t& lo, uint32_t& hi, uint32_t w) {
  lo ^= (w & 0xffu);
  mul_prime(lo, hi);
  lo ^= (w >> 8);
  mul_prime3(lo, hi);
}

__device__ __forceinline__ void hash_word(uint32_t& lo, uint32_t& hi, uint32_t w) {
  if (w < 0x10000u)
    hash_word_small(lo, hi, w);
  else
    hash_word_full(lo, hi, w);
}

__device__ __forceinline__ void hash4(uint32_t& lo, uint32_t& hi, const int4 v) {
  const uint32_t a = (uint32_t)v.x, b = (uint32_t)v.y, c = (uint32_t)v.z, d = (uint32_t)v.w;
  if (((a | b | c | d) >> 16) == 0u) {
    hash_word_small(lo, hi, a);
    hash_word_small(lo, hi, b);
    hash_word_small(lo, hi, c);
    hash_word_small(lo, hi, d);
  } else {
    hash_word(lo, hi, a);
    hash_word(lo, hi, b);
    hash_word(lo, hi, c);
    hash_word(lo, hi, d);
  }
}

__device__ __forceinline__ int4 ld_stream16(const int32_t* p) {
  int4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.s32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void hash_partial(uint32_t& lo, uint32_t& hi, const int4 v, int w) {
  hash_word(lo, hi, (uint32_t)v.x);
  if (w > 1) hash_word(lo, hi, (uint32_t)v.y);
  if (w > 2) hash_word(lo, hi, (uint32_t)v.z);
}

constexpr int kBlockPieces = 8;  // 8 x 16 B = 32 tokens per block

// VEC: tokens 16-byte aligned and row_stride % 4 == 0, so every row starts
// on a 16-byte boundary and its ceil(len/4) 16-byte pieces lie inside the
// row.  A lane hashes one 128-byte block of its row while the next block is
// already in flight.
template <bool VEC>
__global__ void __launch_bounds__(256) fingerprint_kernel(
    const int32_t* __restrict__ tokens, int64_t n, int32_t stride,
    const int32_t* __restrict__ lens, uint64_t seed, uint64_t* __restrict__ fp_out,
    int64_t rows_per_warp, unsigned* err) {
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t r_begin = warp * rows_per_warp;
  if (r_begin >= n) return;
  const int64_t r_end = min(n, r_begin + rows_per_warp);
  const uint32_t seed_lo = (uint32_t)seed, seed_hi = (uint32_t)(seed >> 32);

  bool busy = false;
  int64_t row = 0;
  int32_t len = 0, pos = 0, pieces = 0, full = 0, blk = 0;
  uint32_t lo = seed_lo, hi = seed_hi;
  const int32_t* src = tokens;
  int4 buf[kBlockPieces];

  auto load_block = [&](int b, int4 (&dst)[kBlockPieces]) {
    const int4* base = reinterpret_cast<const int4*>(src) + kBlockPieces * b;
#pragma unroll
    for (int i = 0; i < kBlockPieces; ++i)
      if (kBlockPieces * b + i < pieces) dst[i] = ld_stream16(reinterpret_cast<const int32_t*>(base + i));
  };

  // Start row r on this lane.  Rows of length 0 are finished at once; rows
  // with an invalid length are reported and written as 0.
  auto begin_row = [&](int64_t r) {
    row = r;
    pos = 0;
    blk = 0;
    lo = seed_lo;
    hi = seed_hi;
    src = tokens + r * (int64_t)stride;
    int32_t L = lens ? __ldg(lens + r) : stride;
    if (L < 0 || L > stride) {
      set_error(err, kErrInvalidArg);
      fp_out[r] = 0ull;
      busy = false;
      return;
    }
    len = L;
    if (L == 0) {
      fp_out[r] = seed;
      busy = false;
      return;
    }
    pieces = (L + 3) >> 2;
    full = L >> 2;
    if (VEC) load_block(0, buf);
    busy = true;
  };

  int64_t next = r_begin;
  for (;;) {
    // Hand unclaimed rows to idle lanes, in lane order.
    unsigned idle = __ballot_sync(0xffffffffu, !busy);
    while (idle != 0u && next < r_end) {
      const int64_t avail = r_end - next;
      const int rank = __popc(idle & lanemask_lt());
      if (!busy && rank < avail) begin_row(next + rank);
      next += min((int64_t)__popc(idle), avail);
      idle = __ballot_sync(0xffffffffu, !busy);
    }
    if (!__any_sync(0xffffffffu, busy)) break;
    if (busy) {
      if (VEC) {
        int4 nxt[kBlockPieces];
        const bool more = kBlockPieces * (blk + 1) < pieces;
        if (more) load_block(blk + 1, nxt);
#pragma unroll
        for (int i = 0; i < kBlockPieces; ++i) {
          const int pi = kBlockPieces * blk + i;
          if (pi < full)
            hash4(lo, hi, buf[i]);
          else if (pi < pieces)
            hash_partial(lo, hi, buf[i], len & 3);
        }
        if (more) {
#pragma unroll
          for (int i = 0; i < kBlockPieces; ++i) buf[i] = nxt[i];
          ++blk;
        } else {
          fp_out[row] = ((uint64_t)hi << 32) | lo;
          busy = false;
        }
      } else {
        const int32_t rem = len - pos;
        const int32_t m = rem < 16 ? rem : 16;
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (j < m) hash_word(lo, hi, (uint32_t)__ldg(src + pos + j));
        pos += m;
        if (pos >= len) {
          fp_out[row] = ((uint64_t)hi << 32) | lo;
          busy = false;
        }
      }
    }
  }
}

int resident_warps(const void* kernel) {
  static int cached[2] = {0, 0};
  const int slot = (kernel == (const void*)fingerprint_kernel<true>) ? 0 : 1;
  if (cached[slot] == 0) {
    int blocks = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks, kernel, 256, 0) != cudaSuccess ||
        blocks < 1)
      blocks = 1;
    cached[slot] = blocks * 8 * num_sms();
  }
  return cached[slot];
}

}  // namespace

hs_status launch_fingerprint(const int32_t* tokens, int64_t n, int32_t stride,
                             const int32_t* lens, uint64_t seed, uint64_t* fp_out,
                             cudaStream_t stream) {
  const bool vec = ((reinterpret_cast<uintptr_t>(tokens) & 15u) == 0) && (stride % 4 == 0);
  const void* kfn = vec ? (const void*)fingerprint_kernel<true>
                        : (const void*)fingerprint_kernel<false>;
  const int64_t warps_target = resident_warps(kfn);
  // At least one row per lane; more rows per warp once the grid is full.
  int64_t rpw = (n + warps_target - 1) / warps_target;
  if (rpw < 32) rpw = 32;
  const int64_t warps = (n + rpw - 1) / rpw;
  const int64_t blocks = (warps + 7) / 8;
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  if (vec)
    fingerprint_kernel<true><<<(unsigned)blocks, 256, 0, stream>>>(tokens, n, stride, lens, seed,
                                                                    fp_out, rpw, err);
  else
    fingerprint_kernel<false><<<(unsigned)blocks, 256, 0, stream>>>(tokens, n, stride, lens,
                                                                     seed, fp_out, rpw, err);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "fingerprint launch");
}

}  // namespace hs
