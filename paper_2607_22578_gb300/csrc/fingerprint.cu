// K1: per-row 64-bit FNV-1a fingerprints over int32 token rows — the D_in
// part of the node semantic signature Sig(v) (Section 3.3, Eq. 2).
//
// FNV-1a is a serial chain over the octets of one row, so parallelism comes
// from rows: each lane of a warp owns one row at a time and streams it through
// a private shared-memory ring filled by cp.async several blocks ahead.  Rows
// have different lengths; a lane that has issued its whole row claims the next
// unclaimed row of its warp's range (warp-synchronous ballot, no atomics), so
// the lanes of a warp stay busy until the range is drained.
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
  // (hi * 2^32 + lo) * (2^40 + 0x1b3) mod 2^64: the low word needs only lo,
  // the high word adds hi * 0x1b3, the carry-out of lo * 0x1b3 and lo << 8.
  hi = __umulhi(lo, 0x1b3u) + hi * 0x1b3u + (lo << 8);
  lo = lo * 0x1b3u;
}

__device__ __forceinline__ void mul_prime3(uint32_t& lo, uint32_t& hi) {
  hi = __umulhi(lo, kP3Lo) + lo * kP3Hi + hi * kP3Lo;
  lo = lo * kP3Lo;
}

// Octet-wise rounds for one token, little-endian octet order; octets are
// extracted with byte permutes, no branches.
__device__ __forceinline__ void hash_word_full(uint32_t& lo, uint32_t& hi, uint32_t w) {
  lo ^= __byte_perm(w, 0u, 0x4440u);
  mul_prime(lo, hi);
  lo ^= __byte_perm(w, 0u, 0x4441u);
  mul_prime(lo, hi);
  lo ^= __byte_perm(w, 0u, 0x4442u);
  mul_prime(lo, hi);
  lo ^= w >> 24;
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



// ---- vector path: per-lane cp.async pipeline ----------------------------------------
// A lane owns one row at a time.  Its row is cut into blocks of 16 tokens
// (four 16-byte pieces); the lane keeps kDepth blocks in a private ring in
// shared memory, filled by cp.async (16-byte, L2-only) kDepth-1 blocks ahead
// of the block it hashes.  The issue side claims the next row as soon as the
// current one is fully issued, so a row boundary costs no exposed latency.
// In-flight data lives in shared memory, not registers.  Many rows: a 3-slot
// ring and 128-thread blocks, eight blocks (32 warps) per SM.  Few rows (too
// few to fill the SMs that way): an 8-slot ring and one-warp blocks, so each
// lane keeps seven blocks in flight and the warps spread over all SMs.  The
// ring is padded to an odd multiple of 16 bytes per lane so the eight lanes
// of a quarter-warp read different banks.
constexpr int kBlockWords = 16;
template <int D>
constexpr int lane_bytes() { return D * kBlockWords * 4 + 16; }  // odd multiple of 16 B

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ uint32_t word_of(const int4& v, int j) {
  return (uint32_t)(j == 0 ? v.x : (j == 1 ? v.y : (j == 2 ? v.z : v.w)));
}

// Hash the first w tokens of a block held in shared memory.  One compact
// body: the four-token fast path when all four tokens are below 65536, else
// token by token.
__device__ __forceinline__ void hash_block(uint32_t& lo, uint32_t& hi, const int4* blk, int w) {
#pragma unroll 1
  for (int pc = 0; 4 * pc < w; ++pc) {
    const int4 v = blk[pc];
    const int nw = min(4, w - 4 * pc);
    if (nw == 4) {
      if ((((uint32_t)v.x | (uint32_t)v.y | (uint32_t)v.z | (uint32_t)v.w) >> 16) == 0u) {
        hash_word_small(lo, hi, (uint32_t)v.x);
        hash_word_small(lo, hi, (uint32_t)v.y);
        hash_word_small(lo, hi, (uint32_t)v.z);
        hash_word_small(lo, hi, (uint32_t)v.w);
      } else {
        hash_word_full(lo, hi, (uint32_t)v.x);
        hash_word_full(lo, hi, (uint32_t)v.y);
        hash_word_full(lo, hi, (uint32_t)v.z);
        hash_word_full(lo, hi, (uint32_t)v.w);
      }
    } else {
#pragma unroll 1
      for (int j = 0; j < nw; ++j) hash_word(lo, hi, word_of(v, j));
    }
  }
}

template <int kDepth, int kFpThreads>
__global__ void __launch_bounds__(kFpThreads) fingerprint_async_kernel(
    const int32_t* __restrict__ tokens, int64_t n, int32_t stride,
    const int32_t* __restrict__ lens, uint64_t seed, uint64_t* __restrict__ fp_out,
    int64_t rows_per_warp, unsigned* err) {
  extern __shared__ uint8_t ring_all[];
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t r_begin = warp * rows_per_warp;
  if (r_begin >= n) return;
  const int64_t r_end = min(n, r_begin + rows_per_warp);
  constexpr int kLaneBytes = lane_bytes<kDepth>();
  const uint32_t ring = smem_u32(ring_all + threadIdx.x * kLaneBytes);
  const uint8_t* ring_p = ring_all + threadIdx.x * kLaneBytes;
  const uint32_t seed_lo = (uint32_t)seed, seed_hi = (uint32_t)(seed >> 32);

  // Issue side.
  int64_t irow = -1;
  int32_t ipos = 0, ilen = 0;
  const int32_t* isrc = tokens;
  // Per-slot metadata: row (or -1) and info = words | first << 8 | last << 9.
  int64_t m_row[kDepth];
  int32_t m_info[kDepth];
#pragma unroll
  for (int s = 0; s < kDepth; ++s) {
    m_row[s] = -1;
    m_info[s] = 0;
  }
  // Hash side.
  uint32_t lo = seed_lo, hi = seed_hi;
  int64_t next = r_begin;
  // Row lengths of the next 64 rows of the warp's range, prefetched: lane j
  // holds rows wbase+j (len_a) and wbase+32+j (len_b); claims read them by
  // shuffle, so claiming a row never waits on memory.
  const uint32_t lane = threadIdx.x & 31u;
  int64_t wbase = r_begin;
  auto len_of = [&](int64_t r) -> int32_t {
    return r < r_end ? (lens ? __ldg(lens + r) : stride) : 0;
  };
  int32_t len_a = len_of(wbase + lane), len_b = len_of(wbase + 32 + lane);

  for (;;) {
#pragma unroll
    for (int si = 0; si < kDepth; ++si) {
      // ---- claim rows for lanes whose issue side is free, in lane order
      unsigned need = __ballot_sync(0xffffffffu, irow < 0);
      while (need != 0u && next < r_end) {
        const int64_t avail = r_end - next;
        const int rank = __popc(need & lanemask_lt());
        const int off = (int)(next - wbase) + (irow < 0 ? rank : 0);  // 0..62
        const int32_t La = __shfl_sync(0xffffffffu, len_a, off & 31);
        const int32_t Lb = __shfl_sync(0xffffffffu, len_b, off & 31);
        if (irow < 0 && rank < avail) {
          const int64_t r = next + rank;
          const int32_t L = off < 32 ? La : Lb;
          if (L < 0 || L > stride) {
            set_error(err, kErrInvalidArg);
            fp_out[r] = 0ull;
          } else if (L == 0) {
            fp_out[r] = seed;
          } else {
            irow = r;
            ipos = 0;
            ilen = L;
            isrc = tokens + r * (int64_t)stride;
          }
        }
        next += min((int64_t)__popc(need), avail);
        if (next - wbase >= 32) {        // slide the length window by 32 rows
          wbase += 32;
          len_a = len_b;
          len_b = len_of(wbase + 32 + lane);
        }
        need = __ballot_sync(0xffffffffu, irow < 0);
      }
      // ---- issue one block into slot si
      if (irow >= 0) {
        const int32_t words = min(kBlockWords, ilen - ipos);
        const uint32_t dst = ring + si * kBlockWords * 4;
#pragma unroll
        for (int pc = 0; pc < kBlockWords / 4; ++pc)
          if (4 * pc < words) cp_async16(dst + 16 * pc, isrc + ipos + 4 * pc);
        m_row[si] = irow;
        const bool first = ipos == 0;
        ipos += words;
        const bool last = ipos >= ilen;
        m_info[si] = words | (first ? 256 : 0) | (last ? 512 : 0);
        if (last) irow = -1;
      } else {
        m_row[si] = -1;
      }
      cp_async_commit();
      // ---- hash the oldest slot (issued kDepth-1 rounds ago)
      const int sc = (si + 1) % kDepth;
      cp_async_wait<kDepth - 1>();
      if (m_row[sc] >= 0) {
        const int32_t info = m_info[sc];
        if (info & 256) {
          lo = seed_lo;
          hi = seed_hi;
        }
        hash_block(lo, hi, reinterpret_cast<const int4*>(ring_p + sc * kBlockWords * 4),
                   info & 255);
        if (info & 512) fp_out[m_row[sc]] = ((uint64_t)hi << 32) | lo;
        m_row[sc] = -1;
      }
    }
    bool pending = irow >= 0;
#pragma unroll
    for (int s = 0; s < kDepth; ++s) pending |= m_row[s] >= 0;
    if (!__any_sync(0xffffffffu, pending) && next >= r_end) break;
  }
  cp_async_wait<0>();
}

// ---- vector path, coalesced staging -----------------------------------------------
// A warp owns 32 rows at a time, one per lane.  In each round it stages the
// next chunk of up to 64 tokens of all 32 rows in shared memory: every copy
// instruction moves two rows' contiguous 256-byte chunks (16 lanes per row),
// so an instruction touches a handful of cache lines instead of 32 rows'
// worth.  Each lane then hashes its own row's chunk from shared memory while
// the next round's chunks are in flight (two buffers per warp).  A lane whose
// row is exhausted claims the warp's next row for the following round.  Row
// slots are 272 bytes (17 x 16 B) so the eight lanes of a quarter-warp read
// different banks.
constexpr int kChunk = 64;                       // tokens per row per round
constexpr int kSlotBytes = kChunk * 4 + 16;      // 272 B
constexpr int kRoundBytes = 32 * kSlotBytes;     // one buffer of one warp

template <int WARPS>
__global__ void __launch_bounds__(WARPS * 32) fingerprint_coal_kernel(
    const int32_t* __restrict__ tokens, int64_t n, int32_t stride,
    const int32_t* __restrict__ lens, uint64_t seed, uint64_t* __restrict__ fp_out,
    int64_t rows_per_warp, unsigned* err) {
  extern __shared__ uint8_t coal_smem[];
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t r_begin = warp * rows_per_warp;
  if (r_begin >= n) return;
  const int64_t r_end = min(n, r_begin + rows_per_warp);
  const uint32_t lane = threadIdx.x & 31u;
  uint8_t* wbuf = coal_smem + (threadIdx.x >> 5) * 2 * kRoundBytes;
  const uint32_t wbuf_u32 = smem_u32(wbuf);
  const uint32_t seed_lo = (uint32_t)seed, seed_hi = (uint32_t)(seed >> 32);

  // Issue side: the next chunk of this lane's row to stage.
  int64_t irow = -1;
  int32_t ipos = 0, ilen = 0;
  // Staged chunks per buffer: row (or -1), start position, tokens, row length.
  int64_t prow[2] = {-1, -1};
  int32_t ppos[2] = {0, 0}, pw[2] = {0, 0}, plen[2] = {0, 0};
  uint32_t lo = seed_lo, hi = seed_hi;

  int64_t next = r_begin;
  int64_t wbase = r_begin;
  auto len_of = [&](int64_t r) -> int32_t {
    return r < r_end ? (lens ? __ldg(lens + r) : stride) : 0;
  };
  int32_t len_a = len_of(wbase + lane), len_b = len_of(wbase + 32 + lane);

  // Claim rows for lanes whose issue side is free (lengths prefetched).
  auto claim = [&]() {
    unsigned need = __ballot_sync(0xffffffffu, irow < 0);
    while (need != 0u && next < r_end) {
      const int64_t avail = r_end - next;
      const int rank = __popc(need & lanemask_lt());
      const int off = (int)(next - wbase) + (irow < 0 ? rank : 0);
      const int32_t La = __shfl_sync(0xffffffffu, len_a, off & 31);
      const int32_t Lb = __shfl_sync(0xffffffffu, len_b, off & 31);
      if (irow < 0 && rank < avail) {
        const int64_t r = next + rank;
        const int32_t L = off < 32 ? La : Lb;
        if (L < 0 || L > stride) {
          set_error(err, kErrInvalidArg);
          fp_out[r] = 0ull;
        } else if (L == 0) {
          fp_out[r] = seed;
        } else {
          irow = r;
          ipos = 0;
          ilen = L;
        }
      }
      next += min((int64_t)__popc(need), avail);
      if (next - wbase >= 32) {
        wbase += 32;
        len_a = len_b;
        len_b = len_of(wbase + 32 + lane);
      }
      need = __ballot_sync(0xffffffffu, irow < 0);
    }
  };

  // Stage every lane's next chunk into buffer b, cooperatively.
  auto issue = [&](int b) {
    const int32_t w = irow >= 0 ? min(kChunk, ilen - ipos) : 0;
    const int32_t pieces = (w + 3) >> 2;
    const int32_t* src = tokens + (irow >= 0 ? irow * (int64_t)stride + ipos : 0);
    prow[b] = irow;
    ppos[b] = ipos;
    pw[b] = w;
    plen[b] = ilen;
    if (irow >= 0) {
      ipos += w;
      if (ipos >= ilen) irow = -1;
    }
    const uint32_t dst0 = wbuf_u32 + b * kRoundBytes;
    const uint32_t pc = lane & 15u;
#pragma unroll 4
    for (int i = 0; i < 16; ++i) {
      const int j = 2 * i + (int)(lane >> 4);
      const int32_t* sj = reinterpret_cast<const int32_t*>(
          __shfl_sync(0xffffffffu, reinterpret_cast<uintptr_t>(src), j));
      const int32_t pj = __shfl_sync(0xffffffffu, pieces, j);
      if ((int32_t)pc < pj) cp_async16(dst0 + j * kSlotBytes + 16 * pc, sj + 4 * pc);
    }
    cp_async_commit();
  };

  // Hash this lane's staged chunk in buffer b.
  auto hash = [&](int b) {
    if (prow[b] < 0) return;
    if (ppos[b] == 0) {
      lo = seed_lo;
      hi = seed_hi;
    }
    const int4* blk = reinterpret_cast<const int4*>(wbuf + b * kRoundBytes + lane * kSlotBytes);
    bool done = false;
    if (pw[b] == kChunk) {
      // Whole chunk: check once that every token is below 65536, then run
      // the two-round form straight through.
      uint32_t any_big = 0;
#pragma unroll 4
      for (int pc = 0; pc < kChunk / 4; ++pc) {
        const int4 v = blk[pc];
        any_big |= (uint32_t)v.x | (uint32_t)v.y | (uint32_t)v.z | (uint32_t)v.w;
      }
      if ((any_big >> 16) == 0u) {
#pragma unroll 4
        for (int pc = 0; pc < kChunk / 4; ++pc) {
          const int4 v = blk[pc];
          hash_word_small(lo, hi, (uint32_t)v.x);
          hash_word_small(lo, hi, (uint32_t)v.y);
          hash_word_small(lo, hi, (uint32_t)v.z);
          hash_word_small(lo, hi, (uint32_t)v.w);
        }
        done = true;
      }
    }
    if (!done) hash_block(lo, hi, blk, pw[b]);
    if (ppos[b] + pw[b] >= plen[b]) fp_out[prow[b]] = ((uint64_t)hi << 32) | lo;
    prow[b] = -1;
  };

  claim();
  issue(0);
  for (;;) {
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      claim();
      issue(b ^ 1);
      cp_async_wait<1>();
      __syncwarp();
      hash(b);
      __syncwarp();   // buffer b is reused by the next round's copies
    }
    const bool pending = irow >= 0 || prow[0] >= 0 || prow[1] >= 0;
    if (!__any_sync(0xffffffffu, pending) && next >= r_end) break;
  }
  cp_async_wait<0>();
}

// ---- word path (tokens not 16-byte aligned, or row_stride % 4 != 0) -------------------
__global__ void __launch_bounds__(256) fingerprint_words_kernel(
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
  int32_t len = 0, pos = 0;
  uint32_t lo = seed_lo, hi = seed_hi;
  const int32_t* src = tokens;
  int64_t next = r_begin;
  const uint32_t lane = threadIdx.x & 31u;
  int64_t wbase = r_begin;
  auto len_of = [&](int64_t r) -> int32_t {
    return r < r_end ? (lens ? __ldg(lens + r) : stride) : 0;
  };
  int32_t len_a = len_of(wbase + lane), len_b = len_of(wbase + 32 + lane);
  for (;;) {
    unsigned idle = __ballot_sync(0xffffffffu, !busy);
    while (idle != 0u && next < r_end) {
      const int64_t avail = r_end - next;
      const int rank = __popc(idle & lanemask_lt());
      const int off = (int)(next - wbase) + (!busy ? rank : 0);
      const int32_t La = __shfl_sync(0xffffffffu, len_a, off & 31);
      const int32_t Lb = __shfl_sync(0xffffffffu, len_b, off & 31);
      if (!busy && rank < avail) {
        const int64_t r = next + rank;
        const int32_t L = off < 32 ? La : Lb;
        if (L < 0 || L > stride) {
          set_error(err, kErrInvalidArg);
          fp_out[r] = 0ull;
        } else if (L == 0) {
          fp_out[r] = seed;
        } else {
          row = r;
          pos = 0;
          len = L;
          lo = seed_lo;
          hi = seed_hi;
          src = tokens + r * (int64_t)stride;
          busy = true;
        }
      }
      next += min((int64_t)__popc(idle), avail);
      if (next - wbase >= 32) {
        wbase += 32;
        len_a = len_b;
        len_b = len_of(wbase + 32 + lane);
      }
      idle = __ballot_sync(0xffffffffu, !busy);
    }
    if (!__any_sync(0xffffffffu, busy)) break;
    if (busy) {
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

}  // namespace

hs_status launch_fingerprint(const int32_t* tokens, int64_t n, int32_t stride,
                             const int32_t* lens, uint64_t seed, uint64_t* fp_out,
                             cudaStream_t stream) {
  const bool vec = ((reinterpret_cast<uintptr_t>(tokens) & 15u) == 0) && (stride % 4 == 0);
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const int64_t sms = num_sms();
  if (vec) {
    // Coalesced staging: 4-warp blocks (68 KB of round buffers, three
    // blocks per SM) once there are rows for 12 warps per SM, else one-warp
    // blocks so the warps spread over all SMs.
    const int64_t lanes_full = sms * 12 * 32;
    if (n >= lanes_full) {
      const int64_t warps_target = sms * 12;
      const int64_t rpw = (n + warps_target - 1) / warps_target;
      const int64_t warps = (n + rpw - 1) / rpw;
      const int64_t blocks = (warps + 3) / 4;
      const size_t smem = 4 * 2 * kRoundBytes;
      static bool configured = false;
      if (!configured) {
        const cudaError_t e = cudaFuncSetAttribute(
            fingerprint_coal_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return cuda_fail(e, "fingerprint smem attribute");
        configured = true;
      }
      fingerprint_coal_kernel<4><<<(unsigned)blocks, 128, smem, stream>>>(
          tokens, n, stride, lens, seed, fp_out, rpw, err);
    } else {
      const int64_t warps = (n + 31) / 32;
      fingerprint_coal_kernel<1><<<(unsigned)warps, 32, 2 * kRoundBytes, stream>>>(
          tokens, n, stride, lens, seed, fp_out, 32, err);
    }
  } else {
    const int64_t warps_target = sms * 32;
    int64_t rpw = (n + warps_target - 1) / warps_target;
    if (rpw < 32) rpw = 32;
    const int64_t warps = (n + rpw - 1) / rpw;
    const int64_t blocks = (warps + 7) / 8;
    fingerprint_words_kernel<<<(unsigned)blocks, 256, 0, stream>>>(tokens, n, stride, lens, seed,
                                                                   fp_out, rpw, err);
  }
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "fingerprint launch");
}

}  // namespace hs
