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



// ---- vector path: per-lane bulk copies (TMA) --------------------------------------
// A warp owns 32 rows at a time, one per lane.  In each round every lane
// stages the next chunk of up to kChunk tokens of its own row with one bulk
// copy (cp.async.bulk: a contiguous, 16-byte aligned range of the row) into
// its own slot of the warp's round buffer; the 32 copies of a round complete
// on one mbarrier.  While a round's copies are in flight the lanes hash the
// previous round's chunks (two buffers).  Each lane reads only its own slot,
// so lanes never wait for each other except through the mbarrier.  A lane
// whose row is exhausted claims the warp's next row for the next round
// (lengths prefetched 64 rows ahead, handed out by shuffle).
//
// The hash loop is uniform across lanes: a fixed walk over the chunk's
// 16-byte pieces with tokens past the chunk's end masked per word, so a lane
// at the end of its row does not send the warp down a second path.  Slots
// are 144 bytes (9 x 16 B) so the eight lanes of a quarter-warp hit
// different banks.
// Per-warp shared memory for chunks of C tokens: NB round buffers of 32
// slots (C*4 + 16 bytes each, an odd multiple of 16 for C = 32, 64 or 128),
// then NB mbarriers and an abort word.
template <int C>
constexpr int slot_bytes() { return C * 4 + 16; }
template <int C>
constexpr int round_bytes() { return 32 * slot_bytes<C>(); }
template <int C, int NB>
constexpr int warp_bytes() { return NB * round_bytes<C>() + 8 * NB + 16; }

__device__ __forceinline__ void bulk_copy_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                              uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// Hash tokens [0, w) of a chunk in shared memory (w <= C).  Every lane
// walks the same pieces; words at or past w are masked out of the fast-path
// test and skipped.
template <int C>
__device__ __forceinline__ void hash_chunk(uint32_t& lo, uint32_t& hi, const int4* blk, int w) {
#pragma unroll 2
  for (int pc = 0; pc < C / 4; ++pc) {
    const int n = w - 4 * pc;                     // valid words in this piece (may be <= 0)
    if (__all_sync(0xffffffffu, n <= 0)) break;
    const int4 v = blk[pc];
    const uint32_t x = n > 0 ? (uint32_t)v.x : 0u;
    const uint32_t y = n > 1 ? (uint32_t)v.y : 0u;
    const uint32_t z = n > 2 ? (uint32_t)v.z : 0u;
    const uint32_t q = n > 3 ? (uint32_t)v.w : 0u;
    if (((x | y | z | q) >> 16) == 0u) {
      if (n > 0) hash_word_small(lo, hi, x);
      if (n > 1) hash_word_small(lo, hi, y);
      if (n > 2) hash_word_small(lo, hi, z);
      if (n > 3) hash_word_small(lo, hi, q);
    } else {
      if (n > 0) hash_word(lo, hi, x);
      if (n > 1) hash_word(lo, hi, y);
      if (n > 2) hash_word(lo, hi, z);
      if (n > 3) hash_word(lo, hi, q);
    }
  }
}

template <int WARPS, int kChunk, int NB>
__global__ void __launch_bounds__(WARPS * 32) fingerprint_tma_kernel(
    const int32_t* __restrict__ tokens, int64_t n, int32_t stride,
    const int32_t* __restrict__ lens, uint64_t seed, uint64_t* __restrict__ fp_out,
    int64_t rows_per_warp, unsigned* err) {
  extern __shared__ __align__(16) uint8_t tma_smem[];
  constexpr int kSlotBytes = slot_bytes<kChunk>();
  constexpr int kRoundBytes = round_bytes<kChunk>();
  constexpr int kWarpBytes = warp_bytes<kChunk, NB>();
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t r_begin = warp * rows_per_warp;
  if (r_begin >= n) return;
  const int64_t r_end = min(n, r_begin + rows_per_warp);
  const uint32_t lane = threadIdx.x & 31u;
  uint8_t* wbuf = tma_smem + (threadIdx.x >> 5) * kWarpBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(wbuf + NB * kRoundBytes);
  volatile int* abort_word = reinterpret_cast<volatile int*>(bars + NB);
  const uint32_t wbuf_u32 = smem_u32(wbuf);
  const uint32_t seed_lo = (uint32_t)seed, seed_hi = (uint32_t)(seed >> 32);
  if (lane == 0) {
    for (int b = 0; b < NB; ++b) mbar_init(bars + b, 32);
    *abort_word = 0;
    fence_mbar_init();
  }
  __syncwarp();

  // Issue side: the next chunk of this lane's row to stage.
  int64_t irow = -1;
  int32_t ipos = 0, ilen = 0;
  // Staged chunk per buffer: row (or -1), start position, tokens, row length.
  int64_t prow[NB];
  int32_t ppos[NB], pw[NB], plen[NB];
  uint32_t phase[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    prow[b] = -1;
    ppos[b] = pw[b] = plen[b] = 0;
    phase[b] = 0u;
  }
  uint32_t lo = seed_lo, hi = seed_hi;

  int64_t next = r_begin;
  int64_t wbase = r_begin;
  auto len_of = [&](int64_t r) -> int32_t {
    return r < r_end ? (lens ? __ldg(lens + r) : stride) : 0;
  };
  int32_t len_a = len_of(wbase + lane), len_b = len_of(wbase + 32 + lane);

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

  // Stage this lane's next chunk into its slot of buffer b (one bulk copy).
  auto issue = [&](int b) {
    const int32_t w = irow >= 0 ? min(kChunk, ilen - ipos) : 0;
    const uint32_t bytes = (uint32_t)((w + 3) >> 2) * 16u;
    prow[b] = irow;
    ppos[b] = ipos;
    pw[b] = w;
    plen[b] = ilen;
    mbar_arrive_expect_tx(bars + b, bytes);
    if (bytes) {
      bulk_copy_g2s(wbuf_u32 + b * kRoundBytes + lane * kSlotBytes,
                    tokens + irow * (int64_t)stride + ipos, bytes, smem_u32(bars + b));
      ipos += w;
      if (ipos >= ilen) irow = -1;
    }
  };

  auto hash = [&](int b) -> bool {
    if (!mbar_wait(bars + b, phase[b], abort_word)) return false;
    phase[b] ^= 1u;
    if (prow[b] >= 0 && ppos[b] == 0) {
      lo = seed_lo;
      hi = seed_hi;
    }
    hash_chunk<kChunk>(lo, hi,
                       reinterpret_cast<const int4*>(wbuf + b * kRoundBytes + lane * kSlotBytes),
                       prow[b] >= 0 ? pw[b] : 0);
    if (prow[b] >= 0 && ppos[b] + pw[b] >= plen[b]) fp_out[prow[b]] = ((uint64_t)hi << 32) | lo;
    prow[b] = -1;
    return true;
  };

  // Rounds 0 .. NB-2 in flight before the first hash; then each step stages
  // round r + NB - 1 and hashes round r.
#pragma unroll
  for (int b = 0; b < NB - 1; ++b) {
    claim();
    issue(b);
  }
  for (;;) {
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      claim();
      issue((b + NB - 1) % NB);
      if (!hash(b)) {
        set_error(err, kErrTimeout);
        return;
      }
    }
    bool pending = irow >= 0;
#pragma unroll
    for (int b = 0; b < NB; ++b) pending |= prow[b] >= 0;
    if (!__any_sync(0xffffffffu, pending) && next >= r_end) break;
  }
  // The last NB-1 issue() calls (buffers 0 .. NB-2) staged nothing: every
  // lane was idle.  Their barrier phases complete on the 32 arrivals alone;
  // wait for them so the warp leaves no phase open.
#pragma unroll
  for (int b = 0; b < NB - 1; ++b)
    if (!mbar_wait(bars + b, phase[b], abort_word)) set_error(err, kErrTimeout);
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
    // Per-lane bulk copies: 8-warp blocks with 32-token chunks (74 KB of
    // round buffers, three blocks = 24 warps per SM) once there are rows for
    // all of them; else one-warp blocks with 128-token chunks, so the warps
    // spread over all SMs and each lane has few, large rounds.
    const int64_t lanes_full = sms * 12 * 32;
    if (n >= lanes_full) {
      // 32-token chunks, four buffers (three rounds in flight), 4-warp
      // blocks of 73.9 KB: three blocks = 12 warps per SM.
      const int64_t warps_target = sms * 12;
      const int64_t rpw = (n + warps_target - 1) / warps_target;
      const int64_t warps = (n + rpw - 1) / rpw;
      const int64_t blocks = (warps + 3) / 4;
      const size_t smem = 4 * (size_t)warp_bytes<32, 4>();
      static bool configured = false;
      if (!configured) {
        const cudaError_t e = cudaFuncSetAttribute(fingerprint_tma_kernel<4, 32, 4>,
                                                   cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   (int)smem);
        if (e != cudaSuccess) return cuda_fail(e, "fingerprint smem attribute");
        configured = true;
      }
      fingerprint_tma_kernel<4, 32, 4><<<(unsigned)blocks, 128, smem, stream>>>(
          tokens, n, stride, lens, seed, fp_out, rpw, err);
    } else {
      // Few rows: one-warp blocks, 64-token chunks, four buffers (34 KB).
      const int64_t warps = (n + 31) / 32;
      fingerprint_tma_kernel<1, 64, 4><<<(unsigned)warps, 32, warp_bytes<64, 4>(), stream>>>(
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
