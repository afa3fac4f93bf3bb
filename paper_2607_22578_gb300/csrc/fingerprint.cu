// K1: per-row 64-bit FNV-1a fingerprints over int32 token rows — the D_in
// part of the node semantic signature Sig(v) (Section 3.3, Eq. 2).
//
// FNV-1a is a serial chain over the octets of one row, so parallelism comes
// from rows: each lane of a warp owns one row at a time.  Rows are split into
// full chunks of 32 tokens, hashed in registers by the chunk kernel with a
// straight-line, predicate-free loop, and a tail of L mod 32 tokens, finished
// by a one-thread-per-row tail kernel from the partial state.
// The octet rounds themselves are in fnv.cuh.
#include "fnv.cuh"
#include "hs_internal.cuh"

namespace hs {
namespace {

using namespace fnv;

// ---- vector path: full chunks in registers, tails in a second kernel -------------
// A warp owns 32 rows at a time, one per lane.  The chunk kernel hashes only
// FULL chunks of T = 32 tokens: tokens [0, floor(L/T)*T) of every row with
// L >= T.  Each lane loads its next chunk with 16- or 32-byte vector loads
// straight into registers one chunk ahead of the chunk it hashes (NB register
// buffers), so every lane runs the same straight-line hash over T tokens: no
// per-token predicates and no masking.  After its last full chunk a row's
// state goes to fp_out: the final fingerprint when T divides L, otherwise the
// partial state, which the tail kernel finishes with the last L mod T tokens
// (one thread per row, so the few short tails run with the whole GPU's
// parallelism instead of serially at the end of each warp).  Rows shorter
// than T and rows with an invalid length are left entirely to the tail
// kernel.  A lane that has issued its row's last chunk claims the next
// unclaimed row of its warp's range (lengths prefetched 64 rows ahead and
// handed out by shuffle).
//
// A chunk whose tokens are all below 65536 (in every live lane) takes the
// two-round small-token hash; otherwise the whole chunk takes the octet-wise
// rounds, which are exact for every token.

template <int VB>
__device__ __forceinline__ void load_vec(const int32_t* p, uint32_t* x) {
  if constexpr (VB == 32) {
    asm volatile("ld.global.nc.L1::no_allocate.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=r"(x[0]), "=r"(x[1]), "=r"(x[2]), "=r"(x[3]), "=r"(x[4]), "=r"(x[5]),
                   "=r"(x[6]), "=r"(x[7])
                 : "l"(p));
  } else {
    asm volatile("ld.global.nc.L1::no_allocate.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(x[0]), "=r"(x[1]), "=r"(x[2]), "=r"(x[3])
                 : "l"(p));
  }
}

constexpr int kTailChunk = 32;  // T: tokens per full chunk

template <int VB, int K, int NB>
__global__ void __launch_bounds__(256) fingerprint_chunks_kernel(
    const int32_t* __restrict__ tokens, int64_t n, int32_t stride,
    const int32_t* __restrict__ lens, uint64_t seed, uint64_t* __restrict__ fp_out,
    int64_t rows_per_warp) {
  pdl_wait();
  pdl_trigger();
  constexpr int W = VB / 4;  // tokens per vector load
  constexpr int T = W * K;   // tokens per chunk
  static_assert(T == kTailChunk, "chunk size shared with the tail kernel");
  const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t r_begin = warp * rows_per_warp;
  if (r_begin >= n) return;
  const int64_t r_end = min(n, r_begin + rows_per_warp);
  const uint32_t lane = threadIdx.x & 31u;
  const uint32_t seed_lo = (uint32_t)seed, seed_hi = (uint32_t)(seed >> 32);

  // Issue side: the row being loaded, the next chunk's start, the end of its
  // full chunks.
  int64_t irow = -1;
  int32_t ipos = 0, iend = 0;
  uint32_t buf[NB][T];
  int64_t brow[NB];
  bool bfirst[NB], blast[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    brow[b] = -1;
    bfirst[b] = blast[b] = false;
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
        const int32_t L = off < 32 ? La : Lb;
        if (L >= T && L <= stride) {
          irow = next + rank;
          ipos = 0;
          iend = (L / T) * T;
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

  // Load this lane's next full chunk into buffer b.
  auto issue = [&](int b) {
    brow[b] = irow;
    if (irow >= 0) {
      const int32_t* src = tokens + irow * (int64_t)stride + ipos;
#pragma unroll
      for (int j = 0; j < K; ++j) load_vec<VB>(src + j * W, &buf[b][j * W]);
      bfirst[b] = ipos == 0;
      ipos += T;
      blast[b] = ipos == iend;
      if (blast[b]) irow = -1;
    }
  };

  // Hash buffer b (every lane, live or not: an idle lane's result is dropped).
  auto consume = [&](int b) {
    const bool live = brow[b] >= 0;
    lo = (live && bfirst[b]) ? seed_lo : lo;
    hi = (live && bfirst[b]) ? seed_hi : hi;
    uint32_t any = 0;
#pragma unroll
    for (int t = 0; t < T; ++t) any |= buf[b][t];
    if (__all_sync(0xffffffffu, !live || (any >> 16) == 0u)) {
#pragma unroll
      for (int t = 0; t < T; ++t) hash_word_small(lo, hi, buf[b][t]);
    } else {
#pragma unroll
      for (int t = 0; t < T; ++t) hash_word_full(lo, hi, buf[b][t]);
    }
    if (live && blast[b]) fp_out[brow[b]] = ((uint64_t)hi << 32) | lo;
    brow[b] = -1;
  };

  // Chunks 0 .. NB-2 in flight before the first hash; then each step loads
  // chunk c + NB - 1 and hashes chunk c.
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
      consume(b);
    }
    bool pending = irow >= 0;
#pragma unroll
    for (int b = 0; b < NB; ++b) pending |= brow[b] >= 0;
    if (!__any_sync(0xffffffffu, pending) && next >= r_end) break;
  }
}

// The last L mod T tokens of every row (the whole row when L < T), one thread
// per row, continuing from the partial state the chunk kernel left in fp_out.
// Also the row-length checks: an invalid length sets the error flag and a
// zero fingerprint; an empty row gets the seed.  Needs 16-byte aligned rows.
__global__ void __launch_bounds__(256) fingerprint_tails_kernel(
    const int32_t* __restrict__ tokens, int64_t n, int32_t stride,
    const int32_t* __restrict__ lens, uint64_t seed, uint64_t* __restrict__ fp_out,
    unsigned* err) {
  pdl_wait();
  pdl_trigger();
  constexpr int T = kTailChunk;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n;
       r += (int64_t)gridDim.x * blockDim.x) {
    const int32_t L = lens ? __ldg(lens + r) : stride;
    if (L < 0 || L > stride) {
      set_error(err, kErrInvalidArg);
      fp_out[r] = 0ull;
      continue;
    }
    const int32_t m = L % T;
    if (m == 0 && L > 0) continue;  // the chunk kernel wrote the final value
    uint32_t lo = (uint32_t)seed, hi = (uint32_t)(seed >> 32);
    if (L >= T) {
      const uint64_t st = fp_out[r];
      lo = (uint32_t)st;
      hi = (uint32_t)(st >> 32);
    }
    const int32_t* src = tokens + r * (int64_t)stride + (L - m);
    uint4 v[T / 4];
#pragma unroll
    for (int q = 0; q < T / 4; ++q)
      if (4 * q < m) v[q] = __ldg(reinterpret_cast<const uint4*>(src + 4 * q));
#pragma unroll
    for (int q = 0; q < T / 4; ++q) {
      if (4 * q < m) hash_word(lo, hi, v[q].x);
      if (4 * q + 1 < m) hash_word(lo, hi, v[q].y);
      if (4 * q + 2 < m) hash_word(lo, hi, v[q].z);
      if (4 * q + 3 < m) hash_word(lo, hi, v[q].w);
    }
    fp_out[r] = ((uint64_t)hi << 32) | lo;
  }
}

// ---- word path (tokens not 16-byte aligned, or row_stride % 4 != 0) -------------------
__global__ void __launch_bounds__(256) fingerprint_words_kernel(
    const int32_t* __restrict__ tokens, int64_t n, int32_t stride,
    const int32_t* __restrict__ lens, uint64_t seed, uint64_t* __restrict__ fp_out,
    int64_t rows_per_warp, unsigned* err) {
  pdl_wait();
  pdl_trigger();
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


template <int VB, int K, int NB>
hs_status launch_chunks(const int32_t* tokens, int64_t n, int32_t stride, const int32_t* lens,
                        uint64_t seed, uint64_t* fp_out, int64_t sms, cudaStream_t stream) {
  // Resident warps per SM at this kernel's register count (queried once per
  // device; the kernel uses no shared memory).
  static std::atomic<int> per_device[kMaxDeviceOrdinals];
  const int dev = device_ordinal();
  int warps_per_sm = dev >= 0 ? per_device[dev].load() : 0;
  if (warps_per_sm == 0) {
    int blocks = 0;
    const cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &blocks, fingerprint_chunks_kernel<VB, K, NB>, 256, 0);
    if (e != cudaSuccess) return cuda_fail(e, "fingerprint occupancy");
    warps_per_sm = blocks > 0 ? blocks * 8 : 8;
    if (dev >= 0) per_device[dev].store(warps_per_sm);
  }
  const int64_t warps_target = sms * warps_per_sm;
  int64_t rpw = (n + warps_target - 1) / warps_target;
  if (rpw < 32) rpw = 32;
  const int64_t warps = (n + rpw - 1) / rpw;
  // Few warps: one-warp blocks, so they spread over all SMs.
  const int threads = warps >= sms * 8 ? 256 : 32;
  const int64_t blocks = (warps * 32 + threads - 1) / threads;
  launch_pdl(fingerprint_chunks_kernel<VB, K, NB>, dim3((unsigned)blocks), dim3(threads), 0, stream,
             tokens, n, stride, lens, seed, fp_out, rpw);
  count_launches(1);
  return HS_OK;
}

}  // namespace

// The full 32-token chunks only (the first pass of hs_merge_rows, whose
// second pass finishes the tails): 16-byte aligned rows with stride % 4 == 0.
// Sets *ran = false when no row can have a full chunk (stride < 32).
hs_status launch_fingerprint_chunks(const int32_t* tokens, int64_t n, int32_t stride,
                                    const int32_t* lens, uint64_t seed, uint64_t* fp_out,
                                    bool* ran, cudaStream_t stream) {
  *ran = false;
  if (stride < kTailChunk) return HS_OK;
  const bool vec32 = (reinterpret_cast<uintptr_t>(tokens) & 31u) == 0 && stride % 8 == 0;
  const int64_t sms = num_sms();
  const hs_status st =
      vec32 ? launch_chunks<32, 4, 2>(tokens, n, stride, lens, seed, fp_out, sms, stream)
            : launch_chunks<16, 8, 2>(tokens, n, stride, lens, seed, fp_out, sms, stream);
  if (st == HS_OK) *ran = true;
  return st;
}

hs_status launch_fingerprint(const int32_t* tokens, int64_t n, int32_t stride,
                             const int32_t* lens, uint64_t seed, uint64_t* fp_out,
                             cudaStream_t stream) {
  const uintptr_t base = reinterpret_cast<uintptr_t>(tokens);
  const bool vec32 = (base & 31u) == 0 && stride % 8 == 0;
  const bool vec16 = (base & 15u) == 0 && stride % 4 == 0;
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const int64_t sms = num_sms();
  if (vec16) {
    if (stride >= kTailChunk) {
      const hs_status st =
          vec32 ? launch_chunks<32, 4, 2>(tokens, n, stride, lens, seed, fp_out, sms, stream)
                : launch_chunks<16, 8, 2>(tokens, n, stride, lens, seed, fp_out, sms, stream);
      if (st != HS_OK) return st;
    }
    if (lens || stride % kTailChunk != 0 || stride == 0) {
      int64_t blocks = (n + 255) / 256;
      if (blocks > sms * 64) blocks = sms * 64;
      launch_pdl(fingerprint_tails_kernel, dim3((unsigned)blocks), dim3(256), 0, stream, tokens, n,
                 stride, lens, seed, fp_out, err);
      count_launches(1);
    }
  } else {
    const int64_t warps_target = sms * 32;
    int64_t rpw = (n + warps_target - 1) / warps_target;
    if (rpw < 32) rpw = 32;
    const int64_t warps = (n + rpw - 1) / rpw;
    const int64_t blocks = (warps + 7) / 8;
    launch_pdl(fingerprint_words_kernel, dim3((unsigned)blocks), dim3(256), 0, stream, tokens, n,
               stride, lens, seed, fp_out, rpw, err);
    count_launches(1);
  }
  return cuda_fail(cudaGetLastError(), "fingerprint launch");
}

}  // namespace hs
