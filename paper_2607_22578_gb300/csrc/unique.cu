// K2-K4: exact unique-with-inverse over fingerprinted rows — the merge step of
// topological fusion within a time window (Section 3.3, "Dynamic Fusion and
// Reuse Mechanism" (I)) and the merge sets M(v*) of Appendix A.2.
//
// Pipeline (all on the caller's stream, no host synchronisation):
//   1. histogram of the four 8-bit digits of each fingerprint's upper 32
//      bits (one pass);
//   2. four stable LSD radix passes over (upper 32 fingerprint bits, row
//      index), each a single kernel with decoupled look-back across tiles
//      (bounded spins); stability keeps equal keys in ascending row order, so
//      each run of equal keys starts with its smallest row index;
//   3. segment heads: inclusive max-scan of "key differs from the previous
//      one" positions;
//   4. verify: every non-head row is compared in full (length + tokens) with
//      its segment head by one warp; equal rows take the head as their
//      representative, a mismatch marks the segment as collided.  A segment
//      holds rows whose fingerprints agree in the upper 32 bits; rows that
//      differ (in the lower bits, or in content under a true collision) are
//      never merged, they only send the segment through step 5;
//   5. collided segments only: exact regrouping by repeated peeling (the
//      first unassigned row becomes a representative, all rows equal to it
//      join it);
//   6. exclusive sum-scan of "row is its own representative" gives each
//      group its ordinal in first-occurrence order; the final kernel writes
//      unique_idx and inverse.
#include <mutex>

#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 16;
constexpr int kSortTile = kSortThreads * kSortItems;  // 4096 keys per tile
constexpr int kPasses = 4;   // digits of bits 32..63 of the fingerprint
constexpr int kLookBatch = 8;  // predecessor statuses read per round trip
constexpr uint32_t kFlagA = 1u << 30;  // tile aggregate published
constexpr uint32_t kFlagP = 2u << 30;  // inclusive prefix published
constexpr uint32_t kValMask = (1u << 30) - 1u;

constexpr int kScanThreads = 256;
constexpr int kScanItems = 16;
constexpr int kScanTile = kScanThreads * kScanItems;

constexpr size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct Layout {
  // zero-initialised region first
  size_t hist, status, ctr, coll_flag, coll_count, scan_status0, scan_status1, zero_end;
  size_t keys0, keys1, vals0, vals1, seg_head, rep, uid, coll_list, total;
};

constexpr Layout layout(int64_t n) {
  Layout L{};
  const int64_t sort_tiles = (n + kSortTile - 1) / kSortTile;
  const int64_t scan_tiles = (n + kScanTile - 1) / kScanTile;
  size_t o = 0;
  L.hist = o;          o += align256(sizeof(uint32_t) * kPasses * 256);
  L.status = o;        o += align256(sizeof(uint32_t) * kPasses * 256 * (size_t)sort_tiles);
  L.ctr = o;           o += align256(sizeof(uint32_t) * 16);
  L.coll_flag = o;     o += align256(sizeof(int32_t) * (size_t)n);
  L.coll_count = o;    o += align256(sizeof(uint32_t));
  L.scan_status0 = o;  o += align256(sizeof(uint64_t) * (size_t)scan_tiles);
  L.scan_status1 = o;  o += align256(sizeof(uint64_t) * (size_t)scan_tiles);
  L.zero_end = o;
  L.keys0 = o;         o += align256(sizeof(uint32_t) * (size_t)n);
  L.keys1 = o;         o += align256(sizeof(uint32_t) * (size_t)n);
  L.vals0 = o;         o += align256(sizeof(uint32_t) * (size_t)n);
  L.vals1 = o;         o += align256(sizeof(uint32_t) * (size_t)n);
  L.seg_head = o;      o += align256(sizeof(int32_t) * (size_t)n);
  L.rep = o;           o += align256(sizeof(int32_t) * (size_t)n);
  L.uid = o;           o += align256(sizeof(int32_t) * (size_t)n);
  L.coll_list = o;     o += align256(sizeof(int32_t) * (size_t)n);
  L.total = o;
  return L;
}

// Bounded spin on a 32-bit status word until its flag bits are non-zero.
__device__ __forceinline__ uint32_t wait_flag32(const volatile uint32_t* p, unsigned* err) {
  uint32_t s = *p;
  if (s & ~kValMask) return s;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    s = *p;
    if (s & ~kValMask) return s;
    if ((it & 31u) == 0) {
      __nanosleep(64);
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        set_error(err, kErrTimeout);
        return kFlagP;  // give up: treat as a zero prefix
      }
    }
  }
}

__device__ __forceinline__ uint64_t wait_flag64(const volatile unsigned long long* p,
                                                unsigned* err) {
  unsigned long long s = *p;
  if (s >> 32) return s;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    s = *p;
    if (s >> 32) return s;
    if ((it & 31u) == 0) {
      __nanosleep(64);
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        set_error(err, kErrTimeout);
        return 2ull << 32;
      }
    }
  }
}

// ---- 1. digit histograms ---------------------------------------------------------------
__global__ void __launch_bounds__(256) sort_hist_kernel(const uint64_t* __restrict__ fp, int64_t n,
                                                        uint32_t* __restrict__ hist) {
  __shared__ uint32_t h[kPasses * 256];
  for (int i = threadIdx.x; i < kPasses * 256; i += blockDim.x) h[i] = 0;
  __syncthreads();
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n;
       e += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t k = (uint32_t)(__ldg(fp + e) >> 32);
#pragma unroll
    for (int p = 0; p < kPasses; ++p) atomicAdd(&h[p * 256 + ((k >> (8 * p)) & 0xff)], 1u);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kPasses * 256; i += blockDim.x)
    if (h[i]) atomicAdd(&hist[i], h[i]);
}

// ---- 2. one stable radix pass ----------------------------------------------------------------
// Tile t holds keys [t*4096, (t+1)*4096); warp w of the tile owns the 512 keys
// [w*512, (w+1)*512), read striped (item i of lane l is key w*512 + i*32 + l),
// so processing items in order with lanes in order follows the input order.
// Pass 0 reads the caller's 64-bit fingerprints (fp_in) and implicit row
// indices; later passes read the previous pass's (key, value) arrays.
__global__ void __launch_bounds__(kSortThreads) onesweep_kernel(
    int pass, const uint64_t* __restrict__ fp_in, const uint32_t* __restrict__ keys_in,
    const uint32_t* __restrict__ vals_in, uint32_t* __restrict__ keys_out,
    uint32_t* __restrict__ vals_out, int64_t n,
    const uint32_t* __restrict__ hist, uint32_t* status, uint32_t* tile_ctr, unsigned* err) {
  __shared__ uint32_t s_tile;
  __shared__ uint32_t warp_cnt[kSortThreads / 32][256];
  __shared__ uint32_t digit_base[256];
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  if (tid == 0) s_tile = atomicAdd(tile_ctr + pass, 1u);
  for (int i = tid; i < (kSortThreads / 32) * 256; i += kSortThreads) (&warp_cnt[0][0])[i] = 0;
  // Exclusive scan of this pass's global digit counts (thread = digit).
  {
    const uint32_t c = hist[pass * 256 + tid];
    uint32_t x = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    __shared__ uint32_t wsum[8];
    if (lane == 31) wsum[w] = x;
    __syncthreads();
    uint32_t add = 0;
    for (int i = 0; i < w; ++i) add += wsum[i];
    digit_base[tid] = add + x - c;
  }
  __syncthreads();
  const uint32_t tile = s_tile;
  const int64_t base = (int64_t)tile * kSortTile + w * (kSortItems * 32);
  const int shift = 8 * pass;

  uint32_t k[kSortItems];
  uint32_t v[kSortItems];
  uint32_t rank[kSortItems];
#pragma unroll
  for (int i = 0; i < kSortItems; ++i) {
    const int64_t e = base + i * 32 + lane;
    if (e < n) {
      k[i] = fp_in ? (uint32_t)(fp_in[e] >> 32) : keys_in[e];
      v[i] = fp_in ? (uint32_t)e : vals_in[e];
    } else {
      k[i] = 0;
      v[i] = 0;
    }
  }
#pragma unroll
  for (int i = 0; i < kSortItems; ++i) {
    const int64_t e = base + i * 32 + lane;
    const bool valid = e < n;
    const uint32_t d = valid ? (uint32_t)((k[i] >> shift) & 0xff) : 256u + lane;
    const uint32_t peers = __match_any_sync(0xffffffffu, d);
    const uint32_t before = valid ? warp_cnt[w][d] : 0u;
    rank[i] = before + __popc(peers & lanemask_lt());
    __syncwarp();
    if (valid && (__ffs(peers) - 1) == lane) warp_cnt[w][d] = before + __popc(peers);
    __syncwarp();
  }
  __syncthreads();
  // Thread = digit: turn per-warp counts into per-warp exclusive offsets.
  uint32_t tile_count = 0;
#pragma unroll
  for (int ww = 0; ww < kSortThreads / 32; ++ww) {
    const uint32_t c = warp_cnt[ww][tid];
    warp_cnt[ww][tid] = tile_count;
    tile_count += c;
  }
  // Publish, look back, publish the inclusive prefix.
  volatile uint32_t* st = status + (size_t)pass * 256 * gridDim.x;
  uint32_t prefix = 0;
  if (tile == 0) {
    st[tid] = kFlagP | tile_count;
  } else {
    st[(size_t)tile * 256 + tid] = kFlagA | tile_count;
    // Walk back kLookBatch predecessors per round trip; stop at the first
    // inclusive prefix.
    bool done = false;
    for (int64_t j0 = (int64_t)tile - 1; j0 >= 0 && !done; j0 -= kLookBatch) {
      uint32_t sv[kLookBatch];
#pragma unroll
      for (int b = 0; b < kLookBatch; ++b) sv[b] = j0 - b >= 0 ? st[(size_t)(j0 - b) * 256 + tid] : (2u << 30);
#pragma unroll
      for (int b = 0; b < kLookBatch; ++b) {
        if (done) break;
        uint32_t sb = sv[b];
        if ((sb & ~kValMask) == 0) sb = wait_flag32(st + (size_t)(j0 - b) * 256 + tid, err);
        if (j0 - b >= 0) prefix += sb & kValMask;
        if ((sb & ~kValMask) == kFlagP) done = true;
      }
    }
    st[(size_t)tile * 256 + tid] = kFlagP | ((prefix + tile_count) & kValMask);
  }
  digit_base[tid] += prefix;
  __syncthreads();
#pragma unroll
  for (int i = 0; i < kSortItems; ++i) {
    const int64_t e = base + i * 32 + lane;
    if (e < n) {
      const uint32_t d = (uint32_t)((k[i] >> shift) & 0xff);
      const uint32_t pos = digit_base[d] + warp_cnt[w][d] + rank[i];
      keys_out[pos] = k[i];
      vals_out[pos] = v[i];
    }
  }
}

// ---- 3./6. single-pass scans with decoupled look-back ---------------------------------------
struct HeadPos {  // value(p) = p if the sorted key changes at p, else 0
  const uint32_t* keys;
  __device__ int32_t operator()(int64_t p) const {
    return (p == 0 || keys[p] != keys[p - 1]) ? (int32_t)p : 0;
  }
};
struct IsRep {  // value(i) = 1 if row i represents its group
  const int32_t* rep;
  __device__ int32_t operator()(int64_t i) const { return rep[i] == (int32_t)i ? 1 : 0; }
};
struct OpMax {
  __device__ int32_t operator()(int32_t a, int32_t b) const { return a > b ? a : b; }
  static constexpr int32_t identity = 0;
};
struct OpSum {
  __device__ int32_t operator()(int32_t a, int32_t b) const { return a + b; }
  static constexpr int32_t identity = 0;
};

template <class Src, class Op, bool kExclusive>
__global__ void __launch_bounds__(kScanThreads) scan_kernel(Src src, int64_t n, int32_t* out,
                                                            unsigned long long* status,
                                                            uint32_t* tile_ctr,
                                                            int32_t* total_out, unsigned* err) {
  __shared__ uint32_t s_tile;
  __shared__ int32_t s_warp[kScanThreads / 32];
  __shared__ int32_t s_prefix;
  const Op op;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  if (tid == 0) s_tile = atomicAdd(tile_ctr, 1u);
  __syncthreads();
  const uint32_t tile = s_tile;
  const int64_t base = (int64_t)tile * kScanTile + (int64_t)tid * kScanItems;
  int32_t x[kScanItems];
  int32_t run = Op::identity;
#pragma unroll
  for (int i = 0; i < kScanItems; ++i) {
    const int64_t e = base + i;
    x[i] = e < n ? src(e) : Op::identity;
    run = op(run, x[i]);
  }
  // Warp-level inclusive scan of thread totals.
  int32_t incl = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl = op(y, incl);
  }
  if (lane == 31) s_warp[w] = incl;
  __syncthreads();
  int32_t warp_prefix = Op::identity, tile_total = Op::identity;
  for (int i = 0; i < kScanThreads / 32; ++i) {
    if (i < w) warp_prefix = op(warp_prefix, s_warp[i]);
    tile_total = op(tile_total, s_warp[i]);
  }
  int32_t thread_prefix = __shfl_up_sync(0xffffffffu, incl, 1);
  if (lane == 0) thread_prefix = Op::identity;
  thread_prefix = op(warp_prefix, thread_prefix);
  if (tid == 0) {
    volatile unsigned long long* st = status;
    int32_t prefix = Op::identity;
    if (tile == 0) {
      st[0] = (2ull << 32) | (uint32_t)tile_total;
    } else {
      st[tile] = (1ull << 32) | (uint32_t)tile_total;
      bool done = false;
      for (int64_t j0 = (int64_t)tile - 1; j0 >= 0 && !done; j0 -= kLookBatch) {
        unsigned long long sv[kLookBatch];
#pragma unroll
        for (int b = 0; b < kLookBatch; ++b) sv[b] = j0 - b >= 0 ? st[j0 - b] : (2ull << 32);
#pragma unroll
        for (int b = 0; b < kLookBatch; ++b) {
          if (done) break;
          unsigned long long sb = sv[b];
          if ((sb >> 32) == 0) sb = wait_flag64(st + (j0 - b), err);
          if (j0 - b >= 0) prefix = op((int32_t)(uint32_t)sb, prefix);
          if ((sb >> 32) == 2ull) done = true;
        }
      }
      st[tile] = (2ull << 32) | (uint32_t)op(prefix, tile_total);
    }
    s_prefix = prefix;
    const int64_t tiles = (n + kScanTile - 1) / kScanTile;
    if (total_out && (int64_t)tile == tiles - 1) *total_out = op(prefix, tile_total);
  }
  __syncthreads();
  int32_t acc = op(s_prefix, thread_prefix);
#pragma unroll
  for (int i = 0; i < kScanItems; ++i) {
    const int64_t e = base + i;
    if (kExclusive) {
      if (e < n) out[e] = acc;
      acc = op(acc, x[i]);
    } else {
      acc = op(acc, x[i]);
      if (e < n) out[e] = acc;
    }
  }
}

// ---- 4./5. full-row comparison -------------------------------------------------------------------
__device__ __forceinline__ int32_t clamp_len(const int32_t* lens, int64_t r, int32_t stride,
                                             unsigned* err) {
  int32_t L = lens ? __ldg(lens + r) : stride;
  if (L < 0 || L > stride) {
    set_error(err, kErrInvalidArg);
    L = L < 0 ? 0 : stride;
  }
  return L;
}

// Whole warp: are rows a and b equal (same length, same tokens below it)?
template <bool VEC>
__device__ bool rows_equal_warp(const int32_t* __restrict__ tokens, int32_t stride,
                                const int32_t* __restrict__ lens, int64_t a, int64_t b,
                                unsigned* err) {
  const int lane = threadIdx.x & 31;
  const int32_t la = clamp_len(lens, a, stride, err);
  const int32_t lb = clamp_len(lens, b, stride, err);
  if (la != lb) return false;
  const int32_t* ra = tokens + a * (int64_t)stride;
  const int32_t* rb = tokens + b * (int64_t)stride;
  bool diff = false;
  int32_t done = 0;
  if (VEC) {
    // Up to three 16-byte pieces of each row per lane in flight per round
    // trip: a 384-token row is compared in one round trip.
    const int32_t pieces = la >> 2;
    const int4* pa = reinterpret_cast<const int4*>(ra);
    const int4* pb = reinterpret_cast<const int4*>(rb);
    for (int32_t j0 = 0; j0 < pieces; j0 += 96) {
      int4 x[3], y[3];
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        const int32_t j = j0 + u * 32 + lane;
        if (j < pieces) {
          x[u] = __ldg(pa + j);
          y[u] = __ldg(pb + j);
        }
      }
#pragma unroll
      for (int u = 0; u < 3; ++u) {
        const int32_t j = j0 + u * 32 + lane;
        if (j < pieces)
          diff |= (x[u].x != y[u].x) | (x[u].y != y[u].y) | (x[u].z != y[u].z) | (x[u].w != y[u].w);
      }
    }
    done = pieces << 2;
  }
  for (int32_t t = done + lane; t < la; t += 32) diff |= (__ldg(ra + t) != __ldg(rb + t));
  return !__any_sync(0xffffffffu, diff);
}

// Verify: lane i of a warp loads the metadata of position p0+i (segment head,
// row index, head row, both lengths) so the dependent lookups of 32 positions
// share their round trips; then the two half-warps compare two pairs of rows
// at a time, 16 lanes x up to 6 pieces of each row in flight.
template <bool VEC>
__device__ __forceinline__ bool half_rows_differ(const int32_t* __restrict__ tokens,
                                                 int32_t stride, int64_t a, int64_t b, int32_t len,
                                                 int hl) {
  const int32_t* ra = tokens + a * (int64_t)stride;
  const int32_t* rb = tokens + b * (int64_t)stride;
  bool diff = false;
  int32_t done = 0;
  if (VEC) {
    const int32_t pieces = len >> 2;
    const int4* pa = reinterpret_cast<const int4*>(ra);
    const int4* pb = reinterpret_cast<const int4*>(rb);
    for (int32_t j0 = 0; j0 < pieces; j0 += 96) {
      int4 x[6], y[6];
#pragma unroll
      for (int u = 0; u < 6; ++u) {
        const int32_t j = j0 + u * 16 + hl;
        if (j < pieces) {
          x[u] = __ldg(pa + j);
          y[u] = __ldg(pb + j);
        }
      }
#pragma unroll
      for (int u = 0; u < 6; ++u) {
        const int32_t j = j0 + u * 16 + hl;
        if (j < pieces)
          diff |= (x[u].x != y[u].x) | (x[u].y != y[u].y) | (x[u].z != y[u].z) | (x[u].w != y[u].w);
      }
    }
    done = pieces << 2;
  }
  for (int32_t t = done + hl; t < len; t += 16) diff |= (__ldg(ra + t) != __ldg(rb + t));
  return diff;
}

template <bool VEC>
__global__ void __launch_bounds__(256) verify_kernel(
    const uint32_t* __restrict__ vals, const int32_t* __restrict__ seg_head, int64_t n,
    const int32_t* __restrict__ tokens, int32_t stride, const int32_t* __restrict__ lens,
    int32_t* __restrict__ rep, int32_t* coll_flag, int32_t* coll_list, uint32_t* coll_count,
    unsigned* err) {
  const int lane = threadIdx.x & 31, half = lane >> 4, hl = lane & 15;
  const int64_t warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  for (int64_t p0 = w * 32; p0 < n; p0 += warps * 32) {
    const int64_t p = p0 + lane;
    const bool valid = p < n;
    const int32_t h = valid ? seg_head[p] : 0;
    const bool head = valid && h == (int32_t)p;
    const int64_t a = valid ? (int64_t)vals[p] : 0;
    const int64_t b = (valid && !head) ? (int64_t)vals[h] : a;
    const int32_t la = valid ? clamp_len(lens, a, stride, err) : 0;
    const int32_t lb = (valid && !head) ? clamp_len(lens, b, stride, err) : la;
    bool need = valid && !head;
    if (head) rep[a] = (int32_t)a;
    if (need && la != lb) {               // different lengths: never equal
      rep[a] = (int32_t)a;
      if (atomicCAS(coll_flag + h, 0, 1) == 0) coll_list[atomicAdd(coll_count, 1u)] = h;
      need = false;
    }
    unsigned todo = __ballot_sync(0xffffffffu, need);
    while (todo != 0u) {
      const int j0 = __ffs(todo) - 1;
      todo &= todo - 1;
      int j1 = -1;
      if (todo != 0u) {
        j1 = __ffs(todo) - 1;
        todo &= todo - 1;
      }
      const int j = half == 0 ? j0 : j1;
      const int src = j < 0 ? 0 : j;
      const int64_t aj = __shfl_sync(0xffffffffu, a, src);
      const int64_t bj = __shfl_sync(0xffffffffu, b, src);
      const int32_t lj = __shfl_sync(0xffffffffu, la, src);
      const int32_t hj = __shfl_sync(0xffffffffu, h, src);
      const bool diff = j >= 0 && half_rows_differ<VEC>(tokens, stride, aj, bj, lj, hl);
      const unsigned dm = __ballot_sync(0xffffffffu, diff);
      const bool eq = ((dm >> (half * 16)) & 0xffffu) == 0u;
      if (j >= 0 && hl == 0) {
        rep[aj] = eq ? (int32_t)bj : (int32_t)aj;
        if (!eq && atomicCAS(coll_flag + hj, 0, 1) == 0) coll_list[atomicAdd(coll_count, 1u)] = hj;
      }
    }
  }
}

// Regroup the rows of each collided segment exactly.  Within a segment,
// positions are in ascending row order (stable sort), so the first
// unassigned position is the smallest unassigned row index.
template <bool VEC>
__global__ void __launch_bounds__(256) resolve_kernel(
    const uint32_t* __restrict__ vals, const int32_t* __restrict__ seg_head, int64_t n,
    const int32_t* __restrict__ tokens, int32_t stride, const int32_t* __restrict__ lens,
    int32_t* rep, const int32_t* __restrict__ coll_list, const uint32_t* coll_count,
    unsigned* err) {
  __shared__ int64_t s_end;
  __shared__ int32_t s_first;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5, nw = blockDim.x >> 5;
  const uint32_t count = *coll_count;
  for (uint32_t c = blockIdx.x; c < count; c += gridDim.x) {
    const int32_t h = coll_list[c];
    if (tid == 0) s_end = n;
    __syncthreads();
    for (int64_t p = (int64_t)h + 1 + tid; p < n; p += blockDim.x) {
      if (p >= s_end) break;
      if (seg_head[p] != h) {
        atomicMin(reinterpret_cast<unsigned long long*>(&s_end), (unsigned long long)p);
        break;
      }
    }
    __syncthreads();
    const int64_t end = s_end;
    for (int64_t p = (int64_t)h + tid; p < end; p += blockDim.x) rep[vals[p]] = -1;
    __syncthreads();
    for (;;) {
      if (tid == 0) s_first = 0x7fffffff;
      __syncthreads();
      for (int64_t p = (int64_t)h + tid; p < end; p += blockDim.x)
        if (rep[vals[p]] == -1) {
          atomicMin(&s_first, (int32_t)(p - h));
          break;
        }
      __syncthreads();
      const int32_t first = s_first;
      if (first == 0x7fffffff) break;
      const int64_t r = vals[h + first];
      for (int64_t p = (int64_t)h + first + w; p < end; p += nw) {
        const int64_t a = vals[p];
        const int32_t cur = __shfl_sync(0xffffffffu, lane == 0 ? rep[a] : 0, 0);
        if (cur != -1) continue;
        const bool eq = (a == r) || rows_equal_warp<VEC>(tokens, stride, lens, a, r, err);
        if (eq && lane == 0) rep[a] = (int32_t)r;
      }
      __syncthreads();
    }
  }
}

__global__ void __launch_bounds__(256) finalize_kernel(const int32_t* __restrict__ rep,
                                                       const int32_t* __restrict__ uid, int64_t n,
                                                       const int32_t* __restrict__ n_unique,
                                                       int32_t* __restrict__ unique_idx,
                                                       int32_t* __restrict__ inverse) {
  const int64_t nu = *n_unique;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int32_t r = rep[i];
    inverse[i] = uid[r];
    if (r == (int32_t)i) unique_idx[uid[i]] = (int32_t)i;
    if (i >= nu) unique_idx[i] = 0;     // the tail is a valid row map too
  }
}

unsigned grid_for(int64_t items, int per_block, int max_blocks) {
  int64_t b = (items + per_block - 1) / per_block;
  if (b < 1) b = 1;
  if (b > max_blocks) b = max_blocks;
  return (unsigned)b;
}

}  // namespace

size_t unique_inverse_workspace(int64_t n) { return n <= 0 ? 256 : layout(n).total; }

hs_status launch_unique_inverse(const uint64_t* fp, const int32_t* tokens, int64_t n,
                                int32_t stride, const int32_t* lens, int32_t* n_unique_dev,
                                int32_t* unique_idx, int32_t* inverse, void* ws,
                                cudaStream_t stream) {
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const Layout L = layout(n);
  char* w = static_cast<char*>(ws);
  uint32_t* hist = reinterpret_cast<uint32_t*>(w + L.hist);
  uint32_t* status = reinterpret_cast<uint32_t*>(w + L.status);
  uint32_t* ctr = reinterpret_cast<uint32_t*>(w + L.ctr);
  int32_t* coll_flag = reinterpret_cast<int32_t*>(w + L.coll_flag);
  uint32_t* coll_count = reinterpret_cast<uint32_t*>(w + L.coll_count);
  auto* scan0 = reinterpret_cast<unsigned long long*>(w + L.scan_status0);
  auto* scan1 = reinterpret_cast<unsigned long long*>(w + L.scan_status1);
  uint32_t* keys[2] = {reinterpret_cast<uint32_t*>(w + L.keys0),
                       reinterpret_cast<uint32_t*>(w + L.keys1)};
  uint32_t* vals[2] = {reinterpret_cast<uint32_t*>(w + L.vals0),
                       reinterpret_cast<uint32_t*>(w + L.vals1)};
  int32_t* seg_head = reinterpret_cast<int32_t*>(w + L.seg_head);
  int32_t* rep = reinterpret_cast<int32_t*>(w + L.rep);
  int32_t* uid = reinterpret_cast<int32_t*>(w + L.uid);
  int32_t* coll_list = reinterpret_cast<int32_t*>(w + L.coll_list);

  cudaError_t e = cudaMemsetAsync(w, 0, L.zero_end, stream);
  if (e != cudaSuccess) return cuda_fail(e, "workspace clear");
  const int sms = num_sms();
  const int64_t sort_tiles = (n + kSortTile - 1) / kSortTile;
  const int64_t scan_tiles = (n + kScanTile - 1) / kScanTile;

  sort_hist_kernel<<<grid_for(n, 256 * 8, sms * 4), 256, 0, stream>>>(fp, n, hist);
  // Four passes; pass 0 reads the caller's fingerprints and implicit indices.
  const uint32_t* kin = nullptr;
  const uint32_t* vin = nullptr;
  int out = 0;
  for (int pass = 0; pass < kPasses; ++pass) {
    onesweep_kernel<<<(unsigned)sort_tiles, kSortThreads, 0, stream>>>(
        pass, pass == 0 ? fp : nullptr, kin, vin, keys[out], vals[out], n, hist, status, ctr, err);
    kin = keys[out];
    vin = vals[out];
    out ^= 1;
  }
  const uint32_t* skeys = kin;
  const uint32_t* svals = vin;

  scan_kernel<HeadPos, OpMax, false><<<(unsigned)scan_tiles, kScanThreads, 0, stream>>>(
      HeadPos{skeys}, n, seg_head, scan0, ctr + 8, nullptr, err);

  const bool vec = ((reinterpret_cast<uintptr_t>(tokens) & 15u) == 0) && (stride % 4 == 0);
  const unsigned vgrid = grid_for(n, 256, sms * 8);   // one warp per 32 positions
  if (vec)
    verify_kernel<true><<<vgrid, 256, 0, stream>>>(svals, seg_head, n, tokens, stride, lens, rep,
                                                   coll_flag, coll_list, coll_count, err);
  else
    verify_kernel<false><<<vgrid, 256, 0, stream>>>(svals, seg_head, n, tokens, stride, lens,
                                                    rep, coll_flag, coll_list, coll_count, err);
  if (vec)
    resolve_kernel<true><<<(unsigned)sms, 256, 0, stream>>>(svals, seg_head, n, tokens, stride,
                                                            lens, rep, coll_list, coll_count, err);
  else
    resolve_kernel<false><<<(unsigned)sms, 256, 0, stream>>>(svals, seg_head, n, tokens, stride,
                                                             lens, rep, coll_list, coll_count,
                                                             err);
  scan_kernel<IsRep, OpSum, true><<<(unsigned)scan_tiles, kScanThreads, 0, stream>>>(
      IsRep{rep}, n, uid, scan1, ctr + 9, n_unique_dev, err);
  finalize_kernel<<<grid_for(n, 256, sms * 8), 256, 0, stream>>>(rep, uid, n, n_unique_dev,
                                                                 unique_idx, inverse);
  count_launches(10);  // hist, 4 radix passes, 2 scans, verify, resolve, finalize
  return cuda_fail(cudaGetLastError(), "unique_inverse launch");
}

}  // namespace hs

// ---- allocation-free entry point -------------------------------------------------------------
// Some callers cannot allocate device memory at the moment they merge rows:
// code that runs while a CUDA graph is being captured (an allocation there
// would be recorded into, or break, the graph), plugins and embedded runtimes
// that are handed a fixed memory budget and may not touch the allocator, and
// latency-critical request paths where an allocator call (or a pool that has
// to grow) is an unbounded stall.  hs_unique_inverse_noalloc serves them with
// a scratch area that is part of the library's own module memory: a
// file-scope device array sized for kNoAllocMaxRows rows (about 2.5 MB),
// which every GPU that loads the library holds until the process exits.
namespace hs {
namespace {
constexpr int64_t kNoAllocMaxRows = 65536;
constexpr size_t kNoAllocBytes = layout(kNoAllocMaxRows).total;
static __device__ __align__(256) unsigned char g_noalloc_ws[kNoAllocBytes];
constexpr int kNoAllocDevices = 64;
void* g_noalloc_addr[kNoAllocDevices] = {};
std::mutex g_noalloc_mu;

// Device address of this device's copy of the scratch array.  In host code
// the array's name is only a host-side stand-in, so the address is looked up
// once per device, with that device current, and cached.
hs_status noalloc_scratch(void** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kNoAllocDevices) return fail(HS_ERR_UNSUPPORTED, "device index %d", dev);
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_ws);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(scratch)");
    g_noalloc_addr[dev] = p;
  }
  *out = g_noalloc_addr[dev];
  return HS_OK;
}
}  // namespace
}  // namespace hs

extern "C" hs_status hs_unique_inverse_noalloc(const uint64_t* fp, const int32_t* tokens,
                                               int64_t n_rows, int32_t row_stride,
                                               const int32_t* lens, int32_t* n_unique_dev,
                                               int32_t* unique_idx_out, int32_t* inverse_out,
                                               hs_stream_t stream) {
  using namespace hs;
  clear_last_error();
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (n_rows < 0 || n_rows > kNoAllocMaxRows)
    return fail(HS_ERR_INVALID_ARG, "n_rows outside [0, %lld], the allocation-free limit",
                (long long)kNoAllocMaxRows);
  if (row_stride < 0) return fail(HS_ERR_INVALID_ARG, "row_stride < 0");
  if (!n_unique_dev) return fail(HS_ERR_INVALID_ARG, "n_unique_dev is NULL");
  if (reinterpret_cast<uintptr_t>(n_unique_dev) % 4)
    return fail(HS_ERR_INVALID_ARG, "n_unique_dev misaligned");
  if (n_rows == 0)
    return cuda_fail(cudaMemsetAsync(n_unique_dev, 0, sizeof(int32_t), s), "n_unique clear");
  if (!fp || !unique_idx_out || !inverse_out || (!tokens && row_stride > 0))
    return fail(HS_ERR_INVALID_ARG, "NULL input or output pointer");
  if (reinterpret_cast<uintptr_t>(fp) % 8 || reinterpret_cast<uintptr_t>(tokens) % 4 ||
      (lens && reinterpret_cast<uintptr_t>(lens) % 4) ||
      reinterpret_cast<uintptr_t>(unique_idx_out) % 4 ||
      reinterpret_cast<uintptr_t>(inverse_out) % 4)
    return fail(HS_ERR_INVALID_ARG, "misaligned pointer");
  void* scratch = nullptr;
  const hs_status st = noalloc_scratch(&scratch);
  if (st != HS_OK) return st;
  // launch_unique_inverse clears the parts of the scratch that must start at
  // zero on every call, so what an earlier call left there does not matter.
  return launch_unique_inverse(fp, tokens, n_rows, row_stride, lens, n_unique_dev,
                               unique_idx_out, inverse_out, scratch, s);
}
