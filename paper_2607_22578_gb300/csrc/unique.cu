// K2-K4: exact unique-with-inverse over fingerprinted rows — the merge step of
// topological fusion within a time window (Section 3.3, "Dynamic Fusion and
// Reuse Mechanism" (I)) and the merge sets M(v*) of Appendix A.2.
//
// The window's matching of a new node against the nodes already seen is a
// lookup by signature; here it is a device hash table keyed by the 64-bit
// fingerprint, whose value is the smallest row index carrying that key:
//   1. insert: every row offers (fp, i); equal fingerprints within a warp are
//      combined first, the slot keeps the minimum index (atomicMin);
//   2. lookup + verify: rep[i] = the slot's index; a row with rep[i] != i is
//      compared in full (length + tokens) with row rep[i] (two rows per warp
//      round, 16 lanes each).  A mismatch — rows with equal fingerprints but
//      different contents — sends the row to a collision list;
//   3. collision list (empty unless fingerprints collide): exact regrouping
//      in linear work — the listed rows are grouped again by a second key
//      (a different hash of the row, mixed with its fingerprint) in the now
//      free table, and each is compared with the smallest listed row of its
//      group; rows that collide in both keys (practically never) are peeled:
//      the smallest unassigned one becomes a representative and every one
//      equal to it joins it;
//   4. exclusive sum-scan of "row is its own representative" gives each
//      group its ordinal in first-occurrence order (single pass, decoupled
//      look-back with bounded spins); the final kernel writes unique_idx and
//      inverse.
// Up to kSmallRows rows, one launch does it all: every CTA builds the table
// for all rows in its own shared memory (the same table in each), verifies
// its share of the rows, and the last CTA to finish resolves the collision
// list, scans and writes the outputs.
#include <mutex>

#include "fnv.cuh"
#include "hs_internal.cuh"
#include "row_table.cuh"

namespace hs {
namespace {

using namespace table;

constexpr int kScanThreads = 1024;
constexpr int kScanItems = 16;
constexpr int kScanTile = kScanThreads * kScanItems;
static_assert(kScanThreads % 32 == 0 && kScanThreads <= 1024, "scan block: whole warps, at most 32");
constexpr int kLookBatch = 8;           // predecessor statuses read per round trip
constexpr int64_t kSmallRows = 4096;    // single-launch path
constexpr int kSmallThreads = 512;
constexpr int kResolveThreads = 512;    // one block for the collision list

constexpr size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct Layout {
  int log2T;
  // zero-initialised region first, then the region set to all-ones bytes
  size_t ctr, scan_status, zero_end;
  size_t keys, idx, ones_end;
  size_t rep, uid, coll_list, total;
};

// Counters (uint32 each) in the zeroed region.
constexpr int kCtrColl = 0;   // collision list length
constexpr int kCtrScan = 1;   // scan tile ticket
constexpr int kCtrDone = 2;   // CTAs finished (single-launch path)

constexpr Layout layout(int64_t n) {
  Layout L{};
  L.log2T = table_log2(n);
  const size_t T1 = (size_t(1) << L.log2T) + 1;   // + the slot of fingerprint kEmpty
  const int64_t tiles = (n + kScanTile - 1) / kScanTile;
  size_t o = 0;
  L.ctr = o;          o += align256(sizeof(uint32_t) * 16);
  L.scan_status = o;  o += align256(sizeof(uint64_t) * (size_t)tiles);
  L.zero_end = o;
  L.keys = o;         o += align256(sizeof(uint64_t) * T1);
  L.idx = o;          o += align256(sizeof(uint32_t) * T1);
  L.ones_end = o;
  L.rep = o;          o += align256(sizeof(int32_t) * (size_t)n);
  L.uid = o;          o += align256(sizeof(int32_t) * (size_t)n);
  L.coll_list = o;    o += align256(sizeof(int32_t) * (size_t)n);
  L.total = o;
  return L;
}

// ---- row comparison ---------------------------------------------------------------------------
__device__ __forceinline__ int32_t clamp_len(const int32_t* lens, int64_t r, int32_t stride,
                                             unsigned* err) {
  int32_t L = lens ? __ldg(lens + r) : stride;
  if (L < 0 || L > stride) {
    set_error(err, kErrInvalidArg);
    L = L < 0 ? 0 : stride;
  }
  return L;
}

// Half-warp: do rows a and b differ in their first len tokens?  16 lanes, up
// to six 16-byte pieces of each row per lane in flight per round trip.
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

// Whole warp: lane l holds a pair (a, b) with `need` set if the rows must be
// compared (their lengths, la, are equal).  Pairs are compared two at a time
// (one per half-warp).  Returns, to each lane, whether its pair differs.
template <bool VEC>
__device__ __forceinline__ bool warp_pairs_differ(const int32_t* __restrict__ tokens,
                                                  int32_t stride, bool need, int64_t a, int64_t b,
                                                  int32_t la) {
  const int lane = threadIdx.x & 31, half = lane >> 4, hl = lane & 15;
  unsigned todo = __ballot_sync(0xffffffffu, need);
  unsigned differ = 0u;
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
    const bool diff = j >= 0 && half_rows_differ<VEC>(tokens, stride, aj, bj, lj, hl);
    const unsigned dm = __ballot_sync(0xffffffffu, diff);
    if ((dm & 0xffffu) != 0u) differ |= 1u << j0;
    if (j1 >= 0 && (dm >> 16) != 0u) differ |= 1u << j1;
  }
  return (differ >> lane) & 1u;
}

// Whole warp: are rows a and b equal (same length, same tokens below it)?
template <bool VEC>
__device__ __forceinline__ bool rows_equal_warp(const int32_t* __restrict__ tokens, int32_t stride,
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
    const int32_t pieces = la >> 2;
    const int4* pa = reinterpret_cast<const int4*>(ra);
    const int4* pb = reinterpret_cast<const int4*>(rb);
    for (int32_t j = lane; j < pieces; j += 32) {
      const int4 x = __ldg(pa + j), y = __ldg(pb + j);
      diff |= (x.x != y.x) | (x.y != y.y) | (x.z != y.z) | (x.w != y.w);
    }
    done = pieces << 2;
  }
  for (int32_t t = done + lane; t < la; t += 32) diff |= (__ldg(ra + t) != __ldg(rb + t));
  return !__any_sync(0xffffffffu, diff);
}

// Verify the 32 rows [p0, p0+32) of one warp against their tentative
// representatives r (lane = row).  Returns, per lane, whether the row stays
// merged with r (true for a row that is its own representative).
template <bool VEC>
__device__ __forceinline__ bool verify_warp(const int32_t* __restrict__ tokens, int32_t stride,
                                            const int32_t* __restrict__ lens, bool valid,
                                            int64_t a, int64_t r, unsigned* err) {
  const bool self = !valid || r == a;
  const int32_t la = valid ? clamp_len(lens, a, stride, err) : 0;
  const int32_t lr = self ? la : clamp_len(lens, r, stride, err);
  const bool need = !self && la == lr;
  const bool differ = warp_pairs_differ<VEC>(tokens, stride, need, a, r, la);
  return self || (need && !differ);
}

// Second grouping key of row a for the collision list: a multiply-xorshift
// hash over its length and tokens (structurally unlike FNV-1a, so rows whose
// fingerprints collide almost never collide here too), mixed with the row's
// fingerprint.  Rows with equal contents get equal keys, because their
// fingerprints are equal.  The key only groups rows for the comparison that
// follows, so exactness does not depend on it.
template <bool VEC>
__device__ __forceinline__ uint64_t regroup_key(const uint64_t* __restrict__ fp, const int32_t* __restrict__ tokens,
                                int32_t stride, const int32_t* __restrict__ lens, int64_t a,
                                unsigned* err) {
  constexpr uint64_t kMul = 0x9E3779B97F4A7C15ull, kFin = 0xD6E8FEB86659FD93ull;
  const int32_t len = clamp_len(lens, a, stride, err);
  const int32_t* row = tokens + a * (int64_t)stride;
  uint64_t h = 0x243F6A8885A308D3ull ^ (uint64_t)(uint32_t)len;
  int32_t t = 0;
  if (VEC) {
    const int4* p = reinterpret_cast<const int4*>(row);
#pragma unroll 1
    for (; t + 4 <= len; t += 4) {
      const int4 v = __ldg(p + (t >> 2));
      h = (h ^ (uint32_t)v.x) * kMul;
      h ^= h >> 29;
      h = (h ^ (uint32_t)v.y) * kMul;
      h ^= h >> 29;
      h = (h ^ (uint32_t)v.z) * kMul;
      h ^= h >> 29;
      h = (h ^ (uint32_t)v.w) * kMul;
      h ^= h >> 29;
    }
  }
#pragma unroll 1
  for (; t < len; ++t) {
    h = (h ^ (uint32_t)__ldg(row + t)) * kMul;
    h ^= h >> 29;
  }
  h ^= __ldg(fp + a) * kFin;
  h ^= h >> 32;
  h *= kFin;
  return h ^ (h >> 29);
}

// Exact regrouping of the m listed rows (rep == -1: each differs from the
// smallest row with its fingerprint, so it can only equal other listed
// rows) in linear work; one block.  The listed rows are grouped by
// regroup_key in the table keys/idx (any contents; it needs
// 2^table_log2(m) + 1 slots), each row is compared in full with the
// smallest listed row of its group and joins it if equal (the smallest row
// of a group is its own representative: every row equal to it is listed and
// in its group).  A row that differs from its group's smallest row as well
// goes to list2; returns their number, the same in every thread.
template <bool VEC>
__device__ __forceinline__ uint32_t regroup_block(const uint64_t* __restrict__ fp,
                                  const int32_t* __restrict__ tokens, int32_t stride,
                                  const int32_t* __restrict__ lens, int32_t* rep,
                                  const int32_t* list, uint32_t m, uint64_t* keys, uint32_t* idx,
                                  int32_t* list2, unsigned* err) {
  __shared__ uint32_t s_m2;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5, nw = blockDim.x >> 5;
  const int log2M = table_log2(m);
  const uint32_t T1 = (1u << log2M) + 1u;
  for (uint32_t s = tid; s < T1; s += blockDim.x) {
    keys[s] = kEmpty;
    idx[s] = kNoRow;
  }
  if (tid == 0) s_m2 = 0;
  __syncthreads();
  for (uint32_t c = tid; c < m; c += blockDim.x) {   // list order is arbitrary: no combining
    const int32_t a = list[c];
    const uint32_t s = insert_key(keys, regroup_key<VEC>(fp, tokens, stride, lens, a, err), log2M);
    atomicMin(idx + s, (uint32_t)a);
  }
  __syncthreads();
  for (uint32_t b = (uint32_t)w * 32u; b < m; b += (uint32_t)nw * 32u) {
    const uint32_t c = b + lane;
    const bool valid = c < m;
    const int64_t a = valid ? list[c] : 0;
    int64_t r = a;
    if (valid) {
      const uint64_t k2 = regroup_key<VEC>(fp, tokens, stride, lens, a, err);
      const uint32_t v = idx[find_key(keys, k2, log2M)];
      if (v != kNoRow) r = v;
    }
    const bool merged = verify_warp<VEC>(tokens, stride, lens, valid, a, r, err);
    if (valid) {
      if (merged)
        rep[a] = (int32_t)r;
      else
        list2[atomicAdd(&s_m2, 1u)] = (int32_t)a;
    }
  }
  __syncthreads();
  return s_m2;
}

// Exact regrouping of the listed rows (rep == -1) by peeling; one block.
// Listed rows differ from the representative of their fingerprint, so they
// can only equal each other; the smallest unassigned row of each content
// becomes its representative.  rep may be in shared or global memory.
template <bool VEC>
__device__ __forceinline__ void peel_block(const uint64_t* __restrict__ fp, const int32_t* __restrict__ tokens,
                           int32_t stride, const int32_t* __restrict__ lens, int32_t* rep,
                           const int32_t* coll_list, uint32_t m, unsigned* err) {
  __shared__ int32_t s_first;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5, nw = blockDim.x >> 5;
  for (;;) {
    if (tid == 0) s_first = 0x7fffffff;
    __syncthreads();
    int32_t mine = 0x7fffffff;
    for (uint32_t c = tid; c < m; c += blockDim.x) {
      const int32_t a = coll_list[c];
      if (*reinterpret_cast<volatile int32_t*>(rep + a) == -1 && a < mine) mine = a;
    }
    if (mine != 0x7fffffff) atomicMin(&s_first, mine);
    __syncthreads();
    const int32_t a0 = s_first;
    if (a0 == 0x7fffffff) break;
    const uint64_t f0 = fp[a0];
    for (uint32_t c = w; c < m; c += nw) {
      const int32_t b = coll_list[c];
      if (b == a0 || *reinterpret_cast<volatile int32_t*>(rep + b) != -1 || fp[b] != f0) continue;
      if (rows_equal_warp<VEC>(tokens, stride, lens, a0, b, err) && lane == 0) rep[b] = a0;
    }
    __syncthreads();
    if (tid == 0) rep[a0] = a0;
    __syncthreads();
  }
}

// ---- multi-kernel path ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) insert_kernel(const uint64_t* __restrict__ fp, int64_t n,
                                                     uint64_t* keys, uint32_t* idx, int log2T) {
  pdl_wait();
  pdl_trigger();
  for (int64_t base = (int64_t)blockIdx.x * blockDim.x; base < n;
       base += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = base + threadIdx.x;
    const bool valid = i < n;
    insert_row(keys, idx, log2T, valid, valid ? __ldg(fp + i) : 0ull, (uint32_t)i);
  }
}

template <bool VEC>
__global__ void __launch_bounds__(256) verify_kernel(
    const uint64_t* __restrict__ fp, int64_t n, const uint64_t* __restrict__ keys,
    const uint32_t* __restrict__ idx, int log2T, const int32_t* __restrict__ tokens,
    int32_t stride, const int32_t* __restrict__ lens, int32_t* __restrict__ rep,
    int32_t* coll_list, uint32_t* ctr, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  for (int64_t p0 = w * 32; p0 < n; p0 += warps * 32) {
    const int64_t a = p0 + lane;
    const bool valid = a < n;
    int64_t r = a;
    if (valid) {
      const uint32_t v = idx[find_key(keys, __ldg(fp + a), log2T)];
      if (v < (uint32_t)n) r = v;
      else set_error(err, kErrInvalidArg);   // not reached: every row was inserted
    }
    const bool merged = verify_warp<VEC>(tokens, stride, lens, valid, a, r, err);
    if (valid) {
      rep[a] = merged ? (int32_t)r : -1;
      if (!merged) coll_list[atomicAdd(ctr + kCtrColl, 1u)] = (int32_t)a;
    }
  }
}

// The collision list, after verify: the table is free again (verify was its
// last reader) and so is uid (the scan writes it next), which holds list2.
template <bool VEC>
__global__ void __launch_bounds__(kResolveThreads) resolve_kernel(
    const uint64_t* __restrict__ fp, const int32_t* __restrict__ tokens, int32_t stride,
    const int32_t* __restrict__ lens, int32_t* rep, const int32_t* coll_list,
    const uint32_t* ctr, uint64_t* keys, uint32_t* idx, int32_t* list2, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  const uint32_t m = ctr[kCtrColl];
  if (m == 0) return;
  const uint32_t m2 = regroup_block<VEC>(fp, tokens, stride, lens, rep, coll_list, m, keys, idx,
                                         list2, err);
  if (m2 > 0) peel_block<VEC>(fp, tokens, stride, lens, rep, list2, m2, err);
}

// Single-pass exclusive sum-scan of "rep[i] == i" with decoupled look-back;
// the last tile writes the total (the group count).  A predecessor's status
// is awaited for at most limit_ns of %globaltimer; then the wait gives up,
// sets kErrTimeout and counts the predecessor as a zero prefix (the call's
// outputs are then unspecified, but every write stays in bounds).
__device__ __forceinline__ uint64_t wait_status(const volatile unsigned long long* p,
                                                unsigned* err, uint64_t limit_ns) {
  unsigned long long s = *p;
  if (s >> 32) return s;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    s = *p;
    if (s >> 32) return s;
    if ((it & 31u) == 0) {
      __nanosleep(64);
      if (globaltimer_ns() - t0 > limit_ns) {
        set_error(err, kErrTimeout);
        return 2ull << 32;  // give up: treat as a zero prefix
      }
    }
  }
}

__global__ void __launch_bounds__(kScanThreads) scan_kernel(const int32_t* __restrict__ rep,
                                                            int64_t n, int32_t* __restrict__ uid,
                                                            unsigned long long* status,
                                                            uint32_t* ctr, int32_t* total_out,
                                                            unsigned* err, uint64_t limit_ns,
                                                            int64_t withhold_tile) {
  pdl_wait();
  pdl_trigger();
  __shared__ uint32_t s_tile;
  __shared__ int32_t s_warp[kScanThreads / 32];
  __shared__ int32_t s_prefix;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  if (tid == 0) s_tile = atomicAdd(ctr + kCtrScan, 1u);
  __syncthreads();
  const uint32_t tile = s_tile;
  const int64_t base = (int64_t)tile * kScanTile + (int64_t)tid * kScanItems;
  int32_t x[kScanItems];
  int32_t run = 0;
#pragma unroll
  for (int i = 0; i < kScanItems; i += 4) {
    const int64_t e = base + i;
    if (e + 3 < n) {
      const int4 v = *reinterpret_cast<const int4*>(rep + e);
      x[i] = v.x == (int32_t)e;
      x[i + 1] = v.y == (int32_t)(e + 1);
      x[i + 2] = v.z == (int32_t)(e + 2);
      x[i + 3] = v.w == (int32_t)(e + 3);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) x[i + j] = (e + j < n) ? (rep[e + j] == (int32_t)(e + j)) : 0;
    }
    run += x[i] + x[i + 1] + x[i + 2] + x[i + 3];
  }
  int32_t incl = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) s_warp[w] = incl;
  __syncthreads();
  if (w == 0) {
    constexpr int kWarps = kScanThreads / 32;
    const int32_t v = lane < kWarps ? s_warp[lane] : 0;
    int32_t iv = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t y = __shfl_up_sync(0xffffffffu, iv, o);
      if (lane >= o) iv += y;
    }
    if (lane < kWarps) s_warp[lane] = iv - v;  // exclusive warp offsets
    if (lane == 31) {
      const int32_t tile_total = iv;
      volatile unsigned long long* st = status;
      int32_t prefix = 0;
      // A withheld tile (test hook, -1 in normal use) never publishes, so
      // its successors' waits run out.
      const bool publish = (int64_t)tile != withhold_tile;
      if (tile == 0) {
        if (publish) st[0] = (2ull << 32) | (uint32_t)tile_total;
      } else {
        if (publish) st[tile] = (1ull << 32) | (uint32_t)tile_total;
        bool done = false;
        for (int64_t j0 = (int64_t)tile - 1; j0 >= 0 && !done; j0 -= kLookBatch) {
          unsigned long long sv[kLookBatch];
#pragma unroll
          for (int b = 0; b < kLookBatch; ++b) sv[b] = j0 - b >= 0 ? st[j0 - b] : (2ull << 32);
#pragma unroll
          for (int b = 0; b < kLookBatch; ++b) {
            if (done) break;
            unsigned long long sb = sv[b];
            if ((sb >> 32) == 0) sb = wait_status(st + (j0 - b), err, limit_ns);
            if (j0 - b >= 0) prefix += (int32_t)(uint32_t)sb;
            if ((sb >> 32) == 2ull) done = true;
          }
        }
        if (publish) st[tile] = (2ull << 32) | (uint32_t)(prefix + tile_total);
      }
      s_prefix = prefix;
      const int64_t tiles = (n + kScanTile - 1) / kScanTile;
      if ((int64_t)tile == tiles - 1) *total_out = prefix + tile_total;
    }
  }
  __syncthreads();
  int32_t acc = s_prefix + s_warp[w] + incl - run;
  int32_t u[kScanItems];
#pragma unroll
  for (int i = 0; i < kScanItems; ++i) {
    u[i] = acc;
    acc += x[i];
  }
  if (base + kScanItems <= n) {
#pragma unroll
    for (int i = 0; i < kScanItems; i += 4)
      *reinterpret_cast<int4*>(uid + base + i) = make_int4(u[i], u[i + 1], u[i + 2], u[i + 3]);
  } else {
#pragma unroll
    for (int i = 0; i < kScanItems; ++i)
      if (base + i < n) uid[base + i] = u[i];
  }
}

__global__ void __launch_bounds__(256) finalize_kernel(const int32_t* __restrict__ rep,
                                                       const int32_t* __restrict__ uid, int64_t n,
                                                       const int32_t* __restrict__ n_unique,
                                                       int32_t* __restrict__ unique_idx,
                                                       int32_t* __restrict__ inverse) {
  pdl_wait();
  pdl_trigger();
  const int64_t nu = *n_unique;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int32_t r = rep[i];
    inverse[i] = uid[r];
    if (r == (int32_t)i) unique_idx[uid[i]] = (int32_t)i;
    if (i >= nu) unique_idx[i] = 0;     // the tail is a valid row map too
  }
}

// ---- verify over flat piece lists ------------------------------------------------------------
// Verify of 32 consecutive rows per warp against their representatives (the
// table's smallest row with the same fingerprint).  The rows that need a
// comparison (representative another row, lengths equal) are compared as
// one flat list of 16-byte piece pairs: the warp's pairs are laid end to
// end (a prefix sum of their piece counts in shared memory), and each lane
// takes every 32nd piece pair, kVerifyPieces of them in flight per round,
// so a warp's rows cost about (their bytes / 4 KB) round trips whatever
// their lengths.  The tokens of a pair's last piece past its length are
// masked.  Needs 16-byte aligned rows (stride % 4 == 0).  Verifies rows
// [row0, row_end) of n (row indices, the table and rep are global).
constexpr int kVerifyPieces = 4;
constexpr int kVerifyThreads = 256;

__global__ void __launch_bounds__(kVerifyThreads) verify_flat_kernel(
    const uint64_t* __restrict__ fp, uint64_t key_mask, int64_t n, int64_t row0, int64_t row_end,
    const uint64_t* __restrict__ keys, const uint32_t* __restrict__ idx, int log2T,
    const int32_t* __restrict__ tokens, int32_t stride, const int32_t* __restrict__ lens,
    int32_t* __restrict__ rep, int32_t* coll_list, uint32_t* ctr, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  __shared__ int32_t s_pre[kVerifyThreads / 32][32];
  __shared__ int32_t s_a[kVerifyThreads / 32][32];
  __shared__ int32_t s_b[kVerifyThreads / 32][32];
  __shared__ int32_t s_len[kVerifyThreads / 32][32];
  const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
  const int64_t warps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  for (int64_t p0 = row0 + w * 32; p0 < row_end; p0 += warps * 32) {
    const int64_t a = p0 + lane;
    const bool valid = a < row_end;
    int64_t r = a;
    int32_t la = 0, lr = 0;
    if (valid) {
      const uint32_t v = idx[find_key(keys, __ldg(fp + a) & key_mask, log2T)];
      if (v < (uint32_t)n) r = v;
      else set_error(err, kErrInvalidArg);   // not reached: every row was inserted
      la = clamp_len(lens, a, stride, err);
      lr = r != a ? clamp_len(lens, r, stride, err) : la;
    }
    const bool need = valid && r != a && la == lr;
    int32_t incl = need ? (la + 3) >> 2 : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    s_pre[wl][lane] = incl;
    s_a[wl][lane] = (int32_t)a;
    s_b[wl][lane] = (int32_t)r;
    s_len[wl][lane] = la;
    const int32_t total = __shfl_sync(0xffffffffu, incl, 31);
    __syncwarp();
    uint32_t differ = 0;                       // bit t: a piece of pair t differs
    int t = 0;                                 // this lane's current pair (only moves forward)
    for (int32_t g0 = 0; g0 < total; g0 += 32 * kVerifyPieces) {
      uint4 x[kVerifyPieces], y[kVerifyPieces];
      int tt[kVerifyPieces], vt[kVerifyPieces];
#pragma unroll
      for (int u = 0; u < kVerifyPieces; ++u) {
        const int32_t g = g0 + u * 32 + lane;
        tt[u] = -1;
        if (g < total) {
          while (s_pre[wl][t] <= g) ++t;
          const int32_t j = g - (t > 0 ? s_pre[wl][t - 1] : 0);
          x[u] = __ldg(reinterpret_cast<const uint4*>(tokens + (int64_t)s_a[wl][t] * stride) + j);
          y[u] = __ldg(reinterpret_cast<const uint4*>(tokens + (int64_t)s_b[wl][t] * stride) + j);
          tt[u] = t;
          vt[u] = s_len[wl][t] - 4 * j;        // live tokens in this piece (>= 1)
        }
      }
#pragma unroll
      for (int u = 0; u < kVerifyPieces; ++u) {
        if (tt[u] >= 0) {
          const bool d = (x[u].x != y[u].x) | ((vt[u] > 1) & (x[u].y != y[u].y)) |
                         ((vt[u] > 2) & (x[u].z != y[u].z)) | ((vt[u] > 3) & (x[u].w != y[u].w));
          if (d) differ |= 1u << tt[u];
        }
      }
    }
    differ = __reduce_or_sync(0xffffffffu, differ);
    __syncwarp();                              // shared lists free for the next rows
    if (valid) {
      const bool merged = r == a || (need && !((differ >> lane) & 1u));
      rep[a] = merged ? (int32_t)r : -1;
      if (!merged) coll_list[atomicAdd(ctr + kCtrColl, 1u)] = (int32_t)a;
    }
  }
}

// ---- hs_merge_rows: second pass of the fingerprint, fused with the insert ---------------------
// One thread per row finishes the fingerprint (the last L mod 32 tokens,
// from the state the chunk kernel left in fp_out, or the whole row when it
// is shorter than 32 tokens or the chunk kernel did not run), writes it,
// and offers (fp & key_mask, row) to the table in the same pass: rows of a
// warp with equal keys are combined and the smallest index inserts
// (atomicMin), as insert_kernel does.  An invalid length sets the error
// word and a zero fingerprint, as hs_fingerprint does.  Rows [row0,
// row_end); row0 is a multiple of 32 (warps combine their rows' inserts).
__global__ void __launch_bounds__(256) tails_insert_kernel(
    const int32_t* __restrict__ tokens, int64_t row0, int64_t row_end, int32_t stride,
    const int32_t* __restrict__ lens, uint64_t seed, bool chunks_ran, uint64_t key_mask,
    uint64_t* __restrict__ fp_out, uint64_t* keys, uint32_t* idx, int log2T, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  constexpr int T = 32;
  for (int64_t base = row0 + (int64_t)blockIdx.x * blockDim.x; base < row_end;
       base += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = base + threadIdx.x;
    const bool valid = r < row_end;
    uint64_t f = 0;
    if (valid) {
      const int32_t L = lens ? __ldg(lens + r) : stride;
      if (L < 0 || L > stride) {
        set_error(err, kErrInvalidArg);
      } else {
        const int32_t m = L % T;
        const bool from_chunks = chunks_ran && L >= T;
        if (from_chunks && m == 0) {
          f = fp_out[r];                           // the chunk kernel wrote the final value
        } else {
          uint32_t lo = (uint32_t)seed, hi = (uint32_t)(seed >> 32);
          int32_t t0 = 0;
          if (from_chunks) {
            const uint64_t st = fp_out[r];
            lo = (uint32_t)st;
            hi = (uint32_t)(st >> 32);
            t0 = L - m;
          }
          // at most 31 tokens remain past the full chunks (fewer than 32 in a
          // short row): all their 16-byte pieces are loaded before hashing
          const int32_t* src = tokens + r * (int64_t)stride + t0;
          const int32_t m2 = L - t0;               // tokens to hash here
          if (m2 < T) {
            uint4 v[T / 4];
#pragma unroll
            for (int q = 0; q < T / 4; ++q)
              if (4 * q < m2) v[q] = __ldg(reinterpret_cast<const uint4*>(src + 4 * q));
#pragma unroll
            for (int q = 0; q < T / 4; ++q) {
              if (4 * q < m2) fnv::hash_word(lo, hi, v[q].x);
              if (4 * q + 1 < m2) fnv::hash_word(lo, hi, v[q].y);
              if (4 * q + 2 < m2) fnv::hash_word(lo, hi, v[q].z);
              if (4 * q + 3 < m2) fnv::hash_word(lo, hi, v[q].w);
            }
          } else {                                 // a whole row (no chunk pass ran)
            for (int32_t t = 0; t < m2; t += 4) {  // 16-byte pieces, the last one masked
              const uint4 v = __ldg(reinterpret_cast<const uint4*>(src + t));
              fnv::hash_word(lo, hi, v.x);
              if (t + 1 < m2) fnv::hash_word(lo, hi, v.y);
              if (t + 2 < m2) fnv::hash_word(lo, hi, v.z);
              if (t + 3 < m2) fnv::hash_word(lo, hi, v.w);
            }
          }
          f = ((uint64_t)hi << 32) | lo;
        }
      }
      fp_out[r] = f;
    }
    insert_row(keys, idx, log2T, valid, f & key_mask, (uint32_t)r);
  }
}

// ---- single-launch path (n <= kSmallRows) ----------------------------------------------------
// Dynamic shared memory: keys[T + 1], idx[T + 1], rep[n], uid[n] (T = 2^log2T).
constexpr size_t small_smem(int64_t n) {
  const size_t T1 = (size_t(1) << table_log2(n)) + 1;
  return T1 * 8 + T1 * 4 + (size_t)n * 8 + 16;
}
static_assert(small_smem(kSmallRows) + kSmallThreads / 32 * 4 + 16 <= 232448,
              "one-launch path: the table, rep and uid fit one CTA's shared memory");

template <bool VEC>
__global__ void __launch_bounds__(kSmallThreads, 1) unique_small_kernel(
    const uint64_t* __restrict__ fp, int64_t n, const int32_t* __restrict__ tokens,
    int32_t stride, const int32_t* __restrict__ lens, int32_t* __restrict__ n_unique,
    int32_t* __restrict__ unique_idx, int32_t* __restrict__ inverse, uint32_t* ctr,
    int32_t* coll_list, unsigned* err) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(16) uint8_t sm[];
  __shared__ bool s_last;
  __shared__ int32_t s_warp[kSmallThreads / 32];
  const int log2T = table_log2(n);
  const uint32_t T1 = (1u << log2T) + 1u;
  uint64_t* keys = reinterpret_cast<uint64_t*>(sm);
  uint32_t* idx = reinterpret_cast<uint32_t*>(keys + T1);
  int32_t* rep = reinterpret_cast<int32_t*>(idx + T1);
  int32_t* uid = rep + n;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  constexpr int kWarps = kSmallThreads / 32;

  // 1. the table for all rows (the same in every CTA)
  for (uint32_t s = tid; s < T1; s += kSmallThreads) {
    keys[s] = kEmpty;
    idx[s] = kNoRow;
  }
  __syncthreads();
  for (int64_t base = 0; base < n; base += kSmallThreads) {
    const int64_t i = base + tid;
    const bool valid = i < n;
    insert_row(keys, idx, log2T, valid, valid ? __ldg(fp + i) : 0ull, (uint32_t)i);
  }
  __syncthreads();
  for (int64_t i = tid; i < n; i += kSmallThreads) {
    const uint32_t v = idx[find_key(keys, __ldg(fp + i), log2T)];
    rep[i] = v < (uint32_t)n ? (int32_t)v : (int32_t)i;
  }
  __syncthreads();

  // 2. verify this CTA's rows: warp-rounds of 32 rows, dealt round-robin
  //    over the CTAs first, so every CTA gets a share
  const int64_t rounds = (n + 31) / 32;
  for (int64_t rd = (int64_t)w * gridDim.x + blockIdx.x; rd < rounds;
       rd += (int64_t)gridDim.x * kWarps) {
    const int64_t a = rd * 32 + lane;
    const bool valid = a < n;
    const int64_t r = valid ? rep[a] : a;
    const bool merged = verify_warp<VEC>(tokens, stride, lens, valid, a, r, err);
    if (valid && !merged) coll_list[atomicAdd(ctr + kCtrColl, 1u)] = (int32_t)a;
  }

  // 3. the last CTA to finish writes the outputs
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(ctr + kCtrDone, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const uint32_t m = *reinterpret_cast<volatile uint32_t*>(ctr + kCtrColl);
  for (uint32_t c = tid; c < m; c += kSmallThreads) rep[coll_list[c]] = -1;
  __syncthreads();
  if (m) {   // the table and uid are free here: uid holds the rows left for peeling
    const uint32_t m2 =
        regroup_block<VEC>(fp, tokens, stride, lens, rep, coll_list, m, keys, idx, uid, err);
    if (m2) peel_block<VEC>(fp, tokens, stride, lens, rep, uid, m2, err);
  }
  __syncthreads();
  // exclusive scan of rep[i] == i: contiguous items per thread
  const int64_t per = (n + kSmallThreads - 1) / kSmallThreads;
  const int64_t b0 = tid * per, b1 = min(n, b0 + per);
  int32_t run = 0;
  for (int64_t i = b0; i < b1; ++i) run += rep[i] == (int32_t)i;
  int32_t incl = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) s_warp[w] = incl;
  __syncthreads();
  int32_t off = 0, total = 0;
  for (int i = 0; i < kWarps; ++i) {
    off += i < w ? s_warp[i] : 0;
    total += s_warp[i];
  }
  int32_t acc = off + incl - run;
  for (int64_t i = b0; i < b1; ++i) {
    uid[i] = acc;
    acc += rep[i] == (int32_t)i;
  }
  __syncthreads();
  for (int64_t i = tid; i < n; i += kSmallThreads) {
    const int32_t r = rep[i];
    inverse[i] = uid[r];
    if (r == (int32_t)i) unique_idx[uid[i]] = (int32_t)i;
  }
  for (int64_t i = total + tid; i < n; i += kSmallThreads) unique_idx[i] = 0;
  if (tid == 0) *n_unique = total;
}

// Test hook of the look-back's bounded wait (hs_debug_scan_wait): the wait
// limit and a tile that does not publish its status (-1: none).
std::atomic<uint64_t> g_scan_wait_limit_ns{kWaitLimitNs};
std::atomic<int64_t> g_scan_withhold_tile{-1};

unsigned grid_for(int64_t items, int per_block, int max_blocks) {
  int64_t b = (items + per_block - 1) / per_block;
  if (b < 1) b = 1;
  if (b > max_blocks) b = max_blocks;
  return (unsigned)b;
}

template <bool VEC>
hs_status launch_small(const uint64_t* fp, const int32_t* tokens, int64_t n, int32_t stride,
                       const int32_t* lens, int32_t* n_unique, int32_t* unique_idx,
                       int32_t* inverse, uint32_t* ctr, int32_t* coll_list, unsigned* err,
                       cudaStream_t stream) {
  const size_t smem = small_smem(n);
  static std::atomic<uint64_t> configured{0};
  if (smem > 48 * 1024) {
    const hs_status cst = once_per_device(configured, [] {
      return cuda_fail(cudaFuncSetAttribute(unique_small_kernel<VEC>,
                                            cudaFuncAttributeMaxDynamicSharedMemorySize,
                                            (int)small_smem(kSmallRows)),
                       "unique smem attribute");
    });
    if (cst != HS_OK) return cst;
  }
  // One CTA per 2 warp-rounds of rows (they wait on memory), at most one per SM.
  const unsigned grid = grid_for((n + 31) / 32, 2, num_sms());
  launch_pdl(unique_small_kernel<VEC>, dim3(grid), dim3(kSmallThreads), smem, stream, fp, n, tokens,
             stride, lens, n_unique, unique_idx, inverse, ctr, coll_list, err);
  return HS_OK;
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
  uint32_t* ctr = reinterpret_cast<uint32_t*>(w + L.ctr);
  auto* status = reinterpret_cast<unsigned long long*>(w + L.scan_status);
  uint64_t* keys = reinterpret_cast<uint64_t*>(w + L.keys);
  uint32_t* idx = reinterpret_cast<uint32_t*>(w + L.idx);
  int32_t* rep = reinterpret_cast<int32_t*>(w + L.rep);
  int32_t* uid = reinterpret_cast<int32_t*>(w + L.uid);
  int32_t* coll_list = reinterpret_cast<int32_t*>(w + L.coll_list);
  const bool vec = ((reinterpret_cast<uintptr_t>(tokens) & 15u) == 0) && (stride % 4 == 0);
  const int sms = num_sms();

  cudaError_t e = cudaMemsetAsync(w, 0, L.zero_end, stream);
  if (e != cudaSuccess) return cuda_fail(e, "workspace clear");
  if (n <= kSmallRows) {
    const hs_status st =
        vec ? launch_small<true>(fp, tokens, n, stride, lens, n_unique_dev, unique_idx, inverse,
                                 ctr, coll_list, err, stream)
            : launch_small<false>(fp, tokens, n, stride, lens, n_unique_dev, unique_idx, inverse,
                                  ctr, coll_list, err, stream);
    if (st != HS_OK) return st;
    count_launches(1);
    return cuda_fail(cudaGetLastError(), "unique_inverse launch");
  }
  e = cudaMemsetAsync(w + L.zero_end, 0xff, L.ones_end - L.zero_end, stream);
  if (e != cudaSuccess) return cuda_fail(e, "hash table clear");
  launch_pdl(insert_kernel, dim3(grid_for(n, 256, sms * 8)), dim3(256), 0, stream, fp, n, keys, idx,
             L.log2T);
  const unsigned vgrid = grid_for(n, 256, sms * 8);   // one warp per 32 rows
  if (vec)
    launch_pdl(verify_flat_kernel, dim3(vgrid), dim3(kVerifyThreads), 0, stream, fp, ~0ull, n,
               (int64_t)0, n, (const uint64_t*)keys, (const uint32_t*)idx, L.log2T, tokens,
               stride, lens, rep, coll_list, ctr, err);
  else
    launch_pdl(verify_kernel<false>, dim3(vgrid), dim3(256), 0, stream, fp, n, keys, idx, L.log2T,
               tokens, stride, lens, rep, coll_list, ctr, err);
  if (vec)
    launch_pdl(resolve_kernel<true>, dim3(1), dim3(kResolveThreads), 0, stream, fp, tokens, stride,
               lens, rep, coll_list, ctr, keys, idx, uid, err);
  else
    launch_pdl(resolve_kernel<false>, dim3(1), dim3(kResolveThreads), 0, stream, fp, tokens,
               stride, lens, rep, coll_list, ctr, keys, idx, uid, err);
  const int64_t tiles = (n + kScanTile - 1) / kScanTile;
  launch_pdl(scan_kernel, dim3((unsigned)tiles), dim3(kScanThreads), 0, stream, rep, n, uid, status,
             ctr, n_unique_dev, err, g_scan_wait_limit_ns.load(), g_scan_withhold_tile.load());
  launch_pdl(finalize_kernel, dim3(grid_for(n, 256, sms * 8)), dim3(256), 0, stream, rep, uid, n,
             n_unique_dev, unique_idx, inverse);
  count_launches(5);  // insert, verify, resolve, scan, finalize
  return cuda_fail(cudaGetLastError(), "unique_inverse launch");
}

hs_status launch_fingerprint(const int32_t*, int64_t, int32_t, const int32_t*, uint64_t,
                             uint64_t*, cudaStream_t);
hs_status launch_fingerprint_chunks(const int32_t*, int64_t, int32_t, const int32_t*, uint64_t,
                                    uint64_t*, bool*, cudaStream_t);

// Test hook of hs_merge_rows (hs_debug_merge_key_mask): the table key is
// fp & mask, so a narrow mask forces fingerprint collisions.
std::atomic<uint64_t> g_merge_key_mask{~0ull};

size_t merge_rows_workspace(int64_t n) { return unique_inverse_workspace(n); }

// hs_merge_rows: the fingerprint's chunk pass, then one pass that finishes
// the fingerprints and inserts them (no separate insert pass), then the
// verify, collision resolve, scan and finalize of hs_unique_inverse.
hs_status launch_merge_rows(const int32_t* tokens, int64_t n, int32_t stride, const int32_t* lens,
                            uint64_t seed, uint64_t* fp_out, int32_t* n_unique_dev,
                            int32_t* unique_idx, int32_t* inverse, void* ws, cudaStream_t stream) {
  const bool vec = ((reinterpret_cast<uintptr_t>(tokens) & 15u) == 0) && (stride % 4 == 0);
  const uint64_t mask = g_merge_key_mask.load();
  if (n <= kSmallRows || !vec) {   // few rows, or rows not 16-byte aligned: the two calls
    hs_status st = launch_fingerprint(tokens, n, stride, lens, seed, fp_out, stream);
    if (st != HS_OK) return st;
    return launch_unique_inverse(fp_out, tokens, n, stride, lens, n_unique_dev, unique_idx,
                                 inverse, ws, stream);
  }
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const Layout L = layout(n);
  char* w = static_cast<char*>(ws);
  uint32_t* ctr = reinterpret_cast<uint32_t*>(w + L.ctr);
  auto* status = reinterpret_cast<unsigned long long*>(w + L.scan_status);
  uint64_t* keys = reinterpret_cast<uint64_t*>(w + L.keys);
  uint32_t* idx = reinterpret_cast<uint32_t*>(w + L.idx);
  int32_t* rep = reinterpret_cast<int32_t*>(w + L.rep);
  int32_t* uid = reinterpret_cast<int32_t*>(w + L.uid);
  int32_t* coll_list = reinterpret_cast<int32_t*>(w + L.coll_list);
  const int sms = num_sms();
  cudaError_t e = cudaMemsetAsync(w, 0, L.zero_end, stream);
  if (e != cudaSuccess) return cuda_fail(e, "workspace clear");
  e = cudaMemsetAsync(w + L.zero_end, 0xff, L.ones_end - L.zero_end, stream);
  if (e != cudaSuccess) return cuda_fail(e, "hash table clear");
  bool ran = false;
  const hs_status st =
      launch_fingerprint_chunks(tokens, n, stride, lens, seed, fp_out, &ran, stream);
  if (st != HS_OK) return st;
  launch_pdl(tails_insert_kernel, dim3(grid_for(n, 256, sms * 16)), dim3(256), 0, stream, tokens,
             (int64_t)0, n, stride, lens, seed, ran, mask, fp_out, keys, idx, L.log2T, err);
  launch_pdl(verify_flat_kernel, dim3(grid_for(n, kVerifyThreads, sms * 8)), dim3(kVerifyThreads),
             0, stream, (const uint64_t*)fp_out, mask, n, (int64_t)0, n, (const uint64_t*)keys,
             (const uint32_t*)idx, L.log2T, tokens, stride, lens, rep, coll_list, ctr, err);
  launch_pdl(resolve_kernel<true>, dim3(1), dim3(kResolveThreads), 0, stream,
             (const uint64_t*)fp_out, tokens, stride, lens, rep, (const int32_t*)coll_list,
             (const uint32_t*)ctr, keys, idx, uid, err);
  const int64_t tiles = (n + kScanTile - 1) / kScanTile;
  launch_pdl(scan_kernel, dim3((unsigned)tiles), dim3(kScanThreads), 0, stream,
             (const int32_t*)rep, n, uid, status, ctr, n_unique_dev, err,
             g_scan_wait_limit_ns.load(), g_scan_withhold_tile.load());
  launch_pdl(finalize_kernel, dim3(grid_for(n, 256, sms * 8)), dim3(256), 0, stream,
             (const int32_t*)rep, (const int32_t*)uid, n, (const int32_t*)n_unique_dev,
             unique_idx, inverse);
  count_launches(5);  // tails+insert, verify, resolve, scan, finalize (the chunk launcher
                      // counts its own)
  return cuda_fail(cudaGetLastError(), "merge_rows launch");
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
// file-scope device array sized for kNoAllocMaxRows rows (2,360,320 bytes),
// which every GPU that loads the library holds until the process exits.
namespace hs {
namespace {
constexpr int64_t kNoAllocMaxRows = 65536;
constexpr size_t kNoAllocBytes = layout(kNoAllocMaxRows).total;
static_assert(kNoAllocBytes == 2360320, "the scratch size stated in hs.h");
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

extern "C" hs_status hs_debug_scan_wait(uint64_t limit_ns, int64_t withhold_tile) {
  using namespace hs;
  clear_last_error();
  if (limit_ns > kWaitLimitNs)
    return fail(HS_ERR_INVALID_ARG, "wait limit above the default of %llu ns",
                (unsigned long long)kWaitLimitNs);
  if (withhold_tile < -1) return fail(HS_ERR_INVALID_ARG, "withhold_tile < -1");
  g_scan_wait_limit_ns.store(limit_ns == 0 ? kWaitLimitNs : limit_ns);
  g_scan_withhold_tile.store(withhold_tile);
  return HS_OK;
}

extern "C" hs_status hs_debug_merge_key_mask(uint64_t mask) {
  hs::clear_last_error();
  hs::g_merge_key_mask.store(mask == 0 ? ~0ull : mask);
  return HS_OK;
}

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
