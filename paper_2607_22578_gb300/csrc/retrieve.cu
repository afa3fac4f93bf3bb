// K6/K7: dense retrieval with a fused per-query top-k — the vector-retrieval
// node shared by merged queries (Section 4.1, "Workloads": embed, retrieve the
// top-k chunks; Section 3.3: merged nodes execute once).
//
//   S = Q * C^T   (bf16 x bf16 -> fp32), per query keep the k best (S, j),
//   ordered by score descending, ties to the lower corpus index j.
//
// K6 (retrieve_kernel) is a persistent, warp-specialised tcgen05 kernel:
//   warp 0      TMA producer: 128x64 query tile + 256x64 corpus tile per
//               stage (CTA pair: + the 128x64 half of it), 128-byte swizzle,
//               4-stage (pair: 6-stage) mbarrier ring;
//   warp 1      MMA issuer: 4 x tcgen05.mma (M=128 or pair M=256, N=256,
//               K=16) per stage into a double-buffered fp32 accumulator in
//               tensor memory (2 x 256 columns), tcgen05.commit releases
//               smem stages;
//   warps 2-9   epilogue: two warps per TMEM lane quarter, each reading half
//               of the 128 x 256 score tile with tcgen05.ld; thread = (query,
//               column half); threshold filter + per-query top-k.
// With two or more query blocks the CTAs run as pairs (clusters of two,
// cta_group::2): the even CTA issues M = 256 MMAs that take the two CTAs'
// query blocks as the two halves of A and the two 128-row halves of the
// corpus tile, one staged in each CTA, as B.  Each CTA's tensor memory holds
// the scores of its own query block against the whole tile, so each SM
// stages half of every corpus tile and reads half as much shared memory per
// MMA as a single CTA would.  The producer of each CTA loads its own query
// tile and corpus half; both complete on the even CTA's barrier.
// The Q x N score matrix never leaves the SM.  Work is split into units
// (query block pair, corpus split); units that share a corpus split run at
// the same time on different SMs, so each corpus tile is read from HBM about
// once and served to the other query blocks from L2.
//
// Top-k state per (query, half): for k <= 32 a sorted list in registers
// (KREG = 16 or 32 slots).  A 32-column chunk whose maximum beats no lane's
// threshold costs one max-reduction; otherwise the chunk is staged in shared
// memory and every lane inserts its candidates in one converged loop, so the
// warp pays for the largest candidate count of a lane, not for the sum over
// lanes.  For k > 32 a 16-entry candidate buffer per thread in shared memory
// is sorted and merged into a sorted list in global scratch whenever a
// buffer fills.  Each unit writes its k best per (query, half); K7 merges the
// sorted lists of each query: one warp per query takes the largest head of
// its lists k times (packed (score, index) keys).
#include <float.h>

#include <algorithm>

#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int BM = 128;               // queries per tile: UMMA M = TMEM lanes
constexpr int BN = 256;               // corpus rows per tile: UMMA N
constexpr int BK = 64;                // K per stage: one 128-byte swizzle row
constexpr int UK = 16;                // K per tcgen05.mma, kind::f16
constexpr int kEpiWarps = 8;
constexpr int kEpi = kEpiWarps * 32;  // epilogue threads
constexpr int kThreads = 64 + kEpi;
constexpr int kHalfCols = BN / 2;     // columns per epilogue thread per tile
constexpr uint32_t kABytes = BM * BK * 2;
constexpr uint32_t kBBytes = BN * BK * 2;
constexpr uint32_t kTmemCols = 2 * BN;
constexpr int kCap = 16;              // candidate buffer per thread (large-k path)
constexpr int kMergeMax = 16384;      // bound on lists * k per query (the merge's candidates)
constexpr size_t kBarBytes = 256;
constexpr size_t kEpiSmem = (size_t)kEpi * 32 * 4;  // 32 KB: staging or candidate buffer
static_assert((size_t)kCap * kEpi * 8 == kEpiSmem, "candidate buffer size");
// Shared-memory ring per CTA.  Single CTA: a 128-row query tile and the
// whole 256-row corpus tile per stage, 4 stages.  CTA pair (cta_group::2):
// each CTA stages its own query tile and its 128-row half of the corpus
// tile, so a stage is 32 KB and 6 fit.
template <int CL>
struct Ring {
  static constexpr int stages = CL == 2 ? 6 : 4;
  static constexpr uint32_t b_bytes = kBBytes / CL;
  static constexpr uint32_t stage_bytes = kABytes + b_bytes;
  static constexpr size_t smem = 1024 + (size_t)stages * stage_bytes + kBarBytes + kEpiSmem;
};
static_assert(Ring<1>::smem <= 232448 && Ring<2>::smem <= 232448, "shared memory per CTA");
static_assert(8 * (2 * Ring<2>::stages + 4) + 8 + 8 <= kBarBytes, "barrier area");

struct Params {
  int64_t Qmax, N, tiles;
  const int32_t* count_dev;  // queries to process: min(*count_dev, Qmax); NULL: Qmax
  int32_t k, kb_count;
  int32_t slots;             // concurrent unit executors the plan targets (CTAs / cl)
  int32_t cl;                // CTAs per cluster: 1, or 2 forming a CTA pair (M = 256 MMA)
  float* part_s;     // [Q][2 * nsplit][k]: one list per (split, column half)
  int32_t* part_i;
  float* list_s;     // large-k: [grid][kEpi][2][k]
  int32_t* list_i;
  unsigned* err;
  // Optional per-query score floor (large-k path): query q only keeps scores
  // >= floor[q * floor_stride + floor_index].  A floor never exceeds the
  // query's final k-th best score, so it prunes without changing the result.
  const float* floor;
  int32_t floor_stride, floor_index;
  // k <= 32: per-query shared floor, the largest k-th best score any list of
  // the query has reached so far (order-preserving uint32 code of the float,
  // 0 = none), raised with atomicMax and read once per tile by every list of
  // the query.  Zeroed before each launch.
  uint32_t* qfloor;
  // Optional, one word per query block: a unit whose query blocks are all 0
  // here is skipped (the exact large-k pass re-runs only the flagged blocks).
  const uint32_t* only;
  // Bounded waits of retrieve_kernel: give up after wait_limit_ns.  With
  // withhold_first set (a test hook) every CTA skips the loads of its first
  // stage, so that stage never fills and the waits run out.
  uint64_t wait_limit_ns;
  int32_t withhold_first;
};

// Rows the merge writes: with inv NULL one per query (row q = query q);
// otherwise n_out rows, row o holding the results of query inv[o] — the
// fan-out of each merged query's results to every row merged into it.
struct OutRows {
  const int32_t* inv;
  int64_t n_out;
};

__device__ __forceinline__ uint32_t float_code(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float code_float(uint32_t c) {
  return __uint_as_float((c & 0x80000000u) ? (c ^ 0x80000000u) : ~c);
}

__host__ __device__ inline int64_t gcd64(int64_t a, int64_t b) {
  while (b) {
    const int64_t t = a % b;
    a = b;
    b = t;
  }
  return a;
}

// Largest split count a plan may use: every split needs a corpus tile, and
// the merge sorts 2 * nsplit * k candidates per query.
__host__ __device__ inline int64_t max_splits(int64_t sms, int64_t tiles, int32_t k) {
  int64_t ns = sms;
  if (ns > tiles) ns = tiles;
  if (ns > kMergeMax / (2 * k)) ns = kMergeMax / (2 * k);
  return ns < 1 ? 1 : ns;
}

// Work decomposition for Q queries: query blocks of 128, grouped by cl (the
// CTAs of a cluster take adjacent query blocks over the same corpus tiles),
// and corpus splits; units = groups * nsplit is a multiple of the number of
// unit executors (slots) when the caps allow.  Host and device evaluate the
// same function, so a launch can take its query count from device memory.
struct SplitPlan {
  int32_t qblocks, groups, nsplit;
};
__host__ __device__ inline SplitPlan split_plan(int64_t Q, int64_t tiles, int32_t k,
                                                int64_t slots, int32_t cl) {
  SplitPlan sp;
  sp.qblocks = (int32_t)((Q + BM - 1) / BM);
  sp.groups = (sp.qblocks + cl - 1) / cl;
  int64_t ns = slots / gcd64(slots, sp.groups > 0 ? sp.groups : 1);
  const int64_t cap = max_splits(slots, tiles, k);
  if (ns > cap) ns = cap;
  sp.nsplit = (int32_t)ns;
  return sp;
}

__device__ __forceinline__ int64_t query_count(const Params& p) {
  if (!p.count_dev) return p.Qmax;
  const int64_t c = *p.count_dev;
  return c < 0 ? 0 : (c > p.Qmax ? p.Qmax : c);
}

__device__ __forceinline__ void unit_coords(const SplitPlan& sp, int64_t tiles, int64_t u,
                                            int rank, int cl, int& qb, int& split, int64_t& t0,
                                            int64_t& t1) {
  qb = (int)(u % sp.groups) * cl + rank;
  split = (int)(u / sp.groups);
  t0 = (int64_t)split * tiles / sp.nsplit;
  t1 = (int64_t)(split + 1) * tiles / sp.nsplit;
}

// True when `only` is set and no query block of unit u's group is flagged.
// Every role of a CTA pair evaluates it for the same units, so all skip alike.
__device__ __forceinline__ bool unit_skipped(const Params& p, const SplitPlan& sp, int64_t u,
                                             int cl) {
  if (!p.only) return false;
  const int g = (int)(u % sp.groups);
  for (int r = 0; r < cl; ++r) {
    const int qb = g * cl + r;
    if (qb < sp.qblocks && p.only[qb] != 0u) return false;
  }
  return true;
}

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Maximum of 32 scores as a tree of three-input maxima (17 operations; the
// maximum is exact, so the order does not change the result).
__device__ __forceinline__ float chunk_max(const uint32_t (&r)[32]) {
  float m[11];
#pragma unroll
  for (int j = 0; j < 10; ++j)
    m[j] = max3f(__uint_as_float(r[3 * j]), __uint_as_float(r[3 * j + 1]),
                 __uint_as_float(r[3 * j + 2]));
  m[10] = fmaxf(__uint_as_float(r[30]), __uint_as_float(r[31]));
  const float a = max3f(m[0], m[1], m[2]), b = max3f(m[3], m[4], m[5]);
  const float c = max3f(m[6], m[7], m[8]), e = fmaxf(m[9], m[10]);
  return fmaxf(max3f(a, b, c), e);
}

// Insert (s, idx) into a list sorted by score descending.  idx is larger than
// every index already present, so on equal scores it goes after them.
template <int KREG>
__device__ __forceinline__ void list_insert(float (&ls)[KREG], int32_t (&li)[KREG], float s,
                                            int32_t idx) {
#pragma unroll
  for (int i = KREG - 1; i > 0; --i) {
    const bool up = s > ls[i - 1];
    const bool here = !up && s > ls[i];
    ls[i] = up ? ls[i - 1] : (here ? s : ls[i]);
    li[i] = up ? li[i - 1] : (here ? idx : li[i]);
  }
  if (s > ls[0]) {
    ls[0] = s;
    li[0] = idx;
  }
}

// ---- large-k helpers (per thread, serial) ---------------------------------------------
__device__ void flush_candidates(float* cs, int32_t* ci, int et, int& cnt, float* Ls, int32_t* Li,
                                 int k, int& cur, float& theta, float floor_theta, float& kth) {
  if (cnt == 0) return;
  // Stable insertion sort of the buffer, score descending (buffer order is
  // ascending corpus index, so ties keep the lower index first).
  for (int a = 1; a < cnt; ++a) {
    const float s = cs[a * kEpi + et];
    const int32_t i = ci[a * kEpi + et];
    int b = a - 1;
    while (b >= 0 && s > cs[b * kEpi + et]) {
      cs[(b + 1) * kEpi + et] = cs[b * kEpi + et];
      ci[(b + 1) * kEpi + et] = ci[b * kEpi + et];
      --b;
    }
    cs[(b + 1) * kEpi + et] = s;
    ci[(b + 1) * kEpi + et] = i;
  }
  // Merge with the current list (all of whose entries have lower corpus
  // indices: on equal scores the list entry wins).  The list is consumed in
  // order, so its addresses are known ahead of the comparisons: it is read in
  // windows of 8 with the next window in flight, not one dependent load at a
  // time.
  constexpr int Wn = 8;
  const float* As = Ls + (size_t)cur * k;
  const int32_t* Ai = Li + (size_t)cur * k;
  float* Os = Ls + (size_t)(cur ^ 1) * k;
  int32_t* Oi = Li + (size_t)(cur ^ 1) * k;
  float wa[Wn];
  int32_t wi[Wn];
#pragma unroll
  for (int e = 0; e < Wn; ++e) {
    wa[e] = e < k ? As[e] : -FLT_MAX;
    wi[e] = e < k ? Ai[e] : -1;
  }
  int b = 0, o = 0;
  float sb = cs[et];
  int32_t ib = ci[et];
  float last = -FLT_MAX;
  for (int a0 = 0; a0 < k && o < k; a0 += Wn) {
    float na[Wn];
    int32_t ni[Wn];
    const bool more = a0 + Wn < k;
    if (more) {
#pragma unroll
      for (int e = 0; e < Wn; ++e) {
        const bool in = a0 + Wn + e < k;
        na[e] = in ? As[a0 + Wn + e] : -FLT_MAX;
        ni[e] = in ? Ai[a0 + Wn + e] : -1;
      }
    }
#pragma unroll
    for (int e = 0; e < Wn; ++e) {
      while (b < cnt && o < k && sb > wa[e]) {
        Os[o] = sb;
        Oi[o] = ib;
        last = sb;
        ++o;
        ++b;
        if (b < cnt) {
          sb = cs[b * kEpi + et];
          ib = ci[b * kEpi + et];
        }
      }
      if (o < k && a0 + e < k) {
        Os[o] = wa[e];
        Oi[o] = wi[e];
        last = wa[e];
        ++o;
      }
    }
    if (more) {
#pragma unroll
      for (int e = 0; e < Wn; ++e) {
        wa[e] = na[e];
        wi[e] = ni[e];
      }
    }
  }
  cur ^= 1;
  kth = last;                        // the k-th entry of the new list (-FLT_MAX if not full)
  theta = fmaxf(last, floor_theta);  // ... not below the floor
  cnt = 0;
}

template <int KREG, int CL>
__global__ void __launch_bounds__(kThreads, 1)
    retrieve_kernel(const __grid_constant__ CUtensorMap tmap_q,
                    const __grid_constant__ CUtensorMap tmap_c, const Params p) {
  constexpr int kStages = Ring<CL>::stages;
  constexpr uint32_t kBLocal = Ring<CL>::b_bytes;
  constexpr uint32_t kStageBytes = Ring<CL>::stage_bytes;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * kABytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + kStages;
  uint64_t* tfull = bars + 2 * kStages;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint64_t* drain = tempty + 3;          // after tmem_slot and abort_flag: the MMA drain
  uint8_t* epi_smem = smem + kStages * kStageBytes + kBarBytes;
  const uint64_t lim = p.wait_limit_ns ? p.wait_limit_ns : kWaitLimitNs;

  // CTA pair: the even CTA (rank 0) owns the full and tempty barriers that
  // both CTAs' loads and epilogues signal, and issues every MMA.
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull + a, 1);
      mbar_init(tempty + a, kEpiWarps * CL);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tmap_q);
    prefetch_tmap(&tmap_c);
  }
  if (warp == 1) {
    if (CL == 2) {
      tmem_alloc_pair(tmem_slot, kTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(tmem_slot, kTmemCols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (CL > 1) cluster_sync();            // the pair's barriers exist before any remote signal
  const uint32_t tmem_base = *tmem_slot;
  const int rank = CL > 1 ? (int)cluster_ctarank() : 0;
  // Everything above touched only shared memory, TMEM and the kernel
  // parameters; global memory (the query count, queries, corpus) waits for
  // the previous kernel on the stream.
  pdl_wait();
  pdl_trigger();
  const int64_t Q = query_count(p);
  const SplitPlan sp = split_plan(Q, p.tiles, p.k, p.slots, CL);
  const int64_t units = Q > 0 ? (int64_t)sp.groups * sp.nsplit : 0;
  const int64_t u0 = blockIdx.x / CL, ustep = gridDim.x / CL;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      const uint64_t pol_c = policy_evict_first();
      const uint64_t pol_q = policy_evict_last();
      uint32_t stage = 0, phase = 0;
      int64_t issued = 0;                 // stages armed (or withheld) so far
      for (int64_t u = u0; u < units; u += ustep) {
        if (unit_skipped(p, sp, u, CL)) continue;
        int qb, split;
        int64_t t0, t1;
        unit_coords(sp, p.tiles, u, rank, CL, qb, split, t0, t1);
        for (int64_t t = t0; t < t1; ++t) {
          for (int kb = 0; kb < p.kb_count; ++kb) {
            if (!mbar_wait_limit(empty + stage, phase ^ 1u, abort_flag, lim)) goto producer_done;
            if (p.withhold_first && issued == 0) {   // test hook: this stage never fills
              ++issued;
              if (++stage == kStages) {
                stage = 0;
                phase ^= 1u;
              }
              continue;
            }
            ++issued;
            // A query block past the last addressable row is loaded from
            // row 0 instead: its scores are masked, and no box lies wholly
            // outside the tensor.
            const int32_t qy = (int64_t)qb * BM < p.Qmax ? qb * BM : 0;
            if (CL == 1) {
              mbar_arrive_expect_tx(full + stage, kStageBytes);
              tma_load_2d_hint(sA + stage * kABytes, &tmap_q, full + stage, kb * BK, qy, pol_q);
              tma_load_2d_hint(sB + stage * kBLocal, &tmap_c, full + stage, kb * BK,
                               (int32_t)(t * BN), pol_c);
            } else {
              // Both CTAs' bytes complete on the even CTA's full barrier,
              // armed there for the pair.  A corpus half past the last row
              // re-reads the tile's first half (masked).
              if (rank == 0) mbar_arrive_expect_tx(full + stage, 2 * kStageBytes);
              const uint32_t bar = cluster_smem_addr(full + stage, 0);
              const int64_t cy = t * BN + rank * (BN / CL);
              tma_load_2d_pair_hint(sA + stage * kABytes, &tmap_q, bar, kb * BK, qy, pol_q);
              tma_load_2d_pair_hint(sB + stage * kBLocal, &tmap_c, bar, kb * BK,
                                    (int32_t)(cy < p.N ? cy : t * BN), pol_c);
            }
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
    producer_done:
      // Before it leaves, the even CTA (whose full barriers count both CTAs'
      // bytes) waits, bounded, for every stage it armed that may still be in
      // flight, so no copy lands in shared memory after the CTAs exit, even
      // when some role gave up.  In a normal run these phases have completed
      // or complete within the last tile.
      if (rank == 0) {
        volatile int keep_going = 0;
        for (int64_t i = issued > kStages ? issued - kStages : 0; i < issued; ++i) {
          if (p.withhold_first && i == 0) continue;           // never armed
          if (!mbar_wait_limit(full + (int)(i % kStages), (uint32_t)((i / kStages) & 1),
                               &keep_going, lim))
            break;
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM * CL, BN);
      uint32_t stage = 0, phase = 0, tile_i = 0;
      bool any_mma = false;
      for (int64_t u = u0; u < units; u += ustep) {
        if (unit_skipped(p, sp, u, CL)) continue;
        int qb, split;
        int64_t t0, t1;
        unit_coords(sp, p.tiles, u, rank, CL, qb, split, t0, t1);
        for (int64_t t = t0; t < t1; ++t, ++tile_i) {
          const uint32_t acc = tile_i & 1u, aphase = (tile_i >> 1) & 1u;
          if (!mbar_wait_limit(tempty + acc, aphase ^ 1u, abort_flag, lim)) goto mma_done;
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + acc * BN;
          for (int kb = 0; kb < p.kb_count; ++kb) {
            if (!mbar_wait_limit(full + stage, phase, abort_flag, lim)) goto mma_done;
            tc_fence_after();
            any_mma = true;
            const uint64_t a0 = smem_desc_k_sw128(smem_u32(sA + stage * kABytes));
            const uint64_t b0 = smem_desc_k_sw128(smem_u32(sB + stage * kBLocal));
#pragma unroll
            for (int kk = 0; kk < BK / UK; ++kk) {
              const uint64_t koff = (uint64_t)(kk * UK * 2 / 16);
              if (CL == 1)
                umma_bf16(d_tmem, a0 + koff, b0 + koff, idesc, (kb | kk) != 0 ? 1u : 0u);
              else
                umma_bf16_pair(d_tmem, a0 + koff, b0 + koff, idesc, (kb | kk) != 0 ? 1u : 0u);
            }
            if (CL == 1)
              umma_commit(empty + stage);
            else
              umma_commit_pair_mc(empty + stage, 0x3);
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (CL == 1)
            umma_commit(tfull + acc);
          else
            umma_commit_pair_mc(tfull + acc, 0x3);
        }
      }
    mma_done:
      // Every MMA this thread issued completes before the teardown frees
      // tensor memory, even when some role gave up (one commit to the drain
      // barrier; in a normal run the last tile's MMAs are all it waits for).
      if (any_mma) {
        if (CL == 1)
          umma_commit(drain);
        else
          umma_commit_pair_mc(drain, 0x1);
        volatile int keep_going = 0;
        mbar_wait_limit(drain, 0u, &keep_going, lim);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - 2;                  // 0..7
    const int quarter = warp & 3;             // TMEM lanes [32*quarter, 32*quarter+32)
    const int half = ew >> 2;                 // columns [half*128, half*128+128) of a tile
    const int row = quarter * 32 + lane;      // query within the block
    const int et = ew * 32 + lane;            // epilogue thread index, 0..255
    const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
    const int k = p.k;
    const int lists = 2 * sp.nsplit;
    uint32_t tile_i = 0;
    float* stage_f = reinterpret_cast<float*>(epi_smem);            // KREG: [8][kEpi][4]
    float* cand_s = reinterpret_cast<float*>(epi_smem);             // large k: [kCap][kEpi]
    int32_t* cand_i = reinterpret_cast<int32_t*>(epi_smem + (size_t)kCap * kEpi * 4);
    float* Ls = p.list_s + ((size_t)blockIdx.x * kEpi + et) * 2 * (size_t)k;
    int32_t* Li = p.list_i + ((size_t)blockIdx.x * kEpi + et) * 2 * (size_t)k;
    for (int64_t u = u0; u < units; u += ustep) {
      if (unit_skipped(p, sp, u, CL)) continue;
      int qb, split;
      int64_t t0, t1;
      unit_coords(sp, p.tiles, u, rank, CL, qb, split, t0, t1);
      const int64_t q = (int64_t)qb * BM + row;
      const bool valid_q = q < Q;
      const bool warp_has_query = __any_sync(0xffffffffu, valid_q);
      // Large k: start from the query's floor (a lower bound on its final k-th
      // best score), so only scores that can still make the top k are kept.
      float floor_theta = -FLT_MAX;
      if (KREG == 0 && p.floor && valid_q) {
        const float f = p.floor[(size_t)q * p.floor_stride + p.floor_index];
        if (f > -FLT_MAX) floor_theta = nextafterf(f, -INFINITY);  // keep s >= f
      }
      float theta = floor_theta;
      // Register list (k <= 32): KREG slots sorted descending, the first
      // KREG - k holding +FLT_MAX sentinels that never move, so the last
      // slot is always the k-th best score seen: the list's own threshold.
      float ls[KREG > 0 ? KREG : 1];
      int32_t li[KREG > 0 ? KREG : 1];
      int cnt = 0, cur = 0;
#pragma unroll
      for (int i = 0; i < (KREG > 0 ? KREG : 1); ++i) {
        ls[i] = (KREG > 0 && i < KREG - k) ? FLT_MAX : -FLT_MAX;
        li[i] = -1;
      }
      // The query's shared floor, as a threshold that keeps ties with it
      // (another list may hold an equal score at a higher index).
      uint32_t qf_seen = 0;
      float qf_theta = -FLT_MAX;
      float list_kth = -FLT_MAX;               // large k: this list's k-th best so far
      if (valid_q && p.qfloor) {               // lists of other splits may have set it
        qf_seen = *reinterpret_cast<volatile uint32_t*>(p.qfloor + q);
        if (qf_seen) qf_theta = nextafterf(code_float(qf_seen), -INFINITY);
      }
      if (KREG == 0 && valid_q) {
        for (int i = 0; i < k; ++i) {
          Ls[i] = -FLT_MAX;
          Li[i] = -1;
        }
      }
      for (int64_t t = t0; t < t1; ++t, ++tile_i) {
        const uint32_t acc = tile_i & 1u, aphase = (tile_i >> 1) & 1u;
        if (!mbar_wait_limit(tfull + acc, aphase, abort_flag, lim)) goto epi_done;
        tc_fence_after();
        theta = fmaxf(theta, qf_theta);
        const int64_t col0 = t * BN + half * kHalfCols;
        const bool tail = col0 + kHalfCols > p.N;
        // Register lists: the candidates of the staged chunk (if any) of every
        // lane, inserted in one converged loop (the warp pays for the largest
        // candidate count of a lane); thresholds are re-read per insert.
        bool pending = false;
        int32_t pending_base = 0;
        auto drain = [&]() {
          uint32_t m = 0;
          if (pending) {
#pragma unroll
            for (int v = 0; v < 8; ++v) {
              const uint4 x = reinterpret_cast<const uint4*>(stage_f)[v * kEpi + et];
              m |= (__uint_as_float(x.x) > theta ? 1u : 0u) << (4 * v);
              m |= (__uint_as_float(x.y) > theta ? 1u : 0u) << (4 * v + 1);
              m |= (__uint_as_float(x.z) > theta ? 1u : 0u) << (4 * v + 2);
              m |= (__uint_as_float(x.w) > theta ? 1u : 0u) << (4 * v + 3);
            }
          }
          const int most = __reduce_max_sync(0xffffffffu, (unsigned)__popc(m));
          for (int it = 0; it < most; ++it) {
            const int j = m ? __ffs(m) - 1 : 0;
            const float sc = m ? stage_f[((j >> 2) * kEpi + et) * 4 + (j & 3)] : -FLT_MAX;
            m &= m - 1;
            if (sc > theta) {
              list_insert<(KREG > 0 ? KREG : 1)>(ls, li, sc, pending_base + j);
              theta = fmaxf(ls[(KREG > 0 ? KREG : 1) - 1], qf_theta);
            }
          }
          pending = false;
          __syncwarp();
        };
        // One 32-column chunk: mask columns past N, then the threshold test
        // and candidate handling.
        auto do_chunk = [&](uint32_t(&r)[32], int c) {
          const int32_t cbase = (int32_t)(col0 + c * 32);
          if (tail) {                           // zero-filled rows past N never qualify
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if ((int64_t)cbase + j >= p.N) r[j] = __float_as_uint(-FLT_MAX);
          }
          if (KREG > 0) {
            // A chunk with a candidate is staged in the lane's slot; drain()
            // inserts the staged candidates of all lanes in one converged
            // loop.  Long lists (32 slots, costly inserts) defer it to the end
            // of the tile, so the lanes' candidates of several chunks share
            // one pass (a lane whose slot is taken drains first); short lists
            // drain at once.
            const float mx = chunk_max(r);
            const bool any = valid_q && mx > theta;   // padding query rows never insert
            if (KREG >= 32) {
              if (__any_sync(0xffffffffu, any && pending)) drain();
              if (any) {
#pragma unroll
                for (int v = 0; v < 8; ++v)
                  reinterpret_cast<uint4*>(stage_f)[v * kEpi + et] =
                      make_uint4(r[4 * v], r[4 * v + 1], r[4 * v + 2], r[4 * v + 3]);
                pending = true;
                pending_base = cbase;
              }
            } else if (__any_sync(0xffffffffu, any)) {
              // Short lists: this chunk's candidates at once, the mask built
              // from the registers.
              uint32_t m = 0;
              if (any) {
#pragma unroll
                for (int j = 0; j < 32; ++j) m |= (__uint_as_float(r[j]) > theta ? 1u : 0u) << j;
#pragma unroll
                for (int v = 0; v < 8; ++v)
                  reinterpret_cast<uint4*>(stage_f)[v * kEpi + et] =
                      make_uint4(r[4 * v], r[4 * v + 1], r[4 * v + 2], r[4 * v + 3]);
              }
              const int most = __reduce_max_sync(0xffffffffu, (unsigned)__popc(m));
              for (int it = 0; it < most; ++it) {
                const int j = m ? __ffs(m) - 1 : 0;
                const float sc = m ? stage_f[((j >> 2) * kEpi + et) * 4 + (j & 3)] : -FLT_MAX;
                m &= m - 1;
                if (sc > theta) {
                  list_insert<(KREG > 0 ? KREG : 1)>(ls, li, sc, cbase + j);
                  theta = fmaxf(ls[(KREG > 0 ? KREG : 1) - 1], qf_theta);
                }
              }
              __syncwarp();
            }
          } else {
            // Same first test as above: a chunk whose maximum beats no
            // lane's threshold costs one max-reduction and a vote.
            const float mx = chunk_max(r);
            if (__any_sync(0xffffffffu, valid_q && mx > theta)) {
#pragma unroll
              for (int j0 = 0; j0 < 32; j0 += 4) {
#pragma unroll
                for (int j = j0; j < j0 + 4; ++j) {
                  const float s = __uint_as_float(r[j]);
                  if (valid_q && s > theta) {
                    cand_s[cnt * kEpi + et] = s;
                    cand_i[cnt * kEpi + et] = cbase + j;
                    ++cnt;
                  }
                }
                if (__any_sync(0xffffffffu, cnt > kCap - 4))
                  flush_candidates(cand_s, cand_i, et, cnt, Ls, Li, k, cur, theta,
                                   fmaxf(floor_theta, qf_theta), list_kth);
              }
            }
          }
                };
        // Lists of up to 16 slots: two chunks per TMEM round trip (both loads,
        // one wait).  Longer lists and large k keep one: they need the
        // registers.
        // A warp whose 32 query rows are all padding has nothing to read.
#pragma unroll 1
        for (int c = 0; c < kHalfCols / 32 && warp_has_query; c += (KREG > 0 && KREG < 32 ? 2 : 1)) {
          const uint32_t ta = tmem_base + lane_addr + acc * BN + half * kHalfCols + c * 32;
          uint32_t ra[32];
          if (KREG > 0 && KREG < 32) {
            uint32_t rb[32];
            tmem_ld_32x32b_x32(ta, ra);
            tmem_ld_32x32b_x32(ta + 32, rb);
            tmem_ld_wait();
            do_chunk(ra, c);
            do_chunk(rb, c + 1);
          } else {
            tmem_ld_32x32b_x32(ta, ra);
            tmem_ld_wait();
            do_chunk(ra, c);
          }
        }
        if (KREG >= 32 && __any_sync(0xffffffffu, pending)) drain();
        tc_fence_before();
        __syncwarp();
        if (valid_q && p.qfloor) {
          // Publish this list's k-th best if it raises the query's floor,
          // and fetch the floor for the next tile.
          const float kth = KREG > 0 ? ls[(KREG > 0 ? KREG : 1) - 1] : list_kth;
          const uint32_t mine = kth > -FLT_MAX ? float_code(kth) : 0u;
          if (mine > qf_seen) atomicMax(p.qfloor + q, mine);
          const uint32_t c = *reinterpret_cast<volatile uint32_t*>(p.qfloor + q);
          if (c > qf_seen) {
            qf_seen = c;
            qf_theta = nextafterf(code_float(c), -INFINITY);  // keep s >= floor
          }
        }
        if (lane == 0) {
          if (CL == 1)
            mbar_arrive(tempty + acc);
          else
            mbar_arrive_cluster(cluster_smem_addr(tempty + acc, 0));
        }
      }
      if (valid_q) {
        const size_t o = ((size_t)q * lists + 2 * split + half) * k;
        float* os = p.part_s + o;
        int32_t* oi = p.part_i + o;
        if (KREG > 0) {
#pragma unroll
          for (int i = 0; i < (KREG > 0 ? KREG : 1); ++i)
            if (i >= KREG - k) {
              os[i - (KREG - k)] = ls[i];
              oi[i - (KREG - k)] = li[i];
            }
        } else {
          flush_candidates(cand_s, cand_i, et, cnt, Ls, Li, k, cur, theta,
                           fmaxf(floor_theta, qf_theta), list_kth);
          for (int i = 0; i < k; ++i) {
            os[i] = Ls[(size_t)cur * k + i];
            oi[i] = Li[(size_t)cur * k + i];
          }
        }
      }
    }
  epi_done:;
  }

  tc_fence_before();
  __syncthreads();
  if (CL > 1) cluster_sync();            // the pair's MMAs and remote signals are done
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    if (CL == 2)
      tmem_dealloc_pair(tmem_base, kTmemCols);
    else
      tmem_dealloc(tmem_base, kTmemCols);
  }
  if (CL > 1) cluster_sync();            // no CTA leaves while its peer may still signal it
  if (threadIdx.x == 0 && *abort_flag) set_error(p.err, kErrTimeout);
}

// ---- K7: merge of the per-split lists ----------------------------------------------------
__device__ __forceinline__ uint64_t pack_key(float s, int32_t idx) {
  uint32_t u = __float_as_uint(s);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((uint64_t)u << 32) | (uint64_t)(0xffffffffu - (uint32_t)idx);
}

__device__ __forceinline__ void unpack_key(uint64_t key, float& s, int32_t& idx) {
  uint32_t u = (uint32_t)(key >> 32);
  u = (u & 0x80000000u) ? (u ^ 0x80000000u) : ~u;
  s = __uint_as_float(u);
  idx = (int32_t)(0xffffffffu - (uint32_t)key);
}

// One warp per query runs a tournament over the sorted lists.
// Lane l owns lists l, l+32, ...; it keeps each list's head and the entry
// after it (prefetched) in registers.  Each round the warp takes the largest
// head (keys are unique: a corpus row lives in exactly one list; padding
// keys tie, and the lowest such lane advances), so kout rounds give the kout
// best in order.
constexpr int kMaxListsPerLane = 10;

// Any kout: picks 0..31 are kept one per lane and written together when
// kout <= 32; for larger kout each pick is written as it is made.  With
// out_i NULL only the kout-th pick's score is written, to out_s[o] (the
// floor of the second large-k pass).  With `only` set, rows whose query
// block is not flagged there are skipped.  With `flag_out` set, a query's
// block is flagged when one of its lists may have cut off a member of the
// top kout: a full list whose last (k-th) entry is not below the union's
// kout-th pick.  A list whose last entry is below it holds every row of its
// range that can be in the top kout, so with no list flagged the union's
// first kout entries are exact.  LPL lists per lane at most (the
// launch's bound on 2 * nsplit / 32, rounded up); slots past the query's
// list count are skipped warp-uniformly, so the per-round work and the
// registers follow the lists a launch can have, not the largest count.
template <int LPL>
__global__ void __launch_bounds__(256) merge_warp_kernel(const Params p, float* __restrict__ out_s,
                                                         int32_t* __restrict__ out_i,
                                                         int32_t kout, OutRows rows,
                                                         uint32_t* flag_out, const uint32_t* only) {
  pdl_wait();
  pdl_trigger();
  const int64_t Q = query_count(p);
  const SplitPlan sp = split_plan(Q, p.tiles, p.k, p.slots, p.cl);
  const int k = p.k;
  const int lists = 2 * sp.nsplit;
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t R = rows.inv ? rows.n_out : Q;
  for (int64_t o = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; o < R; o += nwarps) {
    const int64_t q = rows.inv ? (int64_t)__ldg(rows.inv + o) : o;
    if (q < 0 || q >= Q) {                         // warp-uniform
      if (lane == 0) set_error(p.err, kErrInvalidArg);
      continue;
    }
    if (only && only[q / BM] == 0u) continue;      // warp-uniform
    const float* __restrict__ ps = p.part_s + (size_t)q * lists * k;
    const int32_t* __restrict__ pi = p.part_i + (size_t)q * lists * k;
    uint64_t head[LPL], next[LPL];
    int pos[LPL];
#pragma unroll
    for (int j = 0; j < LPL; ++j) {
      const int l = j * 32 + lane;
      pos[j] = 0;
      head[j] = next[j] = 0ull;
      if (j * 32 < lists) {                        // warp-uniform
        if (l < lists) head[j] = pack_key(ps[(size_t)l * k], pi[(size_t)l * k]);
        if (l < lists && k > 1) next[j] = pack_key(ps[(size_t)l * k + 1], pi[(size_t)l * k + 1]);
      }
    }
    float my_s = -FLT_MAX;
    int32_t my_i = -1;
    uint64_t last = 0ull;                          // key of the latest pick
    for (int r = 0; r < kout; ++r) {
      uint64_t best = 0ull;
      int bj = 0;
#pragma unroll
      for (int j = 0; j < LPL; ++j)
        if (j * 32 < lists && head[j] > best) {    // the first test is warp-uniform
          best = head[j];
          bj = j;
        }
      // Warp maximum of the 64-bit keys: the largest high word, then the
      // largest low word among the lanes holding it (two warp reductions).
      const uint32_t bhi = (uint32_t)(best >> 32), blo = (uint32_t)best;
      const uint32_t mhi = __reduce_max_sync(0xffffffffu, bhi);
      const uint32_t mlo = __reduce_max_sync(0xffffffffu, bhi == mhi ? blo : 0u);
      const uint64_t mx = ((uint64_t)mhi << 32) | mlo;
      const unsigned win = __ballot_sync(0xffffffffu, best == mx && mx != 0ull);
      last = mx;
      if (kout <= 32) {
        if (lane == r && mx != 0ull) unpack_key(mx, my_s, my_i);
      } else if (out_i && lane == 0) {
        float sc = -FLT_MAX;
        int32_t id = -1;
        if (mx != 0ull) unpack_key(mx, sc, id);
        out_s[(size_t)o * kout + r] = sc;
        out_i[(size_t)o * kout + r] = id;
      }
      if (win != 0u && lane == __ffs(win) - 1) {
#pragma unroll
        for (int j = 0; j < LPL; ++j)
          if (j == bj) {
            const int l = j * 32 + lane;
            ++pos[j];
            head[j] = next[j];
            next[j] = pos[j] + 1 < k ? pack_key(ps[(size_t)l * k + pos[j] + 1],
                                                pi[(size_t)l * k + pos[j] + 1])
                                     : 0ull;
          }
      }
    }
    if (out_i && kout <= 32 && lane < kout) {
      out_s[(size_t)o * kout + lane] = my_s;
      out_i[(size_t)o * kout + lane] = my_i;
    }
    if (!out_i && lane == 0) {
      float sc = -FLT_MAX;
      int32_t id = -1;
      if (last != 0ull) unpack_key(last, sc, id);
      out_s[o] = sc;
    }
    if (flag_out) {
      bool cut = false;
#pragma unroll
      for (int j = 0; j < LPL; ++j) {
        const int l = j * 32 + lane;
        if (l < lists)
          cut |= pack_key(ps[(size_t)l * k + k - 1], pi[(size_t)l * k + k - 1]) >= last;
      }
      if (__any_sync(0xffffffffu, cut) && lane == 0) atomicOr(flag_out + q / BM, 1u);
    }
  }
}

// ---- K6s: small batches (at most 16 queries) -------------------------------------------
// With few queries the query block of the main kernel is mostly padding and
// is re-streamed with every corpus stage.  Here the roles are swapped: the
// corpus tile is the MMA's M operand (128 rows) and the queries, padded to
// 16, are its N operand, loaded once and kept in shared memory.  The ring
// then carries only corpus boxes (10 stages of 16 KB), which is what an
// HBM-bound pass needs.  TMEM holds four 128 x 16 fp32 accumulators.
//
// Epilogue (warps 2-5, one per TMEM lane quarter): thread = corpus row of the
// tile, holding its 16 scores.  A score above its query's threshold is
// appended to that query's candidate buffer in shared memory; after each
// tile a warp merges each non-empty buffer with the query's sorted top-k list
// (k rounds of a warp-wide maximum over packed (score, ~row) keys) and resets
// the threshold to the new k-th best.  Each CTA covers a contiguous range of
// 128-row tiles and writes one sorted list per query, in the layout of the
// main kernel's lists, so the same merge kernel finishes the job.
constexpr int SQ_N = 16;                    // queries per MMA (N)
constexpr int SQ_BM = 128;                  // corpus rows per tile (M)
constexpr int SQ_STAGES = 10;
constexpr int SQ_MAXKB = 16;                // d <= 1024
constexpr int SQ_TBUF = 4;                  // TMEM accumulators
constexpr uint32_t SQ_TMEM_COLS = 64;       // SQ_TBUF * SQ_N
constexpr int SQ_CAP = SQ_BM;               // candidates per query per tile: at most one per row
constexpr int SQ_THREADS = 64 + 128;        // producer, MMA, 4 epilogue warps
constexpr uint32_t SQ_ABYTES = SQ_BM * BK * 2;   // 16 KB
constexpr uint32_t SQ_QBYTES = SQ_N * BK * 2;    // 2 KB per k-block
constexpr size_t SQ_EPI_BYTES = (size_t)SQ_N * (SQ_CAP + 32) * 8 + SQ_N * 8;
constexpr size_t SQ_SMEM = 1024 + (size_t)SQ_MAXKB * SQ_QBYTES + (size_t)SQ_STAGES * SQ_ABYTES +
                           256 + SQ_EPI_BYTES;
static_assert(SQ_SMEM <= 232448, "small-batch kernel shared memory");
static_assert(8 * (2 * SQ_STAGES + 1 + 2 * SQ_TBUF) + 8 + 8 <= 256, "small-batch barrier area");

__global__ void __launch_bounds__(SQ_THREADS, 1)
    retrieve_small_kernel(const __grid_constant__ CUtensorMap tmap_q,
                          const __grid_constant__ CUtensorMap tmap_c, const Params p,
                          int64_t tiles128) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;
  uint8_t* sA = sQ + SQ_MAXKB * SQ_QBYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sA + SQ_STAGES * SQ_ABYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + SQ_STAGES;
  uint64_t* qfull = bars + 2 * SQ_STAGES;
  uint64_t* tfull = qfull + 1;
  uint64_t* tempty = tfull + SQ_TBUF;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + SQ_TBUF);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  uint64_t* drain = tempty + SQ_TBUF + 1;    // after tmem_slot and abort_flag: the MMA drain
  const uint64_t lim = p.wait_limit_ns ? p.wait_limit_ns : kWaitLimitNs;
  uint64_t* lists = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(bars) + 256);  // [16][32]
  uint64_t* cands = lists + SQ_N * 32;                                                    // [16][128]
  float* theta = reinterpret_cast<float*>(cands + SQ_N * SQ_CAP);                          // [16]
  int32_t* cnt = reinterpret_cast<int32_t*>(theta + SQ_N);                                 // [16]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < SQ_STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    mbar_init(qfull, 1);
    for (int b = 0; b < SQ_TBUF; ++b) {
      mbar_init(tfull + b, 1);
      mbar_init(tempty + b, 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tmap_q);
    prefetch_tmap(&tmap_c);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, SQ_TMEM_COLS);
    tmem_relinquish();
  }
  for (int i = threadIdx.x; i < SQ_N * 32; i += SQ_THREADS) lists[i] = 0ull;
  if (threadIdx.x < SQ_N) {
    theta[threadIdx.x] = -FLT_MAX;
    cnt[threadIdx.x] = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();                            // global memory only after the previous kernel
  pdl_trigger();
  const int64_t Q = query_count(p);
  const int k = p.k;
  const int64_t t0 = (int64_t)blockIdx.x * tiles128 / gridDim.x;
  const int64_t t1 = (int64_t)(blockIdx.x + 1) * tiles128 / gridDim.x;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0 && Q > 0) {
      const uint64_t pol_c = policy_evict_first();
      mbar_arrive_expect_tx(qfull, (uint32_t)p.kb_count * SQ_QBYTES);
      for (int kb = 0; kb < p.kb_count; ++kb)
        tma_load_2d(sQ + kb * SQ_QBYTES, &tmap_q, qfull, kb * BK, 0);
      uint32_t stage = 0, phase = 0;
      int64_t issued = 0;                 // corpus stages armed (or withheld) so far
      for (int64_t t = t0; t < t1; ++t) {
        for (int kb = 0; kb < p.kb_count; ++kb) {
          if (!mbar_wait_limit(empty + stage, phase ^ 1u, abort_flag, lim)) goto sq_producer_done;
          if (p.withhold_first && issued == 0) {   // test hook: this stage never fills
            ++issued;
            if (++stage == SQ_STAGES) {
              stage = 0;
              phase ^= 1u;
            }
            continue;
          }
          ++issued;
          mbar_arrive_expect_tx(full + stage, SQ_ABYTES);
          tma_load_2d_hint(sA + stage * SQ_ABYTES, &tmap_c, full + stage, kb * BK,
                           (int32_t)(t * SQ_BM), pol_c);
          if (++stage == SQ_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    sq_producer_done:
      // Before it leaves, the producer waits, bounded, for the query copies
      // and every corpus stage it armed that may still be in flight, so no
      // copy lands in shared memory after the CTA exits, even when some role
      // gave up (in a normal run these phases have completed or complete
      // within the last tile).
      {
        volatile int keep_going = 0;
        mbar_wait_limit(qfull, 0u, &keep_going, lim);
        for (int64_t i = issued > SQ_STAGES ? issued - SQ_STAGES : 0; i < issued; ++i) {
          if (p.withhold_first && i == 0) continue;           // never armed
          if (!mbar_wait_limit(full + (int)(i % SQ_STAGES), (uint32_t)((i / SQ_STAGES) & 1),
                               &keep_going, lim))
            break;
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && Q > 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(SQ_BM, SQ_N);
      uint32_t stage = 0, phase = 0, tile_i = 0;
      bool any_mma = false;
      if (!mbar_wait_limit(qfull, 0u, abort_flag, lim)) goto sq_mma_done;
      tc_fence_after();
      for (int64_t t = t0; t < t1; ++t, ++tile_i) {
        const uint32_t b = tile_i % SQ_TBUF, bphase = (tile_i / SQ_TBUF) & 1u;
        if (!mbar_wait_limit(tempty + b, bphase ^ 1u, abort_flag, lim)) goto sq_mma_done;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + b * SQ_N;
        for (int kb = 0; kb < p.kb_count; ++kb) {
          if (!mbar_wait_limit(full + stage, phase, abort_flag, lim)) goto sq_mma_done;
          tc_fence_after();
          any_mma = true;
          const uint64_t a0 = smem_desc_k_sw128(smem_u32(sA + stage * SQ_ABYTES));
          const uint64_t b0 = smem_desc_k_sw128(smem_u32(sQ + kb * SQ_QBYTES));
#pragma unroll
          for (int kk = 0; kk < BK / UK; ++kk)
            umma_bf16(d_tmem, a0 + (uint64_t)(kk * UK * 2 / 16), b0 + (uint64_t)(kk * UK * 2 / 16),
                      idesc, (kb | kk) != 0 ? 1u : 0u);
          umma_commit(empty + stage);
          if (++stage == SQ_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        umma_commit(tfull + b);
      }
    sq_mma_done:
      // Every MMA this thread issued completes before the teardown frees
      // tensor memory (one commit to the drain barrier).
      if (any_mma) {
        umma_commit(drain);
        volatile int keep_going = 0;
        mbar_wait_limit(drain, 0u, &keep_going, lim);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - 2;                     // 0..3, merges queries q = ew (mod 4)
    const int quarter = warp & 3;                // TMEM lanes [32*quarter, 32*quarter+32)
    const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
    const int nq = (int)(Q < SQ_N ? Q : SQ_N);
    uint32_t tile_i = 0;
    for (int64_t t = t0; t < t1 && nq > 0; ++t, ++tile_i) {
      const uint32_t b = tile_i % SQ_TBUF, bphase = (tile_i / SQ_TBUF) & 1u;
      // On a timeout every later wait fails at once; the named barriers
      // below stay paired because all four warps walk every tile.
      const bool ok = mbar_wait_limit(tfull + b, bphase, abort_flag, lim);
      tc_fence_after();
      uint32_t r[16];
      tmem_ld_32x32b_x16(tmem_base + lane_addr + b * SQ_N, r);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty + b);
      const int64_t row = t * SQ_BM + quarter * 32 + lane;
      if (ok && row < p.N) {
#pragma unroll
        for (int q = 0; q < SQ_N; ++q) {
          const float sc = __uint_as_float(r[q]);
          if (q < nq && sc > theta[q]) {
            const int slot = atomicAdd(cnt + q, 1);
            if (slot < SQ_CAP) cands[q * SQ_CAP + slot] = pack_key(sc, (int32_t)row);
          }
        }
      }
      named_bar_sync(1, 128);
      // Merge: list (k sorted keys) + candidates -> the k best, per query.
      for (int q = ew; q < nq; q += 4) {
        const int c = min(cnt[q], SQ_CAP);
        if (c == 0) continue;
        uint64_t held[1 + SQ_CAP / 32];
        held[0] = lane < k ? lists[q * 32 + lane] : 0ull;
#pragma unroll
        for (int j = 0; j < SQ_CAP / 32; ++j) {
          const int e = j * 32 + lane;
          held[1 + j] = e < c ? cands[q * SQ_CAP + e] : 0ull;
        }
        uint64_t mine = 0ull;
        for (int rd = 0; rd < k; ++rd) {
          uint64_t best = held[0];
          int bj = 0;
#pragma unroll
          for (int j = 1; j < 1 + SQ_CAP / 32; ++j)
            if (held[j] > best) {
              best = held[j];
              bj = j;
            }
          uint64_t mx = best;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) {
            const uint64_t y = __shfl_xor_sync(0xffffffffu, mx, o);
            mx = y > mx ? y : mx;
          }
          if (lane == rd) mine = mx;
          if (mx == 0ull) continue;
          const unsigned win = __ballot_sync(0xffffffffu, best == mx);
          if (lane == __ffs(win) - 1) {
#pragma unroll
            for (int j = 0; j < 1 + SQ_CAP / 32; ++j)
              if (j == bj) held[j] = 0ull;
          }
        }
        if (lane < k) lists[q * 32 + lane] = mine;
        const uint64_t kth = __shfl_sync(0xffffffffu, mine, k - 1);
        if (lane == 0) {
          float sk = -FLT_MAX;
          int32_t ik;
          if (kth != 0ull) unpack_key(kth, sk, ik);
          theta[q] = sk;
          cnt[q] = 0;
        }
      }
      named_bar_sync(1, 128);
    }
    // This CTA's list per query (list index = blockIdx.x of 2 * nsplit).
    const int nlists = (int)gridDim.x;
    for (int q = ew; q < nq; q += 4) {
      if (lane < k) {
        const uint64_t key = lists[q * 32 + lane];
        float sc = -FLT_MAX;
        int32_t id = -1;
        if (key != 0ull) unpack_key(key, sc, id);
        const size_t o = ((size_t)q * nlists + blockIdx.x) * k + lane;
        p.part_s[o] = sc;
        p.part_i[o] = id;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, SQ_TMEM_COLS);
  }
  if (threadIdx.x == 0 && *abort_flag) set_error(p.err, kErrTimeout);
}

// ---- host side ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

bool make_map(CUtensorMap* map, const uint16_t* base, int64_t rows, int32_t d, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  const cuuint32_t box[2] = {(cuuint32_t)BK, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(base), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Test hook of the main kernel's bounded waits (hs_debug_retrieve_wait): the
// wait limit (0: 2 s) and whether every CTA withholds its first stage.
std::atomic<uint64_t> g_ret_wait_limit_ns{0};
std::atomic<int> g_ret_withhold{0};

template <int KREG, int CL>
hs_status configure_kernel() {
  static std::atomic<uint64_t> done{0};
  return once_per_device(done, [] {
    return cuda_fail(cudaFuncSetAttribute(retrieve_kernel<KREG, CL>,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)Ring<CL>::smem),
                     "retrieve smem attribute");
  });
}

// Clusters of two that can be resident at once (one CTA per SM; pairs must
// share a GPC), cached per kernel variant.
template <int KREG>
int64_t max_pairs() {
  static std::atomic<int64_t> per_device[kMaxDeviceOrdinals];   // 0: not yet queried
  const int dev = device_ordinal();
  int64_t cached = dev >= 0 ? per_device[dev].load() - 1 : -1;
  if (cached < 0) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3((unsigned)(num_sms() & ~1), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = Ring<2>::smem;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, retrieve_kernel<KREG, 2>, &cfg) != cudaSuccess) n = 0;
    cached = n;
    if (dev >= 0) per_device[dev].store(cached + 1);
  }
  return cached;
}

template <int KREG, int CL>
hs_status launch_kernel(const CUtensorMap& mq, const CUtensorMap& mc, const Params& prm,
                        int64_t grid, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = CL;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = Ring<CL>::smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = CL > 1 ? 2 : 1;
  return cuda_fail(cudaLaunchKernelEx(&cfg, retrieve_kernel<KREG, CL>, mq, mc, prm),
                   "retrieve launch");
}

// Plan and launch for one register-list size.  Clusters of two when there
// are at least two query blocks (they share corpus tiles), else single CTAs.
template <int KREG>
hs_status launch_variant(const uint16_t* corpus, int64_t N, int32_t d, const CUtensorMap& mq,
                         Params& prm, cudaStream_t stream) {
  const int64_t sms = num_sms();
  const int64_t qblocks_max = (prm.Qmax + BM - 1) / BM;
  hs_status st = configure_kernel<KREG, 1>();
  if (st != HS_OK) return st;
  int cl = 1;
  // Unit executors: at most 16 * kMaxListsPerLane, so every query's lists
  // (2 per split, nsplit <= slots) fit the warp merge.
  int64_t slots = std::min<int64_t>(sms, 16 * kMaxListsPerLane);
  if (qblocks_max >= 2) {
    st = configure_kernel<KREG, 2>();
    if (st != HS_OK) return st;
    const int64_t pairs = std::min<int64_t>(std::min<int64_t>(max_pairs<KREG>(), sms / 2),
                                            16 * kMaxListsPerLane);
    if (pairs >= 1) {
      cl = 2;
      slots = pairs;
    }
  }
  CUtensorMap mc;
  if (!make_map(&mc, corpus, N, d, BN / cl))
    return fail(HS_ERR_CUDA, "cuTensorMapEncodeTiled failed (driver entry point or arguments)");
  prm.slots = (int32_t)slots;
  prm.cl = cl;
  // With a host-known count the grid covers only the plan's units; with a
  // device count every slot gets a CTA (or pair) and idle ones exit.
  int64_t execs = slots;
  if (!prm.count_dev) {
    const SplitPlan sp = split_plan(prm.Qmax, prm.tiles, prm.k, slots, cl);
    const int64_t units = (int64_t)sp.groups * sp.nsplit;
    if (units < execs) execs = units;
  }
  if (execs < 1) execs = 1;
  return cl == 2 ? launch_kernel<KREG, 2>(mq, mc, prm, execs * 2, stream)
                 : launch_kernel<KREG, 1>(mq, mc, prm, execs, stream);
}

}  // namespace

// Upper bound over every query count up to Q: a plan's split count is at most
// max_splits() and the grid is at most the SM count, so one workspace serves
// every batch of at most Q queries.
size_t retrieve_topk_workspace(int64_t Q, int64_t N, int32_t d, int32_t k) {
  if (Q <= 0 || N <= 0 || k <= 0) return 256;
  (void)d;
  const int64_t sms = num_sms();
  const int64_t ns = max_splits(sms, (N + BN - 1) / BN, k);
  const size_t part = (((size_t)Q * 2 * ns * k * 4) + 255) & ~(size_t)255;
  const size_t list = k <= 32 ? 0 : ((((size_t)sms * kEpi * 2 * k * 4) + 255) & ~(size_t)255);
  const size_t qfloor = (((size_t)Q * 4) + 255) & ~(size_t)255;
  const size_t flags = ((((size_t)(Q + BM - 1) / BM) * 4) + 255) & ~(size_t)255;
  // lists, large-k lists, shared floors, large-k floors, block flags
  return 2 * part + 2 * list + 2 * qfloor + flags + 256;
}

// Qmax rows of `queries` are addressable; the kernels process the first
// count of them, count = *count_dev (clamped to [0, Qmax]) or Qmax if
// count_dev is NULL.  With inv NULL, scores_out / ids_out get one row per
// query; otherwise n_out rows, row o holding the results of query inv[o].
hs_status launch_retrieve_topk(const uint16_t* queries, int64_t Qmax, const int32_t* count_dev,
                               const int32_t* inv, int64_t n_out, const uint16_t* corpus,
                               int64_t N, int32_t d, int32_t k, float* scores_out,
                               int32_t* ids_out, void* ws, size_t ws_bytes, cudaStream_t stream) {
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  const int64_t sms = num_sms();
  const int64_t tiles = (N + BN - 1) / BN;
  const size_t need = retrieve_topk_workspace(Qmax, N, d, k);
  if (ws_bytes < need)
    return fail(HS_ERR_WORKSPACE, "retrieve workspace too small: %zu < %zu", ws_bytes, need);
  CUtensorMap mq;
  if (!make_map(&mq, queries, Qmax, d, BM))
    return fail(HS_ERR_CUDA, "cuTensorMapEncodeTiled failed (driver entry point or arguments)");
  const int64_t ns_max = max_splits(sms, tiles, k);
  const size_t part = (((size_t)Qmax * 2 * ns_max * k * 4) + 255) & ~(size_t)255;
  const size_t list = k <= 32 ? 0 : ((((size_t)sms * kEpi * 2 * k * 4) + 255) & ~(size_t)255);
  char* w = static_cast<char*>(ws);
  Params prm{};
  prm.Qmax = Qmax;
  prm.N = N;
  prm.tiles = tiles;
  prm.count_dev = count_dev;
  prm.k = k;
  prm.kb_count = (d + BK - 1) / BK;
  prm.wait_limit_ns = g_ret_wait_limit_ns.load();
  prm.withhold_first = g_ret_withhold.load();
  prm.part_s = reinterpret_cast<float*>(w);
  prm.part_i = reinterpret_cast<int32_t*>(w + part);
  prm.list_s = reinterpret_cast<float*>(w + 2 * part);
  prm.list_i = reinterpret_cast<int32_t*>(w + 2 * part + list);
  const size_t qfloor_bytes = (((size_t)Qmax * 4) + 255) & ~(size_t)255;
  prm.qfloor = reinterpret_cast<uint32_t*>(w + 2 * part + 2 * list);
  float* kth = reinterpret_cast<float*>(w + 2 * part + 2 * list + qfloor_bytes);
  uint32_t* block_flags =
      reinterpret_cast<uint32_t*>(w + 2 * part + 2 * list + 2 * qfloor_bytes);
  prm.err = err;
  const bool small = Qmax <= SQ_N && k <= 32 && prm.kb_count <= SQ_MAXKB;
  if (!small) {
    // The shared per-query floors of the register-list passes start empty.
    const cudaError_t ze = cudaMemsetAsync(prm.qfloor, 0, (size_t)Qmax * 4, stream);
    if (ze != cudaSuccess) return cuda_fail(ze, "floor clear");
  }
  const OutRows rows{inv, n_out};
  const int64_t R = inv ? n_out : Qmax;             // rows the final merge writes
  auto merge = [&](const Params& pm, int32_t kout, float* os, int32_t* oi, OutRows orows,
                   uint32_t* flag_out = nullptr, const uint32_t* only = nullptr) -> hs_status {
    const int64_t nr = orows.inv ? orows.n_out : Qmax;
    if (nr == 0) return HS_OK;
    // Every plan caps its executors (slots) at 16 * kMaxListsPerLane, so a
    // query has at most 32 * kMaxListsPerLane lists: the warp merge takes
    // every launch.
    if (2 * (int64_t)pm.slots > 32 * kMaxListsPerLane)
      return fail(HS_ERR_UNSUPPORTED, "more lists per query than the merge takes");
    {
      const int64_t blocks = (nr + 7) / 8;          // one warp per row
      const dim3 grid((unsigned)(blocks < sms * 16 ? blocks : sms * 16));
      // lists per query <= 2 * slots (nsplit <= slots): lanes need that / 32
      const int64_t lpl = (2 * (int64_t)pm.slots + 31) / 32;
      if (lpl <= 2)
        launch_pdl(merge_warp_kernel<2>, grid, dim3(256), 0, stream, pm, os, oi, kout, orows,
                   flag_out, only);
      else if (lpl <= 3)
        launch_pdl(merge_warp_kernel<3>, grid, dim3(256), 0, stream, pm, os, oi, kout, orows,
                   flag_out, only);
      else if (lpl <= 5)
        launch_pdl(merge_warp_kernel<5>, grid, dim3(256), 0, stream, pm, os, oi, kout, orows,
                   flag_out, only);
      else
        launch_pdl(merge_warp_kernel<kMaxListsPerLane>, grid, dim3(256), 0, stream, pm, os, oi,
                   kout, orows, flag_out, only);
      return cuda_fail(cudaGetLastError(), "merge launch");
    }
  };
  hs_status st;
  if (small) {
    // Small batch: corpus as the M operand, queries resident (swap-AB).
    CUtensorMap mq16, mc128;
    if (!make_map(&mq16, queries, Qmax, d, SQ_N) || !make_map(&mc128, corpus, N, d, SQ_BM))
      return fail(HS_ERR_CUDA, "cuTensorMapEncodeTiled failed (driver entry point or arguments)");
    static std::atomic<uint64_t> sq_configured{0};
    const hs_status cst = once_per_device(sq_configured, [] {
      return cuda_fail(cudaFuncSetAttribute(retrieve_small_kernel,
                                            cudaFuncAttributeMaxDynamicSharedMemorySize,
                                            (int)SQ_SMEM),
                       "retrieve smem attribute");
    });
    if (cst != HS_OK) return cst;
    // Lists per query = 2 * nsplit of the plan the merge kernel recomputes
    // (one query block, one group: nsplit = min(slots, tiles, 8192 / k)).
    prm.slots = (int32_t)std::max<int64_t>(1, std::min<int64_t>(sms / 2, 16 * kMaxListsPerLane));
    prm.cl = 1;
    const SplitPlan sp = split_plan(1, tiles, k, prm.slots, 1);
    const int64_t grid = 2 * (int64_t)sp.nsplit;
    launch_pdl(retrieve_small_kernel, dim3((unsigned)grid), dim3(SQ_THREADS), SQ_SMEM, stream,
               mq16, mc128, prm, (N + SQ_BM - 1) / SQ_BM);
    st = cuda_fail(cudaGetLastError(), "retrieve launch");
  } else if (k <= 8) {
    st = launch_variant<8>(corpus, N, d, mq, prm, stream);
  } else if (k <= 12) {
    st = launch_variant<12>(corpus, N, d, mq, prm, stream);
  } else if (k <= 16) {
    st = launch_variant<16>(corpus, N, d, mq, prm, stream);
  } else if (k <= 32) {
    st = launch_variant<32>(corpus, N, d, mq, prm, stream);
  } else {
    // Large k.  With at least 64 corpus tiles an optimistic pass runs first:
    // the register-list kernel (32 per list, no shared floor: a floor that
    // bounds 32nd-best scores would cut rows of the top k) over the whole
    // corpus, merged to the first k of the union of its lists.  A list whose
    // last entry is below the union's k-th best holds every row of its range
    // that can be in the top k, so where no list of a query is cut that way
    // the union's first k are exact.  The merge flags the query blocks where
    // some list may have been cut; only those take the exact two-pass path
    // (pass 1: register lists over the first eighth of the corpus, whose
    // union's k-th best is a score k distinct rows reach, hence a floor;
    // pass 2: the large-k kernel over the whole corpus keeping scores >= the
    // floor), and every kernel of it skips the other blocks.  Both passes'
    // lists go through the same workspace; the floors are staged in it.
    if (tiles >= 64) {
      const int64_t nb = (Qmax + BM - 1) / BM;
      cudaError_t ze = cudaMemsetAsync(block_flags, 0, (size_t)nb * 4, stream);
      if (ze != cudaSuccess) return cuda_fail(ze, "flag clear");
      Params pa = prm;
      pa.k = 32;
      pa.qfloor = nullptr;
      pa.floor = nullptr;
      st = launch_variant<32>(corpus, N, d, mq, pa, stream);
      if (st != HS_OK) return st;
      st = merge(pa, k, scores_out, ids_out, rows, block_flags, nullptr);
      if (st != HS_OK) return st;
      count_launches(2);
      Params p1 = prm;
      p1.tiles = tiles / 8;
      p1.N = p1.tiles * BN;
      p1.k = 32;
      p1.floor = nullptr;
      p1.only = block_flags;
      st = launch_variant<32>(corpus, N, d, mq, p1, stream);
      if (st != HS_OK) return st;
      st = merge(p1, k, kth, nullptr, OutRows{nullptr, 0}, nullptr, block_flags);
      if (st != HS_OK) return st;
      count_launches(2);
      prm.floor = kth;
      prm.floor_stride = 1;
      prm.floor_index = 0;
      prm.only = block_flags;
      // Pass 1's shared floors bound 32nd-best scores, not k-th best: clear.
      ze = cudaMemsetAsync(prm.qfloor, 0, (size_t)Qmax * 4, stream);
      if (ze != cudaSuccess) return cuda_fail(ze, "floor clear");
    }
    st = launch_variant<0>(corpus, N, d, mq, prm, stream);
  }
  if (st != HS_OK) return st;
  st = merge(prm, k, scores_out, ids_out, rows, nullptr, prm.only);
  if (st != HS_OK) return st;
  count_launches(R > 0 ? 2 : 1);  // retrieve_kernel + merge_warp_kernel
  return HS_OK;
}

}  // namespace hs

/*
 * Diagnostics only (declared in hs.h as hs_debug_retrieve_wait).
 */
extern "C" hs_status hs_debug_retrieve_wait(uint64_t limit_ns, int32_t withhold_first) {
  hs::clear_last_error();
  if (limit_ns > hs::kWaitLimitNs) return hs::fail(HS_ERR_INVALID_ARG, "limit above 2 s");
  if (withhold_first < 0 || withhold_first > 1)
    return hs::fail(HS_ERR_INVALID_ARG, "withhold_first must be 0 or 1");
  hs::g_ret_wait_limit_ns.store(limit_ns);
  hs::g_ret_withhold.store(withhold_first);
  return HS_OK;
}
