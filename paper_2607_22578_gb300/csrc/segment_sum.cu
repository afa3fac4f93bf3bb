// Reuse-driven priority of fused nodes (Section 3.3, "Reuse-Driven Priority
// Adjustment", Eq. 3): phi(v*) = sum of phi(v) over the logical nodes v
// merged into v*.  With the inverse map of the merge, that is a segmented
// sum: out[u] = sum of phi[i] over the rows i with inverse[i] = u.
//
// Groups are arbitrary (a hot row's copies are scattered over the batch), and
// the hot groups of a Zipf-like merge would serialise any scheme that adds
// every row, or every warp's partial sum, to the output: the L2 processes
// updates of one line one at a time.  So the sum is taken in three levels:
//   1. each warp sums 4 rounds of 32 rows into its own shared-memory table
//      keyed by group ordinal; within a round, rows of one group are first
//      combined with shuffles (pairwise trees), so the keys of a round are
//      distinct and plain adds suffice;
//   2. a group met once in a warp's tile is added to the output at once (a
//      cold group: one global fp64 atomic); the groups met more than once
//      (the hot ones) are merged over the CTA's warps into a CTA table, and
//      so are the groups with ordinals below 4096: ordinals follow first
//      occurrence, so the frequent groups of a batch mostly have small
//      ordinals and share the first output lines, which every CTA would
//      otherwise update;
//   3. each group of the CTA table takes one global fp64 atomic, so a hot
//      group costs one update per CTA tile of 1024 rows.
// The output is cleared with a memset first.  Additions run in fp64 in no
// fixed order: for a group of m rows the result is within
// ((m-1) u / (1 - (m-1) u)) * sum |phi| of the exact sum (u = 2^-53), and
// exact when every partial sum is representable (integers below 2^53).
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kSsThreads = 256;
constexpr int kSsWarps = kSsThreads / 32;
constexpr int kSsRounds = 4;                             // warp-rounds per warp tile
constexpr int kSsTile = 32 * kSsRounds;                  // rows per warp tile
constexpr int kSsCtaRows = kSsWarps * kSsTile;           // rows per CTA tile
constexpr int kSsLog2Slots = 8;
constexpr int kSsSlots = 1 << kSsLog2Slots;              // slots of a warp table
constexpr int kSsLog2CtaSlots = kSsLog2Slots + 3;
constexpr int kSsLowIds = 4096;                          // ordinals always merged per CTA
constexpr int kSsCtaSlots = 1 << kSsLog2CtaSlots;        // slots of the CTA table
constexpr size_t kSsSmem = (size_t)(kSsWarps * kSsSlots + kSsCtaSlots) *
                               (sizeof(double) + sizeof(int32_t)) +
                           (size_t)kSsWarps * kSsSlots * sizeof(int32_t);
static_assert(kSsSlots >= 2 * kSsTile && kSsCtaSlots >= 2 * kSsCtaRows,
              "tables at least twice the rows they hold");
static_assert(kSsSmem <= 232448, "the warp and CTA tables fit one CTA's shared memory");

__device__ __forceinline__ uint32_t ss_slot(int32_t g, int log2_slots) {
  return ((uint32_t)g * 0x9E3779B1u) >> (32 - log2_slots);
}

// Sum of x over the lanes of `peers` (this lane's group), valid in the
// group's lowest lane.  All groups of the warp reduce at once as pairwise
// trees: in each step a member at an even position within its group adds
// the partial sum of the next member, and the odd members drop out — five
// steps reduce a group of 32, one fp64 add per lane per step (fp64 issue is
// scarce on this part, so one tree for all groups beats one butterfly per
// group).
__device__ __forceinline__ double sum_peers(unsigned peers, double x, int lane) {
  int pos = __popc(peers & ((1u << lane) - 1u));      // rank within the group
  unsigned above = peers & (0xfffffffeu << lane);    // members after this lane
  for (int step = 0; step < 5 && __any_sync(0xffffffffu, above != 0u); ++step) {
    const int next = __ffs(above) - 1;               // -1: none
    const double y = __shfl_sync(0xffffffffu, x, next & 31);
    if (above != 0u && (pos & 1) == 0) x += y;
    above &= ~__ballot_sync(0xffffffffu, (pos & 1) != 0);
    pos >>= 1;
  }
  return x;
}

// Slot of group g in a table of 2^log2 slots, claimed if new (a free slot
// always exists: the table has at least twice as many slots as keys).
__device__ __forceinline__ uint32_t claim_slot(int32_t* keys, int32_t g, int log2) {
  const uint32_t mask = (1u << log2) - 1u;
  uint32_t s = ss_slot(g, log2);
#pragma unroll 1
  for (uint32_t probe = 0; probe <= mask; ++probe) {
    const int32_t k = atomicCAS(keys + s, -1, g);
    if (k == -1 || k == g) return s;
    s = (s + 1u) & mask;
  }
  return s;   // not reached
}

__global__ void __launch_bounds__(kSsThreads) segment_sum_kernel(
    const double* __restrict__ phi, const int32_t* __restrict__ inverse, int64_t n,
    const int32_t* __restrict__ count_dev, int64_t max_groups, double* __restrict__ out,
    unsigned* err) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(16) uint8_t sm[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  double* cta_sums = reinterpret_cast<double*>(sm);
  double* sums = cta_sums + kSsCtaSlots + warp * kSsSlots;
  int32_t* cta_keys = reinterpret_cast<int32_t*>(cta_sums + kSsCtaSlots + kSsWarps * kSsSlots);
  int32_t* keys = cta_keys + kSsCtaSlots + warp * kSsSlots;
  int32_t* rows = cta_keys + kSsCtaSlots + kSsWarps * kSsSlots + warp * kSsSlots;
  int64_t count = max_groups;
  if (count_dev) {
    const int64_t c = __ldg(count_dev);
    count = c < 0 ? 0 : (c > max_groups ? max_groups : c);
  }
  const int64_t tiles = (n + kSsCtaRows - 1) / kSsCtaRows;
  for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    const int64_t r0 = t * kSsCtaRows + (int64_t)warp * kSsTile;
    int32_t g[kSsRounds];
    double v[kSsRounds];
#pragma unroll
    for (int j = 0; j < kSsRounds; ++j) {
      const int64_t r = r0 + j * 32 + lane;
      g[j] = -1;
      v[j] = 0.0;
      if (r < n) {
        g[j] = __ldg(inverse + r);
        v[j] = __ldg(phi + r);
        if (g[j] < 0 || (int64_t)g[j] >= count) {
          set_error(err, kErrInvalidArg);
          g[j] = -1;
        }
      }
    }
    for (int s = tid; s < kSsCtaSlots; s += kSsThreads) {
      cta_keys[s] = -1;
      cta_sums[s] = 0.0;
    }
#pragma unroll
    for (int j = 0; j < kSsSlots / 32; ++j) {
      keys[j * 32 + lane] = -1;
      sums[j * 32 + lane] = 0.0;
      rows[j * 32 + lane] = 0;
    }
    __syncwarp();
    // 1. this warp's rows into its own table: per round, the first lane of
    //    each distinct group adds the group's round sum (keys of a round are
    //    distinct, rounds are ordered by warp barriers: plain adds suffice)
#pragma unroll
    for (int j = 0; j < kSsRounds; ++j) {
      const unsigned peers = __match_any_sync(0xffffffffu, g[j]);
      const double x = sum_peers(peers, v[j], lane);
      if (g[j] >= 0 && lane == __ffs(peers) - 1) {
        const uint32_t s = claim_slot(keys, g[j], kSsLog2Slots);
        sums[s] += x;
        rows[s] += __popc(peers);
      }
      __syncwarp();
    }
    __syncthreads();
    // 2. groups seen more than once in a warp tile, and groups with small
    //    ordinals, are merged into the CTA table (a group meets at most one
    //    entry per warp table: shared fp64 atomics with little contention);
    //    the rest go straight to the output
#pragma unroll 1
    for (int j = 0; j < kSsSlots / 32; ++j) {
      const int32_t k = keys[j * 32 + lane];
      if (k >= 0) {
        if (rows[j * 32 + lane] > 1 || k < kSsLowIds)
          atomicAdd(cta_sums + claim_slot(cta_keys, k, kSsLog2CtaSlots), sums[j * 32 + lane]);
        else
          atomicAdd(out + k, sums[j * 32 + lane]);
      }
    }
    __syncthreads();
    // 3. one global fp64 atomic per distinct group of the CTA tile
    for (int s = tid; s < kSsCtaSlots; s += kSsThreads) {
      const int32_t k = cta_keys[s];
      if (k >= 0) atomicAdd(out + k, cta_sums[s]);
    }
    __syncthreads();
  }
}

}  // namespace

hs_status launch_segment_sum(const double* phi, const int32_t* inverse, int64_t n,
                             const int32_t* count_dev, int64_t max_groups, double* out,
                             cudaStream_t stream) {
  unsigned* err = device_error_word();
  if (!err) return fail(HS_ERR_CUDA, "could not resolve the device error word");
  if (max_groups > 0) {
    const cudaError_t e = cudaMemsetAsync(out, 0, (size_t)max_groups * sizeof(double), stream);
    if (e != cudaSuccess) return cuda_fail(e, "output clear");
  }
  if (n == 0) return HS_OK;
  static std::atomic<uint64_t> configured{0};
  const hs_status cst = once_per_device(configured, [] {
    return cuda_fail(cudaFuncSetAttribute(segment_sum_kernel,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)kSsSmem),
                     "segment sum smem attribute");
  });
  if (cst != HS_OK) return cst;
  const int64_t blocks = (n + kSsCtaRows - 1) / kSsCtaRows;
  const int64_t cap = (int64_t)num_sms() * 4;
  const unsigned grid = (unsigned)(blocks < cap ? blocks : cap);
  launch_pdl(segment_sum_kernel, dim3(grid), dim3(kSsThreads), kSsSmem, stream, phi, inverse, n,
             count_dev, max_groups, out, err);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "segment sum launch");
}

}  // namespace hs
