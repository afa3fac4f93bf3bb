// Reuse-driven priority of fused nodes (Section 3.3, "Reuse-Driven Priority
// Adjustment", Eq. 3): phi(v*) = sum of phi(v) over the logical nodes v
// merged into v*.  With the inverse map of the merge, that is a segmented
// sum: out[u] = sum of phi[i] over the rows i with inverse[i] = u.
//
// Groups are arbitrary (a hot row's copies are scattered over the batch).
// Adding every row to the output with a global atomic would serialise the
// hot groups in the L2, and a shared-memory hash table per tile costs more
// than the atomics it saves for the cold groups.  So each CTA sorts its
// rows into three paths:
//   1. per round of 32 rows, the lanes of one group are combined with
//      shuffles (pairwise trees), leaving one partial sum per distinct group;
//   2. a group with ordinal below kSsDense goes to a dense per-CTA array in
//      shared memory (fp64 shared atomics).  Ordinals follow first
//      occurrence, so the frequent groups of a batch mostly have small
//      ordinals; the array is added to the output once per CTA, a warp's
//      32 consecutive ordinals per instruction, zeros skipped;
//   3. a larger ordinal that occurs more than once in its round (a hot group
//      that appeared late) claims a slot of a per-CTA hash table (bounded
//      probing; a full table sends the sum straight to the output), flushed
//      once per CTA; every other partial sum is one global fp64 atomic.
// The output is cleared with a memset first.  Additions run in fp64 in no
// fixed order: for a group of m rows the result is within
// ((m-1) u / (1 - (m-1) u)) * sum |phi| of the exact sum (u = 2^-53), and
// exact when every partial sum is representable (integers below 2^53).
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kSsThreads = 256;
constexpr int kSsWarps = kSsThreads / 32;
constexpr int kSsRounds = 4;                             // rounds of 32 rows per warp tile
constexpr int kSsTile = 32 * kSsRounds;                  // rows per warp tile
constexpr int kSsCtaRows = kSsWarps * kSsTile;           // rows per CTA tile
constexpr int kSsDense = 256;                            // ordinals summed densely per CTA
constexpr int kSsLog2Slots = 9;
constexpr int kSsSlots = 1 << kSsLog2Slots;              // hash slots for repeated large ordinals
constexpr int kSsProbes = 32;                            // probes before going to the output

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

// Slot of group g in the hash table, claimed if new, or -1 when kSsProbes
// slots in a row hold other groups.
__device__ __forceinline__ int claim_slot(int32_t* keys, int32_t g) {
  uint32_t s = ss_slot(g, kSsLog2Slots);
#pragma unroll 1
  for (int probe = 0; probe < kSsProbes; ++probe) {
    const int32_t k = atomicCAS(keys + s, -1, g);
    if (k == -1 || k == g) return (int)s;
    s = (s + 1u) & (kSsSlots - 1u);
  }
  return -1;
}

__global__ void __launch_bounds__(kSsThreads) segment_sum_kernel(
    const double* __restrict__ phi, const int32_t* __restrict__ inverse, int64_t n,
    const int32_t* __restrict__ count_dev, int64_t max_groups, double* __restrict__ out,
    unsigned* err) {
  pdl_wait();
  pdl_trigger();
  __shared__ double dense[kSsDense];
  __shared__ double hsum[kSsSlots];
  __shared__ int32_t hkey[kSsSlots];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int64_t count = max_groups;
  if (count_dev) {
    const int64_t c = __ldg(count_dev);
    count = c < 0 ? 0 : (c > max_groups ? max_groups : c);
  }
  const int32_t H = (int32_t)(count < kSsDense ? count : kSsDense);
  for (int s = tid; s < H; s += kSsThreads) dense[s] = 0.0;
  for (int s = tid; s < kSsSlots; s += kSsThreads) {
    hkey[s] = -1;
    hsum[s] = 0.0;
  }
  __syncthreads();
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
#pragma unroll
    for (int j = 0; j < kSsRounds; ++j) {
      const unsigned peers = __match_any_sync(0xffffffffu, g[j]);
      const double x = sum_peers(peers, v[j], lane);
      if (g[j] >= 0 && lane == __ffs(peers) - 1) {
        if (g[j] < H) {
          atomicAdd(dense + g[j], x);
        } else {
          const int s = peers != (1u << lane) ? claim_slot(hkey, g[j]) : -1;
          if (s >= 0)
            atomicAdd(hsum + s, x);
          else
            atomicAdd(out + g[j], x);
        }
      }
    }
  }
  __syncthreads();
  // Adding a zero changes no output (the output starts at +0), so zero
  // entries are skipped.
  for (int s = tid; s < H; s += kSsThreads) {
    const double x = dense[s];
    if (x != 0.0) atomicAdd(out + s, x);
  }
  for (int s = tid; s < kSsSlots; s += kSsThreads) {
    const int32_t k = hkey[s];
    if (k >= 0) atomicAdd(out + k, hsum[s]);
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
  const int64_t blocks = (n + kSsCtaRows - 1) / kSsCtaRows;
  const int64_t cap = (int64_t)num_sms() * 4;
  const unsigned grid = (unsigned)(blocks < cap ? blocks : cap);
  launch_pdl(segment_sum_kernel, dim3(grid), dim3(kSsThreads), 0, stream, phi, inverse, n,
             count_dev, max_groups, out, err);
  count_launches(1);
  return cuda_fail(cudaGetLastError(), "segment sum launch");
}

}  // namespace hs
