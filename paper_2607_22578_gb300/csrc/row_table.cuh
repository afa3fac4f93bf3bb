// Device hash table of row fingerprints: the lookup by signature with which
// a new node is matched against the nodes already in the window (Section
// 3.3, "Dynamic Fusion and Reuse Mechanism" (I)).  Each slot holds a 64-bit
// fingerprint and the smallest row index that carries it.  The slots may
// live in global or shared memory.
#pragma once

#include <stdint.h>

namespace hs {
namespace table {

constexpr uint64_t kEmpty = ~0ull;      // free slot; fingerprint kEmpty has its own slot
constexpr uint32_t kNoRow = 0xffffffffu;

// log2 of the slot count for n rows: at least twice n, at least 64.
constexpr int table_log2(int64_t n) {
  int l = 6;
  while ((int64_t(1) << l) < 2 * n) ++l;
  return l;
}

// Open addressing with linear probing over 2^log2T slots (at least twice the
// row count, so probes are short and a free slot always exists); the key
// kEmpty marks a free slot, so the fingerprint kEmpty itself uses slot 2^log2T.
__device__ __forceinline__ uint32_t home_slot(uint64_t f, int log2T) {
  return (uint32_t)((f * 0x9E3779B97F4A7C15ull) >> (64 - log2T));
}

__device__ __forceinline__ uint32_t insert_key(uint64_t* keys, uint64_t f, int log2T) {
  const uint32_t mask = (1u << log2T) - 1u;
  if (f == kEmpty) return mask + 1u;
  uint32_t s = home_slot(f, log2T);
  for (uint32_t it = 0; it <= mask; ++it) {
    uint64_t k = *reinterpret_cast<volatile uint64_t*>(keys + s);
    if (k == kEmpty) {
      k = atomicCAS(reinterpret_cast<unsigned long long*>(keys + s), (unsigned long long)kEmpty,
                    (unsigned long long)f);
      if (k == kEmpty) return s;
    }
    if (k == f) return s;
    s = (s + 1u) & mask;
  }
  return mask + 1u;  // not reached: the table has more slots than rows
}

__device__ __forceinline__ uint32_t find_key(const uint64_t* keys, uint64_t f, int log2T) {
  const uint32_t mask = (1u << log2T) - 1u;
  if (f == kEmpty) return mask + 1u;
  uint32_t s = home_slot(f, log2T);
  for (uint32_t it = 0; it <= mask; ++it) {
    const uint64_t k = keys[s];
    if (k == f || k == kEmpty) return k == f ? s : mask + 1u;
    s = (s + 1u) & mask;
  }
  return mask + 1u;
}

// One warp-round of inserts: lane l offers (f, i) if valid, with rows in
// ascending lane order.  Lanes with equal fingerprints are combined; the
// lowest such lane (smallest index) inserts.
__device__ __forceinline__ void insert_row(uint64_t* keys, uint32_t* idx, int log2T, bool valid,
                                           uint64_t f, uint32_t i) {
  const unsigned act = __ballot_sync(0xffffffffu, valid);
  if (!valid) return;
  const unsigned peers = __match_any_sync(act, f);
  if ((int)(__ffs(peers) - 1) != (int)(threadIdx.x & 31)) return;
  const uint32_t s = insert_key(keys, f, log2T);
  if (*reinterpret_cast<volatile uint32_t*>(idx + s) > i) atomicMin(idx + s, i);
}

}  // namespace table
}  // namespace hs
