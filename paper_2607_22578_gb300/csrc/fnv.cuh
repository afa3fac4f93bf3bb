// 64-bit FNV-1a over the little-endian octets of int32 tokens, on (hi:lo)
// 32-bit halves — the hash H of the node signature (Section 3.3, Eq. 2).
//
// A multiply by the prime 2^40 + 0x1b3 is one wide 32x32 multiply, one
// multiply-add and one shift-add.  When a token's two high octets are zero
// (every token below 65536), the last two rounds "xor 0, multiply by prime"
// collapse exactly into one multiply by prime^3 mod 2^64 — xor with zero is
// the identity — so the result is bit-identical to the octet-wise definition.
#pragma once

#include <stdint.h>

namespace hs {
namespace fnv {

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

}  // namespace fnv
}  // namespace hs
