// XXH64 (public xxHash specification) split for a 4-thread chunk group: each
// thread owns one of the four accumulator lanes and consumes the 8-byte word
// at offset 8*lane of every 32-byte stripe; the lanes meet by shuffles.
#pragma once

#include <cstdint>

namespace gleam {

constexpr unsigned long long kXP1 = 0x9E3779B185EBCA87ULL;
constexpr unsigned long long kXP2 = 0xC2B2AE3D27D4EB4FULL;
constexpr unsigned long long kXP3 = 0x165667B19E3779F9ULL;
constexpr unsigned long long kXP4 = 0x85EBCA77C2B2AE63ULL;
constexpr unsigned long long kXP5 = 0x27D4EB2F165667C5ULL;

__device__ __forceinline__ unsigned long long xrotl(unsigned long long x, int r) {
  return (x << r) | (x >> (64 - r));
}

// Accumulator step on one 8-byte little-endian input word.
__device__ __forceinline__ unsigned long long xstep(unsigned long long acc,
                                                    unsigned long long w) {
  acc += w * kXP2;
  acc = xrotl(acc, 31);
  return acc * kXP1;
}

// Seed-0 start value of accumulator lane 0..3.
__device__ __forceinline__ unsigned long long xlane_start(uint32_t lane) {
  return lane == 0 ? kXP1 + kXP2 : lane == 1 ? kXP2 : lane == 2 ? 0ULL : 0ULL - kXP1;
}

// Convergence of the four lanes followed by the four merge rounds.
__device__ __forceinline__ unsigned long long xconverge(unsigned long long a0,
                                                        unsigned long long a1,
                                                        unsigned long long a2,
                                                        unsigned long long a3) {
  unsigned long long h = xrotl(a0, 1) + xrotl(a1, 7) + xrotl(a2, 12) + xrotl(a3, 18);
  const unsigned long long a[4] = {a0, a1, a2, a3};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    h ^= xstep(0ULL, a[k]);
    h = h * kXP1 + kXP4;
  }
  return h;
}

// Little-endian word from any byte address.
__device__ __forceinline__ unsigned long long load_le64_bytes(const uint8_t* p) {
  unsigned long long v = 0;
#pragma unroll
  for (int k = 0; k < 8; ++k) v |= (unsigned long long)p[k] << (8 * k);
  return v;
}

// The trailing rem (< 32) bytes after the last full stripe, then the
// avalanche.  h already includes the length.
__device__ __forceinline__ unsigned long long xfinish(unsigned long long h, const uint8_t* p,
                                                      uint32_t rem) {
  uint32_t off = 0;
  while (rem - off >= 8) {
    h ^= xstep(0ULL, load_le64_bytes(p + off));
    h = xrotl(h, 27) * kXP1 + kXP4;
    off += 8;
  }
  if (rem - off >= 4) {
    const unsigned long long w = (unsigned long long)p[off] |
                                 ((unsigned long long)p[off + 1] << 8) |
                                 ((unsigned long long)p[off + 2] << 16) |
                                 ((unsigned long long)p[off + 3] << 24);
    h ^= w * kXP1;
    h = xrotl(h, 23) * kXP2 + kXP3;
    off += 4;
  }
  while (off < rem) {
    h ^= (unsigned long long)p[off] * kXP5;
    h = xrotl(h, 11) * kXP1;
    ++off;
  }
  h ^= h >> 33;
  h *= kXP2;
  h ^= h >> 29;
  h *= kXP3;
  h ^= h >> 32;
  return h;
}

}  // namespace gleam
