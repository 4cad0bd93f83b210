// Key arithmetic: a ring homomorphism from Q[atoms] into F_p0 x F_p1.
//
// The canonical form of a resolved expression res(y[l]) (Sec. 3.4) is its
// normal form in the polynomial ring Q[atoms] (floats as reals, Sec. 3.3
// "Setup"); atoms are input leaves, uninterpreted-function applications f(a)
// (one UF per transcendental, Sec. 3.4) and max-sets Max{a_i}.  The key maps
//   leaf g       -> mix64(sigma_s + (g + 1) * gamma)            mod p_s
//   constant q   -> q mod p_s   (q = m * 2^e / d, d odd)
//   a + b, a * b -> ring operations mod p_s
//   f(a)         -> mix64(mix64(K0(a) | K1(a) << 32) ^ f * gamma ^ sigma_s) mod p_s
//   Max{a_i}     -> sorted distinct u_i = K0 | K1 << 32; a single member is
//                   itself, else h = kMaxTag, h = mix64(h ^ u_i) in order,
//                   mix64(h ^ sigma_s) mod p_s
// mix64 is the output finaliser of SplitMix64 (Steele, Lea and Flood,
// OOPSLA 2014).  Equal canonical forms map to equal keys; distinct forms of
// degree d collide in one lane with probability <= d / p_s (Schwartz-Zippel),
// and the two lanes are independent.
#pragma once
#include <cstdint>

#include "prog.h"

#ifdef __CUDACC__
#define DHD __host__ __device__ __forceinline__
#else
#define DHD inline
#endif

namespace dirigo {

constexpr uint64_t kSigma0 = 0x243F6A8885A308D3ull;
constexpr uint64_t kSigma1 = 0x13198A2E03707344ull;
constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kMaxTag = 0x4D41585345545F31ull;

DHD uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
  z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
  return z ^ (z >> 31);
}

// x mod p_S for any 64-bit x, using 2^29 = c (mod p) with p = 2^29 - c.
template <int S>
DHD uint32_t reduce(uint64_t x) {
  constexpr uint64_t C = S ? 33u : 3u;
  constexpr uint32_t P = S ? kP1 : kP0;
  constexpr uint64_t M = (1ull << 29) - 1;
  x = (x >> 29) * C + (x & M);   // < 2^41
  x = (x >> 29) * C + (x & M);   // < 2^29 + 2^17
  uint32_t r = (uint32_t)x;
  return r >= P ? r - P : r;
}

// One folding step: keeps a lazily reduced accumulator below 2^41 and
// congruent mod p_S.
template <int S>
DHD uint64_t fold(uint64_t x) {
  constexpr uint64_t C = S ? 33u : 3u;
  return (x >> 29) * C + (x & ((1ull << 29) - 1));
}

template <int S>
DHD uint32_t mulmod(uint32_t a, uint32_t b) {
  return reduce<S>((uint64_t)a * b);
}

template <int S>
DHD uint32_t addmod(uint32_t a, uint32_t b) {
  constexpr uint32_t P = S ? kP1 : kP0;
  uint32_t r = a + b;
  return r >= P ? r - P : r;
}

template <int S>
DHD uint32_t submod(uint32_t a, uint32_t b) {
  constexpr uint32_t P = S ? kP1 : kP0;
  return a >= b ? a - b : a + P - b;
}

DHD uint32_t leaf_key0(uint64_t g) { return reduce<0>(mix64(kSigma0 + (g + 1) * kGamma)); }
DHD uint32_t leaf_key1(uint64_t g) { return reduce<1>(mix64(kSigma1 + (g + 1) * kGamma)); }

DHD void uf_key(int fid, uint32_t a0, uint32_t a1, uint32_t& r0, uint32_t& r1) {
  uint64_t inner = mix64((uint64_t)a0 | ((uint64_t)a1 << 32));
  uint64_t t = (uint64_t)fid * kGamma;
  r0 = reduce<0>(mix64(inner ^ t ^ kSigma0));
  r1 = reduce<1>(mix64(inner ^ t ^ kSigma1));
}

// Key of a max-set whose distinct members, packed as u = K0 | K1 << 32, are
// given sorted ascending (n >= 1).
DHD void maxset_key_sorted(const uint64_t* u, int n, uint32_t& r0, uint32_t& r1) {
  if (n == 1) {
    r0 = (uint32_t)(u[0] & 0xffffffffu);
    r1 = (uint32_t)(u[0] >> 32);
    return;
  }
  uint64_t h = kMaxTag;
  for (int i = 0; i < n; ++i) h = mix64(h ^ u[i]);
  r0 = reduce<0>(mix64(h ^ kSigma0));
  r1 = reduce<1>(mix64(h ^ kSigma1));
}

}  // namespace dirigo
