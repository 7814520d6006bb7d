// rng.cuh -- counter-based generators of the synthetic workload (host and
// device).  Any draw is a pure function of (seed, tag, a, b), so a kernel can
// produce any element of any step without state.
//
//   mix64(z): SplitMix64's output function (Steele, Lea & Flood, OOPSLA 2014)
//             applied to z + 0x9E3779B97F4A7C15.
//   hash(seed, tag, a, b) = mix64(mix64(mix64(mix64(seed) ^ tag) ^ a) ^ b)
//             tags: 1 x0, 2 centre, 3 curvature, 4 noise key, 5 permutation,
//                   6 edge activation, 7 local step counts.
//   fmix32:   MurmurHash3's 32-bit finalizer (Appleby), applied twice per
//             element (fp32 storage) or per pair of elements (bf16 storage)
//             for the gradient noise, so that its cost stays in 32-bit
//             integer arithmetic.
#pragma once
#include <cstdint>

#if defined(__CUDACC__)
#define GL_HD __host__ __device__ __forceinline__
#else
#define GL_HD inline
#endif

namespace gasloc {

enum : uint64_t { kTagX0 = 1, kTagCentre = 2, kTagCurv = 3, kTagNoise = 4, kTagPerm = 5,
                  kTagEdge = 6, kTagSteps = 7 };

GL_HD uint64_t mix64(uint64_t z) {
    z += 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

GL_HD uint64_t hash4(uint64_t seed, uint64_t tag, uint64_t a, uint64_t b) {
    return mix64(mix64(mix64(mix64(seed) ^ tag) ^ a) ^ b);
}

GL_HD uint32_t fmix32(uint32_t h) {
    h ^= h >> 16;
    h *= 0x85EBCA6Bu;
    h ^= h >> 13;
    h *= 0xC2B2AE35u;
    h ^= h >> 16;
    return h;
}

// 24-bit integer uniform in [0, 2^24) from the top bits of a hash.
GL_HD uint32_t top24(uint64_t h) { return static_cast<uint32_t>(h >> 40); }

// Noise word a of step key (klo, khi): with fp32 storage the word of global
// element a; with bf16 storage its 16-bit halves belong to elements 2a (low)
// and 2a + 1 (high).
GL_HD uint32_t noise_word(uint32_t a, uint32_t klo, uint32_t khi) {
    return fmix32(fmix32(a ^ klo) ^ khi);
}

}  // namespace gasloc
