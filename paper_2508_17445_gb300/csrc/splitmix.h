// splitmix.h -- the counter-based generator behind the synthetic stand-in
// model of the rollout driver (host and device).
//
// SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number
// generators", OOPSLA 2014): element i of the stream with seed s is
// mix(s + (i + 1) * 0x9E3779B97F4A7C15) over 64-bit wrap-around arithmetic,
// mix(z) = z1 ^ (z1 >> 31) with z0 = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9 and
// z1 = (z0 ^ (z0 >> 27)) * 0x94D049BB133111EB. Indexing the stream by a
// counter makes every draw addressable: the counter packs
//   tag (4 bits) << 60 | a (28 bits) << 32 | b (20 bits) << 12 | c (12 bits).
#pragma once

#include <stdint.h>

#ifdef __CUDACC__
#define TP_HD __host__ __device__ __forceinline__
#else
#define TP_HD inline
#endif

namespace tp {

// Draw tags. Activations: a = node, b = token index inside the node,
// c = 64-bit word of the row (4 bf16 values per word).
constexpr uint32_t kTagK = 1, kTagV = 2, kTagQ = 3;
// Stand-in model draws. Token level: a = node, b = token index.
constexpr uint32_t kTagEos = 4, kTagTokenLogp = 5;
// Segment level: a = node, b = draw kind (kSeg*).
constexpr uint32_t kTagSegment = 6;
constexpr uint32_t kSegScale = 0, kSegBoxed = 1, kSegFail = 2, kSegCorrect = 3;
// Query level: a = query, b = draw kind (kQuery*), c = fallback count.
constexpr uint32_t kTagQuery = 7;
constexpr uint32_t kQueryInit = 0, kQueryPick = 1, kQueryDepth = 2;

TP_HD uint64_t splitmix64(uint64_t seed, uint64_t i) {
    uint64_t z = seed + (i + 1) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

TP_HD uint64_t draw_counter(uint32_t tag, uint32_t a, uint32_t b, uint32_t c) {
    return (uint64_t)tag << 60 | (uint64_t)(a & 0xfffffffu) << 32 | (uint64_t)(b & 0xfffffu) << 12 | (c & 0xfffu);
}

// Uniform double in [0, 1): the top 53 bits.
TP_HD double draw_uniform(uint64_t seed, uint32_t tag, uint32_t a, uint32_t b, uint32_t c) {
    return (double)(splitmix64(seed, draw_counter(tag, a, b, c)) >> 11) * (1.0 / 9007199254740992.0);
}

// bf16 bit pattern from 16 random bits: random sign and 7-bit mantissa,
// exponent 2^-3 .. 2^0, so values lie in +-[0.125, 2) (root mean square
// about 0.9, the scale of unit-normal activations).
TP_HD uint16_t synth_bf16_bits(uint32_t r16) {
    return (uint16_t)((r16 & 0x8000u) | ((124u + ((r16 >> 7) & 3u)) << 7) | (r16 & 0x7fu));
}

}  // namespace tp
