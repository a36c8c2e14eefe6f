// Stochastic drafting (Sec. 2.2, "sample k candidates"): the k candidates of a depth are
// k draws without replacement from q = softmax(logit / T). They are taken by the
// Gumbel-top-k trick (Vieira 2014; Kool, van Hoof and Welling, ICML 2019): with G_v a
// standard Gumbel deviate per token, the k largest keys logit_v / T + G_v, by descending
// key, have the law of k successive draws without replacement from q.
//
// The deviates are far too many to pass in (one per vocabulary entry and hidden row), so
// they come from a counter-based generator: SplitMix64 (Steele, Lea and Flood, "Fast
// splittable pseudorandom number generators", OOPSLA 2014), whose n-th output for seed s
// is its 64-bit finaliser applied to s + n * golden-gamma. Row r's token v (r = b * N +
// i - 1 for sequence b and depth i) uses output n = r * V + v + 1. The uniform deviate
// keeps the output's top 23 bits plus one half, U = (floor(x / 2^41) + 1/2) / 2^23, an odd
// multiple of 2^-24 that is exact in float32 and never 0 or 1; G = -log(-log U).
#pragma once

#include <stdint.h>

namespace fe {

__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t n) {
    uint64_t z = seed + n * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// U in (0, 1), exact in float32
__device__ __forceinline__ float sample_uniform(uint64_t seed, uint64_t n) {
    return ((float)(uint32_t)(splitmix64_at(seed, n) >> 41) + 0.5f) * (1.0f / 8388608.0f);
}

// G = -log(-log U). logf (not the fast approximation): near U = 1, where the largest
// deviates come from, -log U is about 1 - U and needs its full relative accuracy.
__device__ __forceinline__ float gumbel_of(float u) { return -logf(-logf(u)); }

// the counter of row r's token v
__device__ __forceinline__ uint64_t sample_counter(int row, int V, int v) {
    return (uint64_t)row * (uint64_t)V + (uint64_t)v + 1ull;
}

// the sampling key of one logit
__device__ __forceinline__ float sample_key(float logit, float inv_temp, uint64_t seed, int row, int V, int v) {
    return fmaf(logit, inv_temp, gumbel_of(sample_uniform(seed, sample_counter(row, V, v))));
}

// The largest deviate any token can draw: U <= 1 - 2^-24, so G <= -log(-log(1 - 2^-24)),
// about 16.636; rounded up. A token whose logit / T + kGumbelMax is below a row's current
// k-th best key cannot enter its top-k.
constexpr float kGumbelMax = 16.64f;

// Row r of the LM head's hidden rows (r = i * B + b, depth i 0-based) draws with counter
// row b * N + i.
__device__ __forceinline__ int sample_row(int r, int B, int N) { return (r % B) * N + r / B; }

}  // namespace fe
