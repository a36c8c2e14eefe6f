/*
 * Seeded, counter-based synthetic input generator.
 *
 * This module only draws numbers. It holds none of the drafter's arithmetic and is
 * shared by the tests, the benchmark and the oracle's callers so that both sides of a
 * parity check see byte-identical inputs. Every value is a pure function of
 * (seed, tensor_id, index), so any slice of a tensor can be regenerated on its own
 * and the result does not depend on the number of threads.
 *
 * Hash: the SplitMix64 output function (Steele, Lea and Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014), applied to a counter.
 *
 * Normal deviates: the Irwin-Hall sum of twelve uniform 16-bit integers, centred and
 * scaled (the classic "sum of 12 uniforms" approximation of N(0,1): mean 0, variance
 * 1 - 2^-32, support [-6, 6]). It uses only integer arithmetic and one exactly
 * representable scaling, so every platform produces the same bits.
 *
 * Portable C99: no intrinsics, no -march flags, no reliance on the signedness of char.
 */
#include <stdint.h>
#include <string.h>

static uint64_t sm64(uint64_t z)
{
    z += 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* Key of one tensor's stream. */
static uint64_t stream_key(uint64_t seed, uint64_t tensor_id)
{
    return sm64(sm64(seed) ^ sm64(tensor_id ^ 0x5851F42D4C957F2DULL));
}

static double normal_at(uint64_t key, uint64_t i)
{
    uint64_t w[3];
    int64_t s = 0;
    w[0] = sm64(key + 3u * i);
    w[1] = sm64(key + 3u * i + 1u);
    w[2] = sm64(key + 3u * i + 2u);
    for (int j = 0; j < 3; ++j)
        for (int q = 0; q < 4; ++q)
            s += (int64_t)((w[j] >> (16 * q)) & 0xFFFFu);
    /* 12 * 32767.5 = 393210; dividing by 2^16 is exact */
    return ((double)s - 393210.0) / 65536.0;
}

static uint16_t f32_to_bf16_rne(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu))
        return 0x7FC0u; /* NaN (never produced here) */
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/* dtype: 0 = float32, 1 = bfloat16 (round to nearest even from the float32 value). */
void synth_fill_normal(uint64_t seed, uint64_t tensor_id, int64_t n, double stddev,
                       int32_t dtype, void *out)
{
    const uint64_t key = stream_key(seed, tensor_id);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        float v = (float)(normal_at(key, (uint64_t)i) * stddev);
        if (dtype == 0)
            ((float *)out)[i] = v;
        else
            ((uint16_t *)out)[i] = f32_to_bf16_rne(v);
    }
}

/* Same values as synth_fill_normal, but element i of the stream is written to
 * out[offset + i] for i in [start, start + n): lets a caller regenerate a slice. */
void synth_fill_normal_slice(uint64_t seed, uint64_t tensor_id, int64_t start, int64_t n,
                             double stddev, int32_t dtype, void *out)
{
    const uint64_t key = stream_key(seed, tensor_id);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        float v = (float)(normal_at(key, (uint64_t)(start + i)) * stddev);
        if (dtype == 0)
            ((float *)out)[i] = v;
        else
            ((uint16_t *)out)[i] = f32_to_bf16_rne(v);
    }
}

/* Integers uniform in [lo, hi] (inclusive); modulo bias is below 2^-40 for the ranges used. */
void synth_fill_uniform_int(uint64_t seed, uint64_t tensor_id, int64_t n, int64_t lo,
                            int64_t hi, int32_t *out)
{
    const uint64_t key = stream_key(seed, tensor_id);
    const uint64_t span = (uint64_t)(hi - lo + 1);
    for (int64_t i = 0; i < n; ++i)
        out[i] = (int32_t)(lo + (int64_t)(sm64(key + (uint64_t)i) % span));
}

/* A seeded permutation of 0..n-1 (Fisher-Yates, Durstenfeld's form). */
void synth_permutation(uint64_t seed, uint64_t tensor_id, int64_t n, int32_t *out)
{
    const uint64_t key = stream_key(seed, tensor_id);
    for (int64_t i = 0; i < n; ++i)
        out[i] = (int32_t)i;
    for (int64_t i = n - 1; i > 0; --i) {
        int64_t j = (int64_t)(sm64(key + (uint64_t)i) % (uint64_t)(i + 1));
        int32_t t = out[i];
        out[i] = out[j];
        out[j] = t;
    }
}

/* Raw hash, exported so a test can check it against published SplitMix64 outputs. */
uint64_t synth_splitmix64(uint64_t z) { return sm64(z); }
