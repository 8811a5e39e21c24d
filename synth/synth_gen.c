/*
 * Seeded synthetic-input generator shared by the CUDA path's tests/bench and by the
 * CPU oracle. It holds none of the method's arithmetic: it only turns (seed, stream,
 * element index) into bf16 bit patterns of a scaled standard normal draw.
 *
 * Definition (counter-based, so any slice can be generated independently and in
 * parallel with identical results):
 *   key      = mix64(seed * 0x9E3779B97F4A7C15 + stream * 0xD1B54A32D192ED03 + 1)
 *   z        = mix64(key + index * 0x9E3779B97F4A7C15)       (mix64 = splitmix64 finaliser)
 *   u1       = (z >> 32 + 1) / 2^32   in (0, 1]
 *   u2       = (z & 0xFFFFFFFF) / 2^32 in [0, 1)
 *   n        = sqrt(-2 ln u1) * cos(2 pi u2)                (Box-Muller, one normal per index)
 *   value    = bf16_rne((float)(std * n))
 * splitmix64 is Steele, Lea and Flood, "Fast splittable pseudorandom number
 * generators" (OOPSLA 2014); Box-Muller is Box and Muller (1958).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static inline uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7FFFu + lsb;
    return (uint16_t)(u >> 16);
}

uint64_t synth_key(uint64_t seed, uint64_t stream) {
    return mix64(seed * 0x9E3779B97F4A7C15ull + stream * 0xD1B54A32D192ED03ull + 1ull);
}

/* out[i] = bf16(std * N(0,1)) for element indices [offset, offset + n) of (seed, stream). */
void synth_normal_bf16(uint16_t* out, int64_t n, uint64_t seed, uint64_t stream, double stddev,
                       int64_t offset) {
    const uint64_t key = synth_key(seed, stream);
    const double two_pi = 6.283185307179586476925286766559;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        uint64_t z = mix64(key + (uint64_t)(offset + i) * 0x9E3779B97F4A7C15ull);
        double u1 = ((double)(z >> 32) + 1.0) * (1.0 / 4294967296.0);
        double u2 = (double)(z & 0xFFFFFFFFull) * (1.0 / 4294967296.0);
        double v = stddev * sqrt(-2.0 * log(u1)) * cos(two_pi * u2);
        out[i] = f32_to_bf16_rne((float)v);
    }
}

/* out[i] = bf16(value) for a constant fill (used for RMSNorm gains of 1.0). */
void synth_fill_bf16(uint16_t* out, int64_t n, double value) {
    uint16_t b = f32_to_bf16_rne((float)value);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = b;
}
