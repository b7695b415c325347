/*
 * aio_synth.c -- seeded, counter-based synthetic input generator.
 *
 * Serves both the CUDA path (via host buffers copied to the device) and the
 * fp64 oracle.  It holds none of the linear-layer arithmetic: it only turns
 * (key, element index) into input bytes, so any element of any tensor can be
 * regenerated on its own (random access), independent of thread count.
 *
 * Definitions (all integer steps are exact; the float steps use libm and the
 * default round-to-nearest-even mode of the host):
 *
 *   splitmix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
 *   generators", OOPSLA 2014; the constants are the published ones):
 *     state += 0x9E3779B97F4A7C15
 *     z = state
 *     z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9
 *     z = (z ^ (z >> 27)) * 0x94D049BB133111EB
 *     return z ^ (z >> 31)
 *
 *   bits(key, i)     = splitmix64 output for state = key + i * 0x9E3779B97F4A7C15
 *                      (i.e. the (i+1)-th output of a splitmix64 stream seeded by key)
 *   unit53(b)        = (b >> 11) * 2^-53                      in [0, 1)
 *   normal(key, i)   : Box-Muller on the pair p = i >> 1:
 *                        u1 = ((bits(key,2p) >> 11) + 1) * 2^-53   in (0, 1]
 *                        u2 = unit53(bits(key, 2p+1))
 *                        r  = sqrt(-2 ln u1), th = 2 pi u2
 *                        even i -> r cos th, odd i -> r sin th   (double)
 *   bf16(v)          : double -> float (RNE) -> bf16 (RNE on the upper 16 bits)
 *   code_i8(key, i)  = floor(hi32(bits(key,i)) * 255 / 2^32) - 127, uniform on [-127, 127]
 *   uniform(key,i,lo,hi) = lo + (hi - lo) * unit53(bits(key, i))   (double)
 *
 *   key(seed, a, b, c) = splitmix64 chain: h = sm(seed); h = sm(h ^ a); h = sm(h ^ b); h = sm(h ^ c)
 *   where sm(v) is the splitmix64 output for state v.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>
#include <stddef.h>

#define GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t sm_mix(uint64_t state) {
    uint64_t z = state + GAMMA;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

static inline uint64_t bits_at(uint64_t key, uint64_t i) { return sm_mix(key + i * GAMMA); }

static inline uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return (uint16_t)((u >> 16) | 0x0040u); /* quiet NaN */
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static inline uint16_t d_to_bf16(double v) { return f32_to_bf16_rne((float)v); }

uint64_t aio_synth_splitmix64(uint64_t state) { return sm_mix(state); }

uint64_t aio_synth_key(uint64_t seed, uint64_t a, uint64_t b, uint64_t c) {
    uint64_t h = sm_mix(seed);
    h = sm_mix(h ^ a);
    h = sm_mix(h ^ b);
    h = sm_mix(h ^ c);
    return h;
}

uint64_t aio_synth_bits(uint64_t key, uint64_t i) { return bits_at(key, i); }

static inline void box_muller(uint64_t key, uint64_t p, double* z0, double* z1) {
    const double two53 = 1.0 / 9007199254740992.0; /* 2^-53 */
    double u1 = (double)((bits_at(key, 2 * p) >> 11) + 1) * two53;
    double u2 = (double)(bits_at(key, 2 * p + 1) >> 11) * two53;
    double r = sqrt(-2.0 * log(u1));
    double th = 6.283185307179586476925286766559 * u2;
    *z0 = r * cos(th);
    *z1 = r * sin(th);
}

double aio_synth_normal_at(uint64_t key, uint64_t i) {
    double z0, z1;
    box_muller(key, i >> 1, &z0, &z1);
    return (i & 1) ? z1 : z0;
}

uint16_t aio_synth_f32_to_bf16(float f) { return f32_to_bf16_rne(f); }

/* out[j] = bf16(sigma * normal(key, offset + j)), j in [0, n) */
void aio_synth_normal_bf16(uint64_t key, double sigma, uint64_t offset, uint64_t n, uint16_t* out) {
    if (n == 0) return;
    /* handle a leading odd element so the main loop walks whole pairs */
    uint64_t j = 0;
    if (offset & 1) {
        out[0] = d_to_bf16(sigma * aio_synth_normal_at(key, offset));
        j = 1;
    }
    uint64_t npairs = (n - j) / 2;
    long long P = (long long)npairs;
#pragma omp parallel for schedule(static)
    for (long long q = 0; q < P; ++q) {
        uint64_t e = offset + j + 2 * (uint64_t)q; /* even element index */
        double z0, z1;
        box_muller(key, e >> 1, &z0, &z1);
        out[j + 2 * q] = d_to_bf16(sigma * z0);
        out[j + 2 * q + 1] = d_to_bf16(sigma * z1);
    }
    uint64_t done = j + 2 * npairs;
    if (done < n) out[done] = d_to_bf16(sigma * aio_synth_normal_at(key, offset + done));
}

/* out[j] = int8 code uniform on [-127, 127] for element offset + j */
void aio_synth_codes_i8(uint64_t key, uint64_t offset, uint64_t n, int8_t* out) {
    long long N = (long long)n;
#pragma omp parallel for schedule(static)
    for (long long j = 0; j < N; ++j) {
        uint64_t hi = bits_at(key, offset + (uint64_t)j) >> 32;
        out[j] = (int8_t)((int)((hi * 255ULL) >> 32) - 127);
    }
}

/* out[j] = bf16(lo + (hi - lo) * unit53(bits(key, offset + j))) */
void aio_synth_uniform_bf16(uint64_t key, double lo, double hi, uint64_t offset, uint64_t n, uint16_t* out) {
    const double two53 = 1.0 / 9007199254740992.0;
    long long N = (long long)n;
#pragma omp parallel for schedule(static)
    for (long long j = 0; j < N; ++j) {
        double u = (double)(bits_at(key, offset + (uint64_t)j) >> 11) * two53;
        out[j] = d_to_bf16(lo + (hi - lo) * u);
    }
}
