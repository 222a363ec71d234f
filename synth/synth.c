/*
 * Seeded, counter-based generator of the synthetic inputs shared by the CPU oracle and the
 * GPU path. It holds none of the draft path's arithmetic: it only turns
 * (seed, tensor id, element index) into numbers with a stated distribution, so any slice of a
 * tensor can be regenerated on its own, in any order and on any number of threads.
 *
 * Uniform stream: SplitMix64 (S. Vigna, "Further scramblings of Marsaglia's xorshift
 * generators", and the public-domain splitmix64.c). Element i of stream `key` is
 * mix(key + (i + 1) * 0x9E3779B97F4A7C15), i.e. the (i+1)-th output of a SplitMix64 seeded
 * with `key`. The top 53 bits give a double in (0, 1).
 * Normals: Box-Muller (Box and Muller, 1958) on uniforms 2i and 2i+1 of the stream.
 * bf16 outputs are round-to-nearest-even of the float32 value.
 */
#include <math.h>
#include <stdint.h>

#define GOLDEN 0x9E3779B97F4A7C15ull

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static inline uint64_t stream_key(uint64_t seed, uint64_t tensor_id) {
    return mix64(mix64(seed + GOLDEN) ^ (tensor_id * 0xD1B54A32D192ED03ull));
}

static inline uint64_t bits_at(uint64_t key, uint64_t i) { return mix64(key + (i + 1) * GOLDEN); }

static inline double u01_at(uint64_t key, uint64_t i) {
    return ((double)(bits_at(key, i) >> 11) + 0.5) * (1.0 / 9007199254740992.0);
}

static inline double normal_at(uint64_t key, uint64_t i) {
    const double two_pi = 6.283185307179586476925286766559;
    double u1 = u01_at(key, 2 * i), u2 = u01_at(key, 2 * i + 1);
    return sqrt(-2.0 * log(u1)) * cos(two_pi * u2);
}

static inline uint16_t f32_to_bf16_rne(float f) {
    union { float f; uint32_t u; } v;
    v.f = f;
    if ((v.u & 0x7F800000u) == 0x7F800000u) return (uint16_t)((v.u >> 16) | ((v.u & 0xFFFF) ? 0x40 : 0));
    uint32_t lsb = (v.u >> 16) & 1u;
    return (uint16_t)((v.u + 0x7FFFu + lsb) >> 16);
}

/* out[k] = mean + std * N(0,1)[offset + k] as float32 */
void synth_normal_f32(uint64_t seed, uint64_t tensor_id, uint64_t offset, int64_t n,
                      double mean, double std, float* out) {
    uint64_t key = stream_key(seed, tensor_id);
#pragma omp parallel for schedule(static)
    for (int64_t k = 0; k < n; ++k) out[k] = (float)(mean + std * normal_at(key, offset + (uint64_t)k));
}

/* out[k] = bf16 bits of (float)(mean + std * N(0,1)[offset + k]) */
void synth_normal_bf16(uint64_t seed, uint64_t tensor_id, uint64_t offset, int64_t n,
                       double mean, double std, uint16_t* out) {
    uint64_t key = stream_key(seed, tensor_id);
#pragma omp parallel for schedule(static)
    for (int64_t k = 0; k < n; ++k)
        out[k] = f32_to_bf16_rne((float)(mean + std * normal_at(key, offset + (uint64_t)k)));
}

/* out[k] = U(0,1)[offset + k] as double */
void synth_uniform_f64(uint64_t seed, uint64_t tensor_id, uint64_t offset, int64_t n, double* out) {
    uint64_t key = stream_key(seed, tensor_id);
#pragma omp parallel for schedule(static)
    for (int64_t k = 0; k < n; ++k) out[k] = u01_at(key, offset + (uint64_t)k);
}

/* out[k] = top 32 bits of stream element offset + k (a uniform uint32) */
void synth_uniform_u32(uint64_t seed, uint64_t tensor_id, uint64_t offset, int64_t n, uint32_t* out) {
    uint64_t key = stream_key(seed, tensor_id);
#pragma omp parallel for schedule(static)
    for (int64_t k = 0; k < n; ++k) out[k] = (uint32_t)(bits_at(key, offset + (uint64_t)k) >> 32);
}

/* out[k] = lo + floor(U(0,1)[offset + k] * (hi - lo)), an integer in [lo, hi) */
void synth_randint_i32(uint64_t seed, uint64_t tensor_id, uint64_t offset, int64_t n,
                       int64_t lo, int64_t hi, int32_t* out) {
    uint64_t key = stream_key(seed, tensor_id);
    double span = (double)(hi - lo);
#pragma omp parallel for schedule(static)
    for (int64_t k = 0; k < n; ++k) {
        int64_t v = lo + (int64_t)floor(u01_at(key, offset + (uint64_t)k) * span);
        if (v >= hi) v = hi - 1;
        out[k] = (int32_t)v;
    }
}
