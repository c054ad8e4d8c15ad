/* Bulk draws of the seeded input generator (ckv_synth): the counter-based SplitMix64 stream
 * and Box-Muller normals, rounded to bfloat16, with OpenMP over the draws.  The Python module
 * defines the same stream in numpy (uniform_u64); this file only makes the large tensors
 * (keys and values of long prefixes) fast to draw.  It holds none of the compression method's
 * arithmetic.
 *
 * Draw i (0-based) of stream `key` is the SplitMix64 finaliser (Steele, Lea & Flood, OOPSLA
 * 2014) of key + (i + 1) * 0x9E3779B97F4A7C15 (mod 2^64).  Normal pair p takes draw p: the
 * high and low 32-bit halves give u1, u2 = (half + 0.5) / 2^32, and the pair is
 * (r cos a, r sin a) with r = sqrt(-2 ln u1), a = 2 pi u2, computed in double and rounded to
 * float32.  Rounding the double result first to float32 and then to bfloat16 (nearest, ties
 * to even) makes the bits the same on every machine except where two libm results straddle a
 * rounding boundary, which has a probability of about 2^-40 per value.
 */
#include <math.h>
#include <stdint.h>

#define GOLDEN 0x9E3779B97F4A7C15ull

static inline uint64_t draw(uint64_t key, uint64_t i) {
    uint64_t z = (i + 1) * GOLDEN + key;
    z ^= z >> 30;
    z *= 0xBF58476D1CE4E5B9ull;
    z ^= z >> 27;
    z *= 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z;
}

static inline void normal_pair(uint64_t z, float* a, float* b) {
    const double inv32 = 1.0 / 4294967296.0;
    const double u1 = ((double)(z >> 32) + 0.5) * inv32;
    const double u2 = ((double)(z & 0xFFFFFFFFull) + 0.5) * inv32;
    const double r = sqrt(-2.0 * log(u1));
    const double ang = 6.283185307179586 * u2;
    *a = (float)(r * cos(ang));
    *b = (float)(r * sin(ang));
}

static inline uint16_t bf16_rne(float f) {
    union {
        float f;
        uint32_t u;
    } x;
    x.f = f;
    const uint32_t r = ((x.u >> 16) & 1u) + 0x7FFFu;
    return (uint16_t)((x.u + r) >> 16);
}

/* out[0..count): draws start .. start+count-1 of the stream. */
void synth_u64(uint64_t key, int64_t start, int64_t count, uint64_t* out) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < count; ++i) out[i] = draw(key, (uint64_t)(start + i));
}

/* out[0..count): the first `count` normals of the stream, as float32. */
void synth_normals_f32(uint64_t key, int64_t count, float* out) {
    const int64_t pairs = (count + 1) / 2;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < pairs; ++p) {
        float a, b;
        normal_pair(draw(key, (uint64_t)p), &a, &b);
        out[2 * p] = a;
        if (2 * p + 1 < count) out[2 * p + 1] = b;
    }
}

/* out[0..count): the first `count` normals of the stream, each multiplied in float32 by
 * scale[i % period] (no scaling when scale is NULL), rounded to bfloat16 bits. */
void synth_normals_bf16(uint64_t key, int64_t count, const float* scale, int64_t period,
                        uint16_t* out) {
    const int64_t pairs = (count + 1) / 2;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < pairs; ++p) {
        float v[2];
        normal_pair(draw(key, (uint64_t)p), &v[0], &v[1]);
        for (int e = 0; e < 2; ++e) {
            const int64_t i = 2 * p + e;
            if (i >= count) break;
            float x = v[e];
            if (scale) x *= scale[i % period];
            out[i] = bf16_rne(x);
        }
    }
}
