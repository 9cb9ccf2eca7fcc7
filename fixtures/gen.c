/*
 * Seeded synthetic input generator shared by the test oracle and the GPU path.
 *
 * This file holds no arithmetic of the repair method: it only turns
 * (seed, stream, element index) into numbers.  Both sides of every parity
 * test receive the same bytes from here, so nothing the kernels compute can
 * leak into an oracle input.
 *
 * Generator (all published definitions, written out here):
 *   - SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number
 *     generators", OOPSLA 2014): the c-th output of a stream with start state
 *     `base` is mix64(base + (c + 1) * GAMMA).  Being counter based, any
 *     element can be produced independently, so generation is parallel and
 *     the value of an element never depends on how the work was split.
 *   - Uniform on (0,1): ((r >> 11) + 0.5) * 2^-53.
 *   - Standard normal: Box-Muller (Box & Muller 1958) on the uniform pair
 *     (U(2k), U(2k+1)); element i takes the cosine branch if i is even and
 *     the sine branch if odd, with k = i / 2.
 *   - float -> bfloat16: round to nearest even on the float bit pattern.
 *   - -0.0 is written as +0.0 so that "x + 0 == x" holds bit for bit.
 *
 * Plain C99 + OpenMP, no architecture-specific code: the same source builds
 * on x86-64 and aarch64 hosts.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

static inline uint64_t stream_base(uint64_t seed, uint64_t stream) {
    return mix64(seed * GAMMA ^ mix64(stream + 0x632BE59BD9B4E019ULL));
}

static inline uint64_t draw_bits(uint64_t base, uint64_t c) {
    return mix64(base + (c + 1ULL) * GAMMA);
}

static inline double draw_unit(uint64_t base, uint64_t c) {
    return ((double)(draw_bits(base, c) >> 11) + 0.5) * (1.0 / 9007199254740992.0);
}

static inline double draw_normal(uint64_t base, uint64_t i) {
    uint64_t k = i >> 1;
    double u1 = draw_unit(base, 2 * k);
    double u2 = draw_unit(base, 2 * k + 1);
    double r = sqrt(-2.0 * log(u1));
    double t = 6.283185307179586476925286766559 * u2;
    return (i & 1) ? r * sin(t) : r * cos(t);
}

static inline float no_negzero(float f) { return f == 0.0f ? 0.0f : f; }

static inline uint16_t f32_to_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return 0x7FC0;
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/* Raw 64-bit draws: out[i] = bits(seed, stream, offset + i). */
void fx_bits(uint64_t seed, uint64_t stream, uint64_t offset, int64_t n, uint64_t *out) {
    uint64_t base = stream_base(seed, stream);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = draw_bits(base, offset + (uint64_t)i);
}

/* Uniform draws in (0,1) as double. */
void fx_unit_f64(uint64_t seed, uint64_t stream, uint64_t offset, int64_t n, double *out) {
    uint64_t base = stream_base(seed, stream);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = draw_unit(base, offset + (uint64_t)i);
}

/*
 * Row-structured normal draws: element (r, j) of an [n_rows, width] block is
 *   scale * col_scale[j] * N(seed, stream, (row0 + r) * width + j)
 * rounded once to float (dtype 0) or to float then bfloat16 (dtype 1).
 * col_scale may be NULL (all ones).  `out` is n_rows * width elements.
 */
void fx_normal_rows(uint64_t seed, uint64_t stream, int64_t row0, int64_t n_rows,
                    int64_t width, double scale, const float *col_scale, int dtype,
                    void *out) {
    uint64_t base = stream_base(seed, stream);
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < n_rows; ++r) {
        uint64_t idx0 = (uint64_t)(row0 + r) * (uint64_t)width;
        for (int64_t j = 0; j < width; ++j) {
            double s = scale * (col_scale ? (double)col_scale[j] : 1.0);
            float f = no_negzero((float)(s * draw_normal(base, idx0 + (uint64_t)j)));
            if (dtype == 0)
                ((float *)out)[r * width + j] = f;
            else
                ((uint16_t *)out)[r * width + j] = f32_to_bf16(f);
        }
    }
}

/*
 * Symmetric uniform draws: out[i] = a * (2 U(seed, stream, i) - 1), rounded
 * once to float (dtype 0) or float then bfloat16 (dtype 1).  Used for
 * Xavier-uniform weights, a = sqrt(6 / (fan_in + fan_out)).
 */
void fx_uniform_sym(uint64_t seed, uint64_t stream, int64_t n, double a, int dtype, void *out) {
    uint64_t base = stream_base(seed, stream);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        float f = no_negzero((float)(a * (2.0 * draw_unit(base, (uint64_t)i) - 1.0)));
        if (dtype == 0)
            ((float *)out)[i] = f;
        else
            ((uint16_t *)out)[i] = f32_to_bf16(f);
    }
}

/* Round a float array to bfloat16 (round to nearest even). */
void fx_f32_to_bf16(const float *in, int64_t n, uint16_t *out) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = f32_to_bf16(no_negzero(in[i]));
}
