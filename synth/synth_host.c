/*
 * Seeded synthetic-input generator, host implementation (plain C, OpenMP).
 *
 * This module holds no arithmetic of the attention method. It only draws the
 * seeded inputs (q, K, V, dO and the additive structure of the workloads) so
 * that the CPU oracle and the CUDA path see bit-identical tensors. The device
 * implementation (synth_dev.cu) is written separately from the same published
 * definitions; a test cross-checks the two bit for bit.
 *
 * Definitions
 *   SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
 *   generators", OOPSLA 2014): the state advances by the odd constant
 *   GAMMA = 0x9E3779B97F4A7C15 per draw and each output is the state passed
 *   through the 64-bit finaliser mix64(). The n-th output (n >= 0) of a stream
 *   that starts in state s0 is therefore mix64(s0 + (n + 1) * GAMMA), which
 *   makes the generator counter-based: any element can be drawn on its own.
 *   A seed selects the starting state s0 = mix64(seed).
 *
 *   Irwin-Hall(12) standard normal: element e takes the outputs 3e, 3e+1, 3e+2
 *   of the stream, splits each into four 16-bit uniforms u_0..u_11 and returns
 *   x = (2 * sum(u) - 786420) / 2^17. The sum of twelve uniforms on
 *   {0..65535} has mean 393210 and variance 12 * (65536^2 - 1) / 12, so x has
 *   mean 0 and variance 1 - 2^-32; it is bounded by |x| <= 6. Every step is
 *   integer arithmetic followed by one exact scaling by a power of two, so the
 *   fp32 value is identical on every machine.
 *
 *   bf16 rounding: round-to-nearest-even of the fp32 bit pattern to its upper
 *   16 bits (IEEE 754 roundTiesToEven applied to an 8-bit significand). The
 *   inputs here are finite, so no NaN handling is needed.
 */
#include <stdint.h>
#include <stddef.h>
#include <string.h>

#define SYNTH_GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t synth_mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

static inline uint64_t synth_draw(uint64_t s0, uint64_t n) {
    return synth_mix64(s0 + (n + 1ULL) * SYNTH_GAMMA);
}

static inline float synth_ih12(uint64_t s0, uint64_t e) {
    uint32_t u = 0;
    for (uint64_t r = 0; r < 3; ++r) {
        uint64_t x = synth_draw(s0, 3ULL * e + r);
        u += (uint32_t)(x & 0xFFFFu) + (uint32_t)((x >> 16) & 0xFFFFu) +
             (uint32_t)((x >> 32) & 0xFFFFu) + (uint32_t)(x >> 48);
    }
    int32_t centred = (int32_t)(2u * u) - 786420;
    return (float)centred * (1.0f / 131072.0f);
}

static inline uint16_t synth_bf16_rne(float x) {
    uint32_t u;
    memcpy(&u, &x, 4);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

uint64_t synth_stream_start(uint64_t seed) { return synth_mix64(seed); }

/* Raw outputs n0 .. n0+count-1 of the stream that starts in state s0 (used by tests). */
void synth_draws_state(uint64_t s0, uint64_t n0, int64_t count, uint64_t* out) {
    for (int64_t i = 0; i < count; ++i) out[i] = synth_draw(s0, n0 + (uint64_t)i);
}

/* Raw 64-bit draws n0 .. n0+count-1 of the stream for `seed` (used by tests). */
void synth_draws(uint64_t seed, uint64_t n0, int64_t count, uint64_t* out) {
    uint64_t s0 = synth_mix64(seed);
    for (int64_t i = 0; i < count; ++i) out[i] = synth_draw(s0, n0 + (uint64_t)i);
}

/*
 * Fill a box of a row-major 4-D tensor of logical shape dims[0..3] whose
 * element with flat index f is ih12(seed, f). The box is lo[k] <= i_k < hi[k];
 * out receives it densely in row-major order. fp32 values (exact) or their
 * bf16 rounding.
 */
static void synth_box_impl(uint64_t seed, const int64_t* dims, const int64_t* lo,
                           const int64_t* hi, float* out_f32, uint16_t* out_bf16) {
    uint64_t s0 = synth_mix64(seed);
    int64_t n0 = hi[0] - lo[0], n1 = hi[1] - lo[1], n2 = hi[2] - lo[2], n3 = hi[3] - lo[3];
    if (n0 <= 0 || n1 <= 0 || n2 <= 0 || n3 <= 0) return;
    int64_t rows = n0 * n1 * n2;
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; ++r) {
        int64_t i2 = r % n2, i1 = (r / n2) % n1, i0 = r / (n1 * n2);
        int64_t base = (((lo[0] + i0) * dims[1] + (lo[1] + i1)) * dims[2] + (lo[2] + i2)) * dims[3] + lo[3];
        for (int64_t i3 = 0; i3 < n3; ++i3) {
            float v = synth_ih12(s0, (uint64_t)(base + i3));
            if (out_f32) out_f32[r * n3 + i3] = v;
            if (out_bf16) out_bf16[r * n3 + i3] = synth_bf16_rne(v);
        }
    }
}

void synth_box_f32(uint64_t seed, const int64_t* dims, const int64_t* lo, const int64_t* hi, float* out) {
    synth_box_impl(seed, dims, lo, hi, out, NULL);
}

void synth_box_bf16(uint64_t seed, const int64_t* dims, const int64_t* lo, const int64_t* hi, uint16_t* out) {
    synth_box_impl(seed, dims, lo, hi, NULL, out);
}

/* x[i] <- bf16_rne(float(x[i]) + add[i]) for a dense array (one fp32 add each). */
void synth_add_f32_to_bf16(uint16_t* x, const float* add, int64_t n) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        uint32_t u = (uint32_t)x[i] << 16;
        float f;
        memcpy(&f, &u, 4);
        x[i] = synth_bf16_rne(f + add[i]);
    }
}

/* Exact widening of bf16 bit patterns to fp64 (every bf16 value is a double). */
void synth_bf16_to_f64(const uint16_t* x, double* out, int64_t n) {
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        uint32_t u = (uint32_t)x[i] << 16;
        float f;
        memcpy(&f, &u, 4);
        out[i] = (double)f;
    }
}
