/*
 * Seeded synthetic-input core shared by the CPU oracle and the CUDA path.
 *
 * Holds no arithmetic of the allocation method or of the decoder: it only
 * turns (seed, stream, index) into random numbers.  The generator is
 * SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number
 * generators", OOPSLA 2014) used in counter mode: output number c of a stream
 * whose state starts at `s` is mix64(s + c * GOLDEN).  Normal deviates use the
 * Box-Muller transform (Box and Muller, 1958) in double precision.
 *
 * Built as a shared library by synth/__init__.py (gcc, -fopenmp).
 */
#include <math.h>
#include <stdint.h>

#define GOLDEN 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* Output number c (1-based) of SplitMix64 seeded with `seed`. */
uint64_t synth_splitmix64_at(uint64_t seed, uint64_t c) { return mix64(seed + c * GOLDEN); }

/* Round-to-nearest-even float -> bfloat16 bit pattern (inputs are finite). */
static inline uint16_t f32_to_bf16_rne(float f) {
    union { float f; uint32_t u; } v;
    v.f = f;
    uint32_t u = v.u;
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/*
 * out[i] = bf16(std * z_i), z_i standard normal, for i in [0, n).
 * Pair p = i/2 draws h1 = output 2p+1 and h2 = output 2p+2 of the stream
 * whose seed is output (stream+1) of SplitMix64(seed); even i takes
 * r*cos(theta), odd i takes r*sin(theta).
 */
void synth_fill_normal_bf16(uint64_t seed, uint64_t stream, uint64_t n, double std_dev,
                            uint16_t *out) {
    const uint64_t base = synth_splitmix64_at(seed, stream + 1);
    const int64_t npairs = (int64_t)((n + 1) / 2);
    const double two_pi = 6.283185307179586476925286766559;
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < npairs; ++p) {
        uint64_t h1 = mix64(base + (uint64_t)(2 * p + 1) * GOLDEN);
        uint64_t h2 = mix64(base + (uint64_t)(2 * p + 2) * GOLDEN);
        double u1 = ((double)(h1 >> 11) + 0.5) * 0x1.0p-53; /* (0,1) */
        double u2 = (double)(h2 >> 11) * 0x1.0p-53;         /* [0,1) */
        double r = sqrt(-2.0 * log(u1));
        double th = two_pi * u2;
        uint64_t i0 = (uint64_t)(2 * p);
        out[i0] = f32_to_bf16_rne((float)(std_dev * r * cos(th)));
        if (i0 + 1 < n) out[i0 + 1] = f32_to_bf16_rne((float)(std_dev * r * sin(th)));
    }
}

/* out[i] = bf16(value) for i in [0, n) (norm weights). */
void synth_fill_const_bf16(uint64_t n, float value, uint16_t *out) {
    uint16_t b = f32_to_bf16_rne(value);
    for (uint64_t i = 0; i < n; ++i) out[i] = b;
}
