/*
 * Seeded synthetic inputs for the emulated GEMM workloads.
 *
 * This module holds no arithmetic of the emulation method: it only turns a
 * seed and an element counter into matrix entries.  Both the CPU oracle and
 * the CUDA path receive the very same host buffers produced here.
 *
 * Generator: SplitMix64 (G. Steele, D. Lea, C. Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014), used as a counter-based
 * generator: the i-th draw of stream `seed` is mix(seed + (i + 1) * gamma),
 * gamma = 0x9e3779b97f4a7c15.  Matrix A is filled row-major first, then B
 * continues the same stream (the caller passes the running counter offset).
 *
 * Distributions (the paper's input classes, Section 6.3):
 *   uniform_f64 : x = 2 * (r >> 11) * 2^-53 - 1            (U[-1,1), exact)
 *   uniform_f32 : x = 2 * (r >> 40) * 2^-24 - 1            (U[-1,1), exact in FP32)
 *   scaled_f64  : x = (u - 0.5) * exp(phi * g), u ~ U(0,1), g ~ N(0,1) by
 *                 Box-Muller, clamped into the BF16 exponent range (the
 *                 "scaled or log-uniform" class); three draws per element.
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>

#define SM64_GAMMA 0x9e3779b97f4a7c15ULL

static inline uint64_t sm64_at(uint64_t seed, uint64_t i)
{
    uint64_t z = seed + (i + 1ULL) * SM64_GAMMA;
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

uint64_t synth_splitmix64(uint64_t seed, uint64_t i) { return sm64_at(seed, i); }

void synth_uniform_f64(uint64_t seed, uint64_t offset, double *out, int64_t n)
{
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        uint64_t r = sm64_at(seed, offset + (uint64_t)i);
        out[i] = 2.0 * ldexp((double)(r >> 11), -53) - 1.0;
    }
}

void synth_uniform_f32(uint64_t seed, uint64_t offset, float *out, int64_t n)
{
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        uint64_t r = sm64_at(seed, offset + (uint64_t)i);
        out[i] = (float)(2.0 * ldexp((double)(r >> 40), -24) - 1.0);
    }
}

/* (u - 0.5) * exp(phi * g), clamped: nonzero |x| is kept inside
 * [2^-126, (2 - 2^-7) * 2^127]; zero stays zero. */
void synth_scaled_f64(uint64_t seed, uint64_t offset, double phi, double *out, int64_t n)
{
    const double two_pi = 6.283185307179586476925286766559;
    const double lo = ldexp(1.0, -126);
    const double hi = ldexp(2.0 - ldexp(1.0, -7), 127);
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        uint64_t c = 3ULL * (offset + (uint64_t)i);
        double u = ldexp((double)(sm64_at(seed, c) >> 11), -53);
        double u1 = ldexp((double)((sm64_at(seed, c + 1) >> 11) + 1ULL), -53); /* (0,1] */
        double u2 = ldexp((double)(sm64_at(seed, c + 2) >> 11), -53);
        double g = sqrt(-2.0 * log(u1)) * cos(two_pi * u2);
        double x = (u - 0.5) * exp(phi * g);
        if (x != 0.0) {
            double a = fabs(x);
            if (a < lo) a = lo;
            if (a > hi) a = hi;
            x = copysign(a, x);
        }
        out[i] = x;
    }
}
