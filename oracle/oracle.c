/*
 * ORACLE -- test infrastructure, not part of the product.
 *
 * A plain, slow, CPU-only restatement of the BF16 component-product GEMM
 * emulation of arXiv 2609.04663 ("BF16 Component-Product Emulation of FP32 and
 * FP64 GEMM on Intel AMX").  It exists only to check the CUDA path: tests/,
 * __graft_entry__.smoke() and bench.py's CPU-baseline / reference leg are the
 * only callers.  It shares no code with the CUDA library.
 *
 * Build: gcc -O2 -ffp-contract=off -fopenmp (no fast-math), so every fl32 /
 * fl64 of the paper is exactly one IEEE-754 operation in the stated format and
 * nothing is contracted into an FMA or reassociated.  OpenMP only splits
 * independent output elements (or independent input entries) between threads;
 * it never changes the order of any floating-point sum.
 *
 * Layouts (all row-major, dense):
 *   A planes  [s][M][K]  BF16 bit patterns (uint16), slice r at offset r*M*K
 *   B planes  [s][K][N]  BF16 bit patterns
 *   C         [nrows][N] rows r0 .. r0+nrows-1 of the product
 *
 * Readings of points the paper leaves open (each also listed in the design notes):
 *   - fl_BF16 rounds to nearest, ties to even, with BF16 subnormals and
 *     overflow to infinity (Section 4.2 says "round-to-nearest").
 *   - v^(r) of Eq. (fp64split) is one scalar per operand and level: the max is
 *     taken over the whole matrix, as the equation is written.
 *   - K-chunk = B_K = 256 (Section 6.1); the last chunk may be shorter.
 *   - FP32 mode: inside one chunk the six products are interleaved per 32-wide
 *     K step in the operand-reuse order of Eq. (fp32reuseorder), one FP32
 *     accumulator per chunk, chunk results added into an FP32 output
 *     accumulator (Section 6.3, reconstruction of the FP32 path).
 *   - FP64 mode, two summation orders of the same exact FP32 chunk partials:
 *     ORDER_CHUNK_OUTER: chunk outer, products inner in diagonal order (l
 *       ascending, i ascending within a diagonal), each partial widened and
 *       added in FP64 (the per-panel reconstruction of Section 6.3);
 *     ORDER_PRODUCT_OUTER: products in diagonal order outer, as Algorithm 2
 *       is written (C <- fl64(C + fl32(A_i B_j))): the FP32 component product
 *       is formed per K-chunk and its chunk partials are summed exactly (they
 *       are integers in one unit, see oracle_prodsum_f64), then added once.
 */
#include <float.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_FLAG_NONFINITE 0x1u /* a non-finite input entry            */
#define ORACLE_FLAG_RANGE     0x2u /* FP64 entry outside F64^B, Eq. (bf16rangefp64) */
#define ORACLE_FLAG_SLICE     0x4u /* a slice is not a normal BF16 value (or is non-finite) */

#define ORACLE_ZERO_LEVEL INT32_MIN /* v^(r) of an all-zero residual */
#define ORACLE_ORDER_CHUNK_OUTER 0
#define ORACLE_ORDER_PRODUCT_OUTER 1
#define ORACLE_KCHUNK 256           /* B_K of Section 6.1 */

/* ------------------------------------------------------------------------ */
/* fl_BF16 (Section 4.2): keep an 8-bit significand (implicit bit included), */
/* round to nearest, ties to even.  Written from the definition: find the    */
/* binade, scale to an integer significand, round, scale back.               */
/* ------------------------------------------------------------------------ */
uint16_t oracle_fl_bf16(double x)
{
    if (isnan(x)) return 0x7FC0u;
    uint16_t sign = signbit(x) ? 0x8000u : 0u;
    double a = fabs(x);
    if (a == 0.0) return sign;
    if (isinf(a)) return (uint16_t)(sign | 0x7F80u);
    int e;
    (void)frexp(a, &e);          /* a = f * 2^e, f in [0.5, 1)            */
    int E = e - 1;               /* a = (2f) * 2^E, 2f in [1, 2)           */
    if (E < -126) E = -126;      /* below the normal range: fixed quantum  */
    double q = ldexp(1.0, E - 7);           /* spacing of 8-bit significands */
    double n = nearbyint(a / q);            /* a/q is exact; RNE to integer  */
    double r = n * q;                       /* rounded magnitude, exact      */
    if (r >= ldexp(1.0, 128)) return (uint16_t)(sign | 0x7F80u); /* overflow */
    if (r == 0.0) return sign;
    if (r < ldexp(1.0, -126)) {              /* BF16 subnormal: n * 2^-133   */
        return (uint16_t)(sign | (uint16_t)(r / ldexp(1.0, -133)));
    }
    (void)frexp(r, &e);
    int Er = e - 1;                          /* r = m * 2^Er, m in [1, 2)     */
    int frac = (int)((r / ldexp(1.0, Er) - 1.0) * 128.0); /* exact, 0..127 */
    return (uint16_t)(sign | (uint16_t)((Er + 127) << 7) | (uint16_t)frac);
}

/* Exact real value of a stored BF16 number, as a double. */
double oracle_bf16_value(uint16_t b)
{
    int s = (b >> 15) & 1, ex = (b >> 7) & 0xFF, fr = b & 0x7F;
    double v;
    if (ex == 0xFF) v = fr ? NAN : INFINITY;
    else if (ex == 0) v = ldexp((double)fr, -133);
    else v = ldexp(1.0 + fr / 128.0, ex - 127);
    return s ? -v : v;
}

/* ceil(log2(m)) for m > 0, via frexp: m = f * 2^e, f in [0.5, 1).          */
int oracle_ceil_log2(double m)
{
    int e;
    double f = frexp(m, &e);
    return (f == 0.5) ? e - 1 : e;
}

/* ------------------------------------------------------------------------ */
/* FP32 three-component split, Eq. (fp32split), Algorithm 1 (Split_FP32):   */
/*   A_r = fl_BF16(A^(r)),  A^(r+1) = fl32(A^(r) - A_r),  r = 0, 1, 2.      */
/* planes: [3][rows][cols].                                                 */
/* ------------------------------------------------------------------------ */
uint32_t oracle_split_f32(const float *X, int64_t rows, int64_t cols, int64_t ldx,
                          uint16_t *planes)
{
    uint32_t flags = 0;
    const int64_t plane = rows * cols;
    #pragma omp parallel for schedule(static) reduction(|:flags)
    for (int64_t i = 0; i < rows; ++i) {
        for (int64_t j = 0; j < cols; ++j) {
            float a = X[i * ldx + j];               /* A^(0) */
            if (!isfinite(a)) flags |= ORACLE_FLAG_NONFINITE;
            for (int r = 0; r < 3; ++r) {
                uint16_t s = oracle_fl_bf16((double)a);
                planes[r * plane + i * cols + j] = s;
                float sv = (float)oracle_bf16_value(s);   /* exact */
                if (!isfinite(sv)) flags |= ORACLE_FLAG_SLICE;
                a = a - sv;                          /* fl32 subtraction */
            }
        }
    }
    return flags;
}

/* ------------------------------------------------------------------------ */
/* FP64 fixed six-slice simplified Ozaki split, Eq. (fp64split), Alg. 2:    */
/*   v^(r) = ceil(log2(max_ij |A^(r)_ij|))                                   */
/*   Z^(r) = fl64(fl64(A^(r) + 2^(v+rho)) - 2^(v+rho)),  rho = 45            */
/*   A_r   = fl_BF16(Z^(r)),   A^(r+1) = fl64(A^(r) - A_r),   r = 0..5        */
/* An all-zero residual ends the split: its slice and all later ones are 0  */
/* and their v is reported as ORACLE_ZERO_LEVEL.  planes: [6][rows][cols].  */
/* Domain, Eq. (bf16rangefp64): x = 0 or 2^-126 <= |x| <= (2-2^-7) 2^127;    */
/* a slice must be a normal BF16 value equal to Z (Section 4.3).            */
/* ------------------------------------------------------------------------ */
uint32_t oracle_split_f64(const double *X, int64_t rows, int64_t cols, int64_t ldx,
                          uint16_t *planes, int32_t *v)
{
    uint32_t flags = 0;
    const int64_t plane = rows * cols;
    const double lo = ldexp(1.0, -126), hi = ldexp(2.0 - ldexp(1.0, -7), 127);
    double *R = (double *)malloc((size_t)(plane > 0 ? plane : 1) * sizeof(double));
    if (!R) return 0xFFFFFFFFu;

    #pragma omp parallel for schedule(static) reduction(|:flags)
    for (int64_t i = 0; i < rows; ++i)
        for (int64_t j = 0; j < cols; ++j) {
            double x = X[i * ldx + j];
            R[i * cols + j] = x;                            /* A^(0) = A */
            if (!isfinite(x)) flags |= ORACLE_FLAG_NONFINITE;
            else if (x != 0.0 && (fabs(x) < lo || fabs(x) > hi)) flags |= ORACLE_FLAG_RANGE;
        }

    int r = 0;
    for (; r < 6; ++r) {
        double m = 0.0;
        #pragma omp parallel for schedule(static) reduction(max:m)
        for (int64_t e = 0; e < plane; ++e) {
            double a = fabs(R[e]);
            if (a > m) m = a;                               /* NaN never wins */
        }
        if (m == 0.0) break;                                 /* A^(r) = 0 */
        v[r] = oracle_ceil_log2(m);
        const double sigma = ldexp(1.0, v[r] + 45);
        uint16_t *P = planes + r * plane;
        #pragma omp parallel for schedule(static) reduction(|:flags)
        for (int64_t e = 0; e < plane; ++e) {
            double t = R[e] + sigma;                         /* fl64 */
            double Z = t - sigma;                            /* fl64 */
            uint16_t s = oracle_fl_bf16(Z);
            double sv = oracle_bf16_value(s);
            if (sv != Z || (Z != 0.0 && fabs(Z) < lo) || !isfinite(sv)) flags |= ORACLE_FLAG_SLICE;
            P[e] = s;
            R[e] = R[e] - sv;                                /* fl64 */
        }
    }
    for (; r < 6; ++r) {
        v[r] = ORACLE_ZERO_LEVEL;
        memset(planes + r * plane, 0, (size_t)plane * sizeof(uint16_t));
    }
    free(R);
    return flags;
}

/* ------------------------------------------------------------------------ */
/* Product sets and executed orders.                                        */
/*   S_d = {(i,j): i + j < d}, N_p(d) = |S_d|, Eq. (product-selection);      */
/*   FP32: d = 3 in the operand-reuse order of Eq. (fp32reuseorder);         */
/*   FP64: N_p(3,4,5,6) = 6, 10, 15, 21, Eq. (fp64productcounts), executed   */
/*         diagonal by diagonal (Algorithm 2), i ascending in a diagonal.    */
/* Writes pairs[2q], pairs[2q+1] = (i_q, j_q); returns the count or -1.     */
/* ------------------------------------------------------------------------ */
int oracle_products(int mode, int nprod, int *pairs)
{
    if (mode == 32) {
        static const int chain[6][2] = {{1, 1}, {1, 0}, {2, 0}, {0, 0}, {0, 1}, {0, 2}};
        if (nprod != 6) return -1;
        for (int q = 0; q < 6; ++q) { pairs[2 * q] = chain[q][0]; pairs[2 * q + 1] = chain[q][1]; }
        return 6;
    }
    int d;
    switch (nprod) { case 6: d = 3; break; case 10: d = 4; break;
                     case 15: d = 5; break; case 21: d = 6; break; default: return -1; }
    int q = 0;
    for (int l = 0; l < d; ++l)
        for (int i = 0; i <= l; ++i) { pairs[2 * q] = i; pairs[2 * q + 1] = l - i; ++q; }
    return q;
}

static float bf16f(uint16_t b) { return (float)oracle_bf16_value(b); }

/* Expand BF16 planes of A rows [r0, r0+nr) to float; and B to [s][N][K] float
 * (a transposed copy, so that a dot product walks contiguous memory; the
 * arithmetic and its order are unchanged by this layout). */
static float *expand_a(const uint16_t *Ap, int s, int64_t M, int64_t K, int64_t r0, int64_t nr)
{
    float *a = (float *)malloc((size_t)s * nr * K * sizeof(float) + 1);
    for (int t = 0; t < s; ++t)
        for (int64_t i = 0; i < nr; ++i)
            for (int64_t k = 0; k < K; ++k)
                a[(t * nr + i) * K + k] = bf16f(Ap[t * M * K + (r0 + i) * K + k]);
    return a;
}

static float *expand_bt(const uint16_t *Bp, int s, int64_t K, int64_t N)
{
    float *b = (float *)malloc((size_t)s * N * K * sizeof(float) + 1);
    #pragma omp parallel for schedule(static)
    for (int64_t n = 0; n < N; ++n)
        for (int t = 0; t < s; ++t)
            for (int64_t k = 0; k < K; ++k)
                b[(t * N + n) * K + k] = bf16f(Bp[t * K * N + k * N + n]);
    return b;
}

/* ------------------------------------------------------------------------ */
/* FP32-mode product-sum, Eq. (fp32six) with the blocked FP32 reconstruction */
/* of Section 6.3: per K-chunk an FP32 accumulator takes the six products    */
/* (interleaved per 32-wide step, Eq. (fp32reuseorder)); each chunk result   */
/* is added into the FP32 output accumulator.  Every product of two BF16    */
/* values is exact in FP32 (Section 5.2); only the additions round.         */
/* ------------------------------------------------------------------------ */
void oracle_prodsum_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                        int64_t r0, int64_t nr, float *C)
{
    int pairs[12];
    oracle_products(32, 6, pairs);
    float *a = expand_a(Ap, 3, M, K, r0, nr);
    float *b = expand_bt(Bp, 3, K, N);
    #pragma omp parallel for collapse(2) schedule(dynamic, 16)
    for (int64_t i = 0; i < nr; ++i) {
        for (int64_t n = 0; n < N; ++n) {
            float c32 = 0.0f;
            for (int64_t c0 = 0; c0 < K; c0 += ORACLE_KCHUNK) {
                const int64_t c1 = (c0 + ORACLE_KCHUNK < K) ? c0 + ORACLE_KCHUNK : K;
                float acc = 0.0f;
                for (int64_t k0 = c0; k0 < c1; k0 += 32) {
                    const int64_t k1 = (k0 + 32 < c1) ? k0 + 32 : c1;
                    for (int q = 0; q < 6; ++q) {
                        const float *ai = a + (pairs[2 * q] * nr + i) * K;
                        const float *bj = b + (pairs[2 * q + 1] * N + n) * K;
                        for (int64_t k = k0; k < k1; ++k) acc = acc + ai[k] * bj[k];
                    }
                }
                c32 = c32 + acc;
            }
            C[i * N + n] = c32;
        }
    }
    free(a);
    free(b);
}

/* ------------------------------------------------------------------------ */
/* FP64-mode product-sum, Eq. (fp64reconstruction), Algorithm 2.  Every      */
/* chunk partial P = fl32(sum_k A_i B_j) is formed in FP32 (k ascending).    */
/* Slices lie on the grid of Eq. (fp64split): integers times 2^(v-8) of     */
/* magnitude <= 256, so a BF16 product is <= 2^16 units and a 256-long chunk */
/* <= 2^24 units: P is exact (Section 5.2 extended to the chunk).            */
/*   order 0 (chunk outer): for chunk, for pair: C = fl64(C + (double)P).    */
/*   order 1 (product outer): for pair: S = sum over chunks of (double)P --  */
/*     exact in FP64, a sum of integers in one unit below 2^53 units -- then */
/*     C = fl64(C + S).                                                      */
/* If n_inexact is non-NULL each partial is also formed in FP64 and the     */
/* number of partials that differ is counted.                               */
/* ------------------------------------------------------------------------ */
void oracle_prodsum_f64(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                        int nprod, int order, int64_t r0, int64_t nr, double *C, int64_t *n_inexact)
{
    int pairs[42];
    const int np = oracle_products(64, nprod, pairs);
    if (np < 0) return;
    float *a = expand_a(Ap, 6, M, K, r0, nr);
    float *b = expand_bt(Bp, 6, K, N);
    const int64_t nch = (K + ORACLE_KCHUNK - 1) / ORACLE_KCHUNK;
    int64_t bad = 0;
    #pragma omp parallel for collapse(2) schedule(dynamic, 16) reduction(+:bad)
    for (int64_t i = 0; i < nr; ++i) {
        for (int64_t n = 0; n < N; ++n) {
            double c64 = 0.0;
            double s = 0.0;
            for (int64_t t = 0; t < nch * np; ++t) {
                const int64_t c = (order == ORACLE_ORDER_CHUNK_OUTER) ? t / np : t % nch;
                const int q = (int)((order == ORACLE_ORDER_CHUNK_OUTER) ? t % np : t / nch);
                const int64_t c0 = c * ORACLE_KCHUNK;
                const int64_t c1 = (c0 + ORACLE_KCHUNK < K) ? c0 + ORACLE_KCHUNK : K;
                const float *ai = a + (pairs[2 * q] * nr + i) * K;
                const float *bj = b + (pairs[2 * q + 1] * N + n) * K;
                float p = 0.0f;
                for (int64_t k = c0; k < c1; ++k) p = p + ai[k] * bj[k];
                if (n_inexact) {
                    double pd = 0.0;
                    for (int64_t k = c0; k < c1; ++k) pd = pd + (double)ai[k] * (double)bj[k];
                    if ((double)p != pd) ++bad;
                }
                if (order == ORACLE_ORDER_CHUNK_OUTER) {
                    c64 = c64 + (double)p;
                } else {
                    s = s + (double)p;                       /* exact */
                    if (c == nch - 1) { c64 = c64 + s; s = 0.0; }
                }
            }
            C[i * N + n] = c64;
        }
    }
    if (n_inexact) *n_inexact = bad;
    free(a);
    free(b);
}

/* ------------------------------------------------------------------------ */
/* Double-double reference product (for the accuracy metrics of Section 7.3, */
/* Eqs. (froerror), (scalederror)): sum_k A[m,k] B[k,n] with an error-free   */
/* product (TwoProd via fma) and error-free additions (TwoSum), Dekker/Knuth */
/* style.  Returns hi + lo per element, rows [r0, r0+nr).                    */
/* ------------------------------------------------------------------------ */
void oracle_ref_dd(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda,
                   const double *B, int64_t ldb, int64_t r0, int64_t nr, double *hi, double *lo)
{
    (void)M;
    double *bt = (double *)malloc((size_t)N * K * sizeof(double) + 1);
    #pragma omp parallel for schedule(static)
    for (int64_t n = 0; n < N; ++n)
        for (int64_t k = 0; k < K; ++k) bt[n * K + k] = B[k * ldb + n];
    #pragma omp parallel for collapse(2) schedule(dynamic, 16)
    for (int64_t i = 0; i < nr; ++i) {
        for (int64_t n = 0; n < N; ++n) {
            const double *ar = A + (r0 + i) * lda;
            const double *bc = bt + n * K;
            double sh = 0.0, sl = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                double p = ar[k] * bc[k];
                double pe = fma(ar[k], bc[k], -p);          /* TwoProd error */
                double s = sh + p;                           /* TwoSum(sh, p) */
                double bb = s - sh;
                double se = (sh - (s - bb)) + (p - bb);
                sl = sl + (se + pe);
                double t = s + sl;                           /* renormalise */
                sl = sl - (t - s);
                sh = t;
            }
            hi[i * N + n] = sh;
            lo[i * N + n] = sl;
        }
    }
    free(bt);
}
