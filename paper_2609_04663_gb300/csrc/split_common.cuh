// Shared pieces of the split kernels (split_f32.cu, split_f64.cu,
// split_rc.cu): tile constants, the FP64 rounding steps of Eq. (fp64split),
// the literal level passes, the plane rewrite, the verifier and its grid
// barrier, and the speculative per-element split.  Each translation unit
// that includes this gets its own copies (unnamed namespace).
#pragma once
#include "launchers.cuh"

#pragma nv_diag_suppress 177      // helpers a translation unit does not use

namespace emu {

namespace {

constexpr int kTile = 64;            // tile edge (elements)
constexpr int kSRow = kTile + 2;     // shared-memory row pitch in uint16 (odd word pitch)
constexpr int kThreads = 256;

// --------------------------------------------------------------- rounding
// fl_BF16 of an FP64 value, one rounding, by integer arithmetic on its bits:
// the BF16 quantum is 2^(max(e, -126) - 7) for a leading-bit exponent e;
// subnormal BF16 spacing 2^-133; overflow to infinity.
__device__ uint16_t bf16_rne_f64(double z)
{
    const uint64_t b = (uint64_t)__double_as_longlong(z);
    const uint16_t sign = (uint16_t)((b >> 48) & 0x8000u);
    const uint64_t a = b & 0x7FFFFFFFFFFFFFFFull;
    if (a > 0x7FF0000000000000ull) return 0x7FC0u;
    if (a == 0x7FF0000000000000ull) return (uint16_t)(sign | 0x7F80u);
    if (a == 0) return sign;
    int E = (int)(a >> 52);
    uint64_t m = a & 0x000FFFFFFFFFFFFFull;
    int e;                                        // exponent of the leading bit
    if (E) { m |= 1ull << 52; e = E - 1023; }
    else { E = 1; e = -1022 - (__clzll((long long)m) - 11); }
    const int qe = (e < -126 ? -126 : e) - 7;     // quantum exponent
    const int s = qe - (E - 1075);                // value = m * 2^(E-1075)
    uint64_t n;
    if (s <= 0) n = m << (-s);
    else if (s >= 64) n = 0;
    else {
        n = m >> s;
        const uint64_t rem = m & ((1ull << s) - 1ull), half = 1ull << (s - 1);
        if (rem > half || (rem == half && (n & 1ull))) ++n;
    }
    if (qe == -133) return (uint16_t)(sign | (uint16_t)n);   // subnormal (n <= 128)
    int ebits = qe + 7 + 127;
    if (n == 256) { n = 128; ++ebits; }
    if (ebits >= 255) return (uint16_t)(sign | 0x7F80u);
    return (uint16_t)(sign | (uint16_t)(ebits << 7) | (uint16_t)(n - 128));
}

__device__ __forceinline__ double pow2_d(int e)
{
    e = e < -1022 ? -1022 : (e > 1023 ? 1023 : e);
    return __longlong_as_double((long long)(e + 1023) << 52);
}

// ceil(log2(m)) for m > 0 given as the bit pattern of a non-negative double.
__device__ __host__ __forceinline__ int ceil_log2_bits(unsigned long long b)
{
    const int E = (int)(b >> 52) & 0x7FF;
    const unsigned long long f = b & 0x000FFFFFFFFFFFFFull;
    if (E == 0) {                                 // subnormal
#ifdef __CUDA_ARCH__
        const int msb = 63 - __clzll((long long)f);
#else
        const int msb = 63 - __builtin_clzll(f);
#endif
        return ((f & (f - 1)) == 0 ? msb : msb + 1) - 1074;
    }
    return (E - 1023) + (f != 0 ? 1 : 0);
}

// One level of Eq. (fp64split) for one entry: Z = (R + 2^(v+45)) - 2^(v+45)
// in FP64 round-to-nearest (no contraction), A_r = fl_BF16(Z),
// R <- R - A_r.  Sets *bad if A_r is not exactly Z or is a nonzero value
// below the normal BF16 range.
__device__ __forceinline__ uint16_t f64_level(double &R, int v, bool &bad)
{
    if (v == kZeroLevel) return 0;                // residual is zero here
    const double sigma = pow2_d(v + 45);
    const double Z = __dsub_rn(__dadd_rn(R, sigma), sigma);
    const float f = __double2float_rn(Z);
    const uint32_t fb = __float_as_uint(f);
    uint16_t s;
    if ((double)f == Z && (fb & 0xFFFFu) == 0u && (Z == 0.0 || (fb & 0x7F800000u) != 0u) &&
        (fb & 0x7F800000u) != 0x7F800000u) {
        s = (uint16_t)(fb >> 16);
    } else {
        bad = true;
        s = bf16_rne_f64(Z);
    }
    const double sv = (double)__uint_as_float((uint32_t)s << 16);
    R = __dsub_rn(R, sv);
    return s;
}

// The same level computed with integer operations only (GB300 runs FP64 at a
// small fraction of its integer rate).  It restates the projection exactly:
// for |R| <= 2^v, fl64(R + 2^(v+45)) lies in the binade above 2^(v+45) when
// R >= 0 (spacing 2^(v-7)) and in the binade below it when R < 0 (spacing
// 2^(v-8)), and the subtraction of 2^(v+45) is exact; so Z is R rounded to
// nearest, ties to even, on the grid G = 2^(v-7) or 2^(v-8): Z = sign * n * G
// with n <= 256.  R - Z is exact and is renormalised from the integer
// difference.  Values it cannot take this way (non-finite input, R not below
// 2^v, or Z outside the normal BF16 range) go through f64_level.
__device__ __noinline__ uint16_t f64_level_int(double &R, int v, bool &bad)
{
    if (v == kZeroLevel) return 0;
    const uint64_t b = (uint64_t)__double_as_longlong(R);
    const uint64_t a = b & 0x7FFFFFFFFFFFFFFFull;
    if (a == 0) return 0;                                      // Z = +0, R unchanged
    const uint32_t sgn = (uint32_t)(b >> 63);
    int E = (int)(a >> 52);
    if (E == 0x7FF) return f64_level(R, v, bad);
    uint64_t M = a & 0x000FFFFFFFFFFFFFull;
    if (E == 0) E = 1; else M |= 1ull << 52;                  // |R| = M * 2^(E - 1075)
    const int G = v - (sgn ? 8 : 7);                           // grid exponent
    const int sh = G - (E - 1075);
    if (sh <= 0 || sh > 60) {
        if (sh > 60) return 0;                                 // |R| < G / 2: Z = +0
        return f64_level(R, v, bad);
    }
    uint64_t n = M >> sh;
    const uint64_t rem = M & ((1ull << sh) - 1ull), half = 1ull << (sh - 1);
    if (rem > half || (rem == half && (n & 1ull))) ++n;
    if (n == 0) return 0;
    if (n > 256) return f64_level(R, v, bad);                 // |R| > 2^v: not this level's grid
    const int p = 31 - __clz((unsigned)n);                     // leading bit of n, 0..8
    const int ez = G + p;                                      // exponent of Z's leading bit
    if (ez < -126 || ez > 127) return f64_level(R, v, bad);
    // residual R - Z = sign * (M - n * 2^sh) * 2^(E - 1075), exact
    const int64_t d = (int64_t)M - (int64_t)(n << sh);
    if (d == 0) {
        R = 0.0;
    } else {
        const uint64_t ad = (uint64_t)(d < 0 ? -d : d);
        const uint64_t rs = (uint64_t)(sgn ^ (d < 0 ? 1u : 0u)) << 63;
        const int lz = __clzll((long long)ad) - 11;            // bring the leading bit to bit 52
        int er = E - lz;
        uint64_t rb;
        if (er >= 1) rb = rs | ((uint64_t)er << 52) | ((ad << lz) & 0x000FFFFFFFFFFFFFull);
        else rb = rs | ((ad << lz) >> (1 - er));              // subnormal result, still exact
        R = __longlong_as_double((long long)rb);
    }
    const uint32_t mant = (p <= 7 ? ((uint32_t)n << (7 - p)) : ((uint32_t)n >> 1)) & 0x7Fu;
    return (uint16_t)((sgn << 15) | ((uint32_t)(ez + 127) << 7) | mant);
}

// The six speculative levels v^(r) = v0 - 8r of one entry in fixed point.
// x is converted once to a signed integer X in units of 2^F, F = v0 - 50 (two
// bits below the finest grid 2^(v0 - 48)), truncating with a sticky ("jam")
// bit in the last place when x has bits below 2^F.  Every grid and every
// half-grid is an even multiple of 2^F, and a jammed value is odd and within
// one unit of the true one, so all round-to-nearest-even decisions and all
// comparisons with powers of two >= 2^(F+1) are those of the exact value;
// exact values stay exact.  Level r rounds X to nearest, ties to even, on the
// grid 2^(43 - 8r) (X >= 0) or 2^(42 - 8r) (X < 0) units -- the sign-dependent
// grid of the add-subtract projection -- and subtracts it.  |X| before level
// r goes to mx[r - 1] (in units of 2^F).  Levels 0-2 need 64-bit words; from
// level 3 on |X| < 2^27 and 32-bit words suffice.
__device__ __forceinline__ void spec_levels(double x, int v0, uint16_t (&s)[6], uint32_t &badmask,
                                            unsigned long long (&mx)[5])
{
    const uint64_t b = (uint64_t)__double_as_longlong(x);
    const uint32_t xs = (uint32_t)(b >> 63);
    const int E = (int)((b >> 52) & 0x7FFu);
    uint64_t M = b & 0x000FFFFFFFFFFFFFull;
    int Ee = E;
    if (E == 0) Ee = 1; else M |= 1ull << 52;
    const int F = v0 - 50;
    const int sh0 = (Ee - 1075) - F;                   // left shift into units of 2^F
    uint64_t mag;
    if (E == 0x7FF) badmask |= 1u;                     // a non-finite slice 0 (NONFINITE comes from the max pass)
    if (E == 0x7FF || M == 0) mag = 0;
    else if (sh0 >= 0) mag = sh0 < 12 ? (M << sh0) : (1ull << 62);   // (|x| > 2^v0 cannot occur)
    else if (sh0 > -64) mag = (M >> (-sh0)) | ((M << (64 + sh0)) != 0 ? 1ull : 0ull);
    else mag = 1;
    int64_t X = xs ? -(int64_t)mag : (int64_t)mag;
    // levels 0..2 in 64-bit
#pragma unroll
    for (int r = 0; r < 3; ++r) {
        const uint32_t sg = X < 0 ? 1u : 0u;
        const uint64_t a = (uint64_t)(sg ? -X : X);
        if (r > 0) mx[r - 1] = a > mx[r - 1] ? a : mx[r - 1];
        const int g = 43 - 8 * r - (int)sg;            // grid in units of 2^F
        const uint64_t n = (a + (1ull << (g - 1)) - 1ull + ((a >> g) & 1ull)) >> g;
        const int64_t zm = (int64_t)(n << g);
        X = sg ? (zm - (int64_t)a) : ((int64_t)a - zm);
        uint16_t out = 0;
        if (n) {
            const int p = 31 - __clz((unsigned)n);
            const int ez = F + g + p;                  // exponent of Z's leading bit
            if (ez < -126 || ez > 127) badmask |= 1u << r;
            const uint32_t mant = (p <= 7 ? ((uint32_t)n << (7 - p)) : ((uint32_t)n >> 1)) & 0x7Fu;
            out = (uint16_t)((sg << 15) | ((uint32_t)(ez + 127) << 7) | mant);
        }
        s[r] = out;
    }
    // levels 3..5 in 32-bit: |X| <= 2^26 + 1 here
    int32_t Y = (int32_t)X;
#pragma unroll
    for (int r = 3; r < 6; ++r) {
        const uint32_t sg = Y < 0 ? 1u : 0u;
        const uint32_t a = (uint32_t)(sg ? -Y : Y);
        mx[r - 1] = a > mx[r - 1] ? a : mx[r - 1];
        const int g = 43 - 8 * r - (int)sg;
        const uint32_t n = (a + (1u << (g - 1)) - 1u + ((a >> g) & 1u)) >> g;
        const int32_t zm = (int32_t)(n << g);
        Y = sg ? (zm - (int32_t)a) : ((int32_t)a - zm);
        uint16_t out = 0;
        if (n) {
            const int p = 31 - __clz(n);
            const int ez = F + g + p;
            if (ez < -126 || ez > 127) badmask |= 1u << r;
            const uint32_t mant = (p <= 7 ? (n << (7 - p)) : (n >> 1)) & 0x7Fu;
            out = (uint16_t)((sg << 15) | ((uint32_t)(ez + 127) << 7) | mant);
        }
        s[r] = out;
    }
}

// Final v^(0..5) of operand `slot` once verification and fix passes ran
// (levels up to fix_from come from the verifier, later ones from the fix
// maxima).  Levels past an all-zero residual are kZeroLevel.
__device__ __forceinline__ void final_levels(const WsHeader *ws, int slot, int upto, int (&v)[6])
{
    const int ff = ws->fix_from[slot];
    bool zero = false;
    for (int r = 0; r < 6; ++r) {
        if (r >= upto || zero) { v[r] = kZeroLevel; continue; }
        if (r <= ff) v[r] = ws->v[slot][r];
        else {
            const unsigned long long m = ws->fixmax[slot][r];
            v[r] = m ? ceil_log2_bits(m) : kZeroLevel;
        }
        if (v[r] == kZeroLevel) zero = true;
    }
}

__device__ __forceinline__ unsigned long long warp_max(unsigned long long x)
{
    for (int o = 16; o; o >>= 1) {
        const unsigned long long y = __shfl_xor_sync(0xFFFFFFFFu, x, o);
        x = y > x ? y : x;
    }
    return x;
}

// Block-wide max of one value per thread, then one atomicMax: the values are
// bit patterns of non-negative doubles, which order like the doubles.
__device__ __forceinline__ void block_max_to(unsigned long long x, unsigned long long *dst, unsigned long long *red)
{
    x = warp_max(x);
    const int w = threadIdx.x >> 5;
    if (lane_id() == 0) red[w] = x;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned long long m = 0;
        for (int i = 0; i < kThreads / 32; ++i) m = red[i] > m ? red[i] : m;
        if (m) atomicMax(dst, m);
    }
    __syncthreads();
}

// ------------------------------------------------------------ tile kernel
// Literal FP64 plane pass (T is double).  MODE 2: rewrite with the final
// whole-matrix levels (runs only when verification failed).  MODE 3: levels
// per plane row (per input row, or per input column when transposed), read
// from vrc[6][plane rows].
template <typename T, int MODE, bool TRANSPOSE>
__device__ __forceinline__ void
split_tile_pass(const T *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                uint16_t *__restrict__ comps, int64_t ldcomp, int64_t plane, WsHeader *ws, int slot,
                const int32_t *__restrict__ vrc, const int32_t *__restrict__ ff, int64_t bid, int64_t nblk,
                uint16_t *smdyn)
{
    static_assert(MODE == 2 || MODE == 3, "literal FP64 split modes only");
    constexpr int NS = 6;
    auto sm = [&](int r, int row, int col) -> uint16_t & {
        return smdyn[((size_t)r * kTile + row) * kSRow + col];
    };

    int v[6] = {0, 0, 0, 0, 0, 0};
    if constexpr (MODE == 2) {
        if (ws->fix_from[slot] >= 6) return;     // speculation held: nothing to redo
        final_levels(ws, slot, 6, v);
    }
    const int64_t nvec = TRANSPOSE ? cols : rows;        // plane rows (MODE 3's level vectors)
    // MODE 3 rewrites only the vectors whose speculative levels failed (ff < 6)
    if constexpr (MODE == 3) {
        if (ws->fix_any == 0) return;
    }
    uint32_t badmask = 0;
    const int64_t tiles_r = (rows + kTile - 1) / kTile, tiles_c = (cols + kTile - 1) / kTile;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;   // 16 x 16 threads

    for (int64_t t = bid; t < tiles_r * tiles_c; t += nblk) {
        const int64_t r0 = (t / tiles_c) * kTile, c0 = (t % tiles_c) * kTile;
        // ---- load, split, stage: thread (ty, tx) owns rows ty + 16p, columns 4tx..4tx+3
#pragma unroll
        for (int p = 0; p < 4; ++p) {
            const int li = ty + 16 * p;
            const int64_t gi = r0 + li;
            T x[4];
            const int64_t gj = c0 + 4 * tx;
            const T *src = X + gi * ldx + gj;
            const bool row_ok = gi < rows;
            if (row_ok && gj + 4 <= cols && ((reinterpret_cast<uintptr_t>(src) & 15u) == 0)) {
                if constexpr (sizeof(T) == 4) {
                    const float4 q = *reinterpret_cast<const float4 *>(src);
                    x[0] = q.x; x[1] = q.y; x[2] = q.z; x[3] = q.w;
                } else {
                    const double2 q0 = reinterpret_cast<const double2 *>(src)[0];
                    const double2 q1 = reinterpret_cast<const double2 *>(src)[1];
                    x[0] = q0.x; x[1] = q0.y; x[2] = q1.x; x[3] = q1.y;
                }
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) x[e] = (row_ok && gj + e < cols) ? src[e] : T(0);
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int lj = 4 * tx + e;
                uint16_t s[NS];
                int vv[6];
                if constexpr (MODE == 3) {
                    const int64_t vec = TRANSPOSE ? c0 + lj : gi;
#pragma unroll
                    for (int r = 0; r < 6; ++r) vv[r] = vec < nvec ? vrc[r * nvec + vec] : kZeroLevel;
                } else {
#pragma unroll
                    for (int r = 0; r < 6; ++r) vv[r] = v[r];
                }
                double R = x[e];
#pragma unroll
                for (int r = 0; r < 6; ++r) {
                    bool bad = false;
                    s[r] = f64_level_int(R, vv[r], bad);
                    if (bad) badmask |= 1u << r;
                }
#pragma unroll
                for (int r = 0; r < NS; ++r) {
                    if (TRANSPOSE) sm(r, lj, li) = s[r];
                    else sm(r, li, lj) = s[r];
                }
            }
        }
        __syncthreads();
        // ---- write plane rows in 16-byte chunks (8 BF16 per chunk)
        const int64_t orow0 = TRANSPOSE ? c0 : r0, ocol0 = TRANSPOSE ? r0 : c0;
        const int64_t orows = TRANSPOSE ? cols : rows, ocols = TRANSPOSE ? rows : cols;
        for (int c = threadIdx.x; c < NS * kTile * (kTile / 8); c += kThreads) {
            const int r = c / (kTile * (kTile / 8));
            const int rem = c % (kTile * (kTile / 8));
            const int orow = rem / (kTile / 8), ch = rem % (kTile / 8);
            const int64_t go = orow0 + orow, gc = ocol0 + 8 * ch;
            if (go >= orows || gc >= ocols) continue;
            if (MODE == 3 && ff[go] >= 6) continue;
            uint16_t *dst = comps + r * plane + go * ldcomp + gc;
            const uint32_t *w = reinterpret_cast<const uint32_t *>(&sm(r, orow, 8 * ch));
            if (gc + 8 <= ocols && ((reinterpret_cast<uintptr_t>(dst) & 15u) == 0)) {
                *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
            } else {
                for (int e = 0; e < 8 && gc + e < ocols; ++e) dst[e] = sm(r, orow, 8 * ch + e);
            }
        }
        __syncthreads();
    }

    badmask = __reduce_or_sync(0xFFFFFFFFu, badmask);
    if (badmask && lane_id() == 0) {
        if constexpr (MODE == 2) atomicOr(&ws->slice_bad[slot], badmask << 8);
        else atomicOr(&ws->flags, (uint32_t)EMU_FLAG_SLICE);
    }
}

// The pass above as a kernel of its own (smdyn: [NS][kTile][kSRow]).
template <typename T, int MODE, bool TRANSPOSE>
__global__ void __launch_bounds__(kThreads)
split_tile_kernel(const T *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                  uint16_t *__restrict__ comps, int64_t ldcomp, int64_t plane, WsHeader *ws, int slot,
                  const int32_t *__restrict__ vrc, const int32_t *__restrict__ ff)
{
    extern __shared__ __align__(16) uint16_t smdyn[];
    split_tile_pass<T, MODE, TRANSPOSE>(X, rows, cols, ldx, comps, ldcomp, plane, ws, slot, vrc, ff, blockIdx.x,
                                        gridDim.x, smdyn);
}

// --------------------------------------------- row-segment FP64 passes
// LEVEL = 0: max |x| and the input-domain checks of Eq. (bf16rangefp64).
// LEVEL = L in 1..5: max |A^(L)| recomputed literally from x with the final
// levels 0..L-1 (only when the trusted speculative levels end before L).
template <int LEVEL>
__device__ __forceinline__ void f64_max_pass(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                                             WsHeader *ws, int slot, int64_t bid, int64_t nblk,
                                             unsigned long long *red)
{
    int v[6] = {0, 0, 0, 0, 0, 0};
    if constexpr (LEVEL > 0) {
        if (ws->fix_from[slot] >= LEVEL) return;
        final_levels(ws, slot, LEVEL, v);
        if (v[LEVEL - 1] == kZeroLevel) return;   // residual already zero
    }
    // bit patterns of |x|: 2^-126 and (2 - 2^-7) * 2^127, and the exponent mask
    constexpr unsigned long long kLo = 0x3810000000000000ull, kHi = 0x47EFE00000000000ull;
    constexpr unsigned long long kInf = 0x7FF0000000000000ull;
    unsigned long long m = 0;
    uint32_t flagbits = 0;
    const int64_t segs = (cols + 4 * kThreads - 1) / (4 * kThreads);
    // four entries of row i from column j0 on
    auto body = [&](int64_t i, int64_t j0) {
        const double *src = X + i * ldx + j0;
        double x[4];
        if (j0 + 4 <= cols && ((reinterpret_cast<uintptr_t>(src) & 15u) == 0)) {
            const double2 q0 = reinterpret_cast<const double2 *>(src)[0];
            const double2 q1 = reinterpret_cast<const double2 *>(src)[1];
            x[0] = q0.x; x[1] = q0.y; x[2] = q1.x; x[3] = q1.y;
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) x[e] = (j0 + e < cols) ? src[e] : 0.0;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            double R = x[e];
            if constexpr (LEVEL > 0) {
                bool bad = false;
#pragma unroll
                for (int r = 0; r < LEVEL; ++r) (void)f64_level_int(R, v[r], bad);
            }
            const unsigned long long ab = (unsigned long long)__double_as_longlong(R) & 0x7FFFFFFFFFFFFFFFull;
            if constexpr (LEVEL == 0) {
                if (ab >= kInf) flagbits |= EMU_FLAG_NONFINITE;
                else if (ab != 0 && (ab < kLo || ab > kHi)) flagbits |= EMU_FLAG_RANGE;
                if (ab <= kInf) m = ab > m ? ab : m;                  // NaN never wins
            } else {
                m = ab > m ? ab : m;
            }
        }
    };
    if (nblk >= segs) {
        // block bid walks rows bid / segs, + rstride, ... of column segment
        // bid % segs (no division in the loop); blocks past rstride * segs idle
        const int64_t rstride = nblk / segs;
        if (bid < rstride * segs) {
            const int64_t j0 = (bid % segs) * (4 * kThreads) + 4 * threadIdx.x;
#pragma unroll 2
            for (int64_t i = bid / segs; i < rows; i += rstride) body(i, j0);
        }
    } else {
        for (int64_t it = bid; it < rows * segs; it += nblk) body(it / segs, (it % segs) * (4 * kThreads) + 4 * threadIdx.x);
    }
    if constexpr (LEVEL == 0) {
        flagbits = __reduce_or_sync(0xFFFFFFFFu, flagbits);
        if (flagbits && lane_id() == 0) atomicOr(&ws->flags, flagbits);
        block_max_to(m, &ws->maxbits[slot][0], red);
    } else {
        block_max_to(m, &ws->fixmax[slot][LEVEL], red);
    }
}

template <int LEVEL>
__global__ void __launch_bounds__(kThreads)
f64_max_kernel(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx, WsHeader *ws, int slot)
{
    __shared__ unsigned long long red[kThreads / 32];
    f64_max_pass<LEVEL>(X, rows, cols, ldx, ws, slot, blockIdx.x, gridDim.x, red);
}

// One thread: checks the speculative levels in order.  Level r's max from
// the fused pass is literal as long as levels < r were right and it spans
// at least two units 2^(v0 - 50) of the fixed point (below that the sticky
// bit of the truncated residual decides its power of two), so the first
// mismatch r gives the true v^(r) directly when v^(r) >= v0 - 48 and levels
// after r are redone; a smaller one is redone from level r itself.  A
// slice outside the BF16 normal range at level r (a domain violation, which
// the finalizer flags) also ends the trusted levels at r: the fused pass
// subtracts the exact projection Z there, while Eq. (fp64split) subtracts
// fl_BF16(Z), so the literal passes redo the levels after r.
// Only levels below nlev are checked (the speculative pass formed no more);
// later ones are reported as zero levels.
__device__ __forceinline__ int f64_verify_levels(const WsHeader *ws, int slot, int (&v)[6], int nlev = 6)
{
    int ff = 6;
    const uint32_t sb = ws->slice_bad[slot] & 0x3Fu;
    const int badlvl = (sb && !(ws->flags & EMU_FLAG_NONFINITE)) ? __ffs(sb) - 1 : 6;
    const unsigned long long m0 = ws->maxbits[slot][0];
    for (int r = 0; r < 6; ++r) v[r] = 0;
    if (m0 == 0) {
        for (int r = 0; r < 6; ++r) v[r] = kZeroLevel;
    } else {
        const int v0 = ceil_log2_bits(m0);
        v[0] = v0;
        if (badlvl == 0) ff = 0;
        bool zero = false;
        for (int r = 1; r < 6 && ff == 6; ++r) {
            if (zero || r >= nlev) { v[r] = kZeroLevel; continue; }
            const unsigned long long m = ws->maxbits[slot][r];
            if (m == 0) { v[r] = kZeroLevel; zero = true; continue; }
            const int vr = ceil_log2_bits(m);
            v[r] = vr;
            if (r == badlvl) ff = r;
            else if (vr != v0 - 8 * r) ff = vr >= v0 - 48 ? r : r - 1;
        }
    }
    return ff;
}

// One thread: publishes v_out and the slice flag of the levels actually used:
// those of slices 0 .. nlev-1, the only ones a product-sum of nlev diagonals
// reads (the checked general form of the speculative pass, and the literal
// passes, examine all six levels).
__device__ __forceinline__ void f64_finalize(WsHeader *ws, int slot, int32_t *v_out, int nlev = 6)
{
    int v[6];
    final_levels(ws, slot, 6, v);
    if (v_out)
        for (int r = 0; r < 6; ++r) v_out[r] = v[r];
    const int ff = ws->fix_from[slot];
    const uint32_t keep = (1u << ff) - 1u;                       // levels taken from the fused pass
    const uint32_t used = (1u << nlev) - 1u;
    const uint32_t sb = ws->slice_bad[slot];
    const uint32_t bad = ((sb & keep) | ((sb >> 8) & ~keep)) & used;
    if (bad) atomicOr(&ws->flags, (uint32_t)EMU_FLAG_SLICE);
}

// Bounded barrier over all blocks of a cooperative launch (ws->bar_*[slot]
// start at zero; the last block to arrive resets the count and opens the next
// generation).  After kWaitLimitNs a waiting block sets EMU_FLAG_TIMEOUT and
// goes on; the results of that call are then void, as the flag says.
__device__ __forceinline__ void grid_sync(WsHeader *ws, int slot)
{
    __syncthreads();
    if (threadIdx.x == 0) {
        volatile uint32_t *gen = &ws->bar_gen[slot];
        const uint32_t g = *gen;
        __threadfence();
        if (atomicAdd(&ws->bar_count[slot], 1u) == gridDim.x - 1) {
            ws->bar_count[slot] = 0;
            __threadfence();
            atomicAdd(&ws->bar_gen[slot], 1u);
        } else {
            const unsigned long long t0 = globaltimer_ns();
            for (uint32_t it = 0; *gen == g; ++it) {
                if ((it & 63u) == 63u && globaltimer_ns() - t0 > kWaitLimitNs) {
                    atomicOr(&ws->flags, (uint32_t)EMU_FLAG_TIMEOUT);
                    break;
                }
            }
        }
        __threadfence();
    }
    __syncthreads();
}

// ------------------------------------------ FP64 speculative pass kernels
// The levels of spec_levels restated so that most steps are 32-bit: levels 0
// and 1 have grids of 2^32 units or coarser and round on the upper word of
// the fixed-point magnitude (the lower word only breaks ties and is carried
// into the residual), level 2 rounds a value below 2^35 through its quotient
// and remainder, and levels 3-5 work in 32 bits.  At each level the grid
// splits |X| into t = |X| >> g and a remainder; rounding up (remainder above
// half the grid, or exactly half with t odd) leaves the grid minus the
// remainder with the opposite sign.  No range check is needed when
// v0 >= -78: every nonzero slice then lies between 2^(v0 - 48) >= 2^-126 and
// 2^v0 <= 2^127.  Results are bit-identical to spec_levels.
// Slices are returned as 32-bit words holding the FP32 value of the slice,
// whose upper 16 bits are its BF16 bits (the value has at most 8 significant
// bits, so the lower 16 are zero); two words pack into one plane word with a
// byte permutation.  The arithmetic runs on the FP32 pipe: n (an integer
// <= 256) is converted exactly (2^23 + n by bits, minus 2^23) and scaled by
// the level's unit, a power of two, with the sign of the residual (whose grid
// is half as coarse when negative: -1/2).  All values are normal floats on
// the fast path.  The FMA with +0 keeps a zero slice +0.
__device__ __forceinline__ uint32_t slice_word(uint32_t n, uint32_t sg, float unit)
{
    const float fn = __fsub_rn(__uint_as_float(0x4B000000u + n), 8388608.0f);
    const float us = __fmul_rn(unit, __uint_as_float(0x3F800000u + sg * 0x7F800000u));   // +1 or -1/2
    return __float_as_uint(__fmaf_rn(fn, us, 0.0f));
}

// Slice word of an FP32 value z (a multiple of the level's grid 2^c or 2^(c-1)
// units, at most nine significant bits) in units of 2^F: z * 2^-c * 2^(F + c),
// both steps exact; a zero z gives +0.
__device__ __forceinline__ uint32_t slice_word_scaled(float z, float inv_grid, float unit)
{
    return __float_as_uint(__fmul_rn(__fmul_rn(z, inv_grid), unit));
}

// Units of the six levels of the fast path: 2^(F + 43 - 8r), r = 0..5 (the
// grid of a non-negative residual at level r, in value).
__device__ __forceinline__ void spec_units(int F, float (&P)[6])
{
    P[0] = __int_as_float((F + 43 + 127) << 23);
#pragma unroll
    for (int r = 1; r < 6; ++r) P[r] = __fmul_rn(P[r - 1], 0.00390625f);          // 2^-8
}

template <int NLEV>
__device__ __forceinline__ void spec_levels_fast(double x, int F, const float (&P)[6], uint32_t (&s)[6],
                                                 uint32_t &badmask, unsigned long long &m1, unsigned long long &m2,
                                                 uint32_t (&m)[3])
{
    const uint64_t b = (uint64_t)__double_as_longlong(x);
    uint32_t sg = (uint32_t)(b >> 63);
    const int E = (int)((b >> 52) & 0x7FFu);
    uint64_t M = b & 0x000FFFFFFFFFFFFFull;
    int Ee = E;
    if (E == 0) Ee = 1; else M |= 1ull << 52;
    if (E == 0x7FF) { badmask |= 1u; M = 0; }          // a non-finite slice 0
    const int sh0 = (Ee - 1075) - F;
    uint64_t a;
    if (M == 0) a = 0;
    else if (sh0 >= 0) a = sh0 < 12 ? (M << sh0) : (1ull << 62);
    else if (sh0 > -64) a = (M >> (-sh0)) | ((M << (64 + sh0)) != 0 ? 1ull : 0ull);
    else a = 1;
    uint32_t H = (uint32_t)(a >> 32), L = (uint32_t)a;
    // At every level the rounding is written as multiply-adds where it can
    // be: with the grid 2^g (g one lower for a negative residual), t the
    // truncated quotient, rem = X - t 2^g and b the bits below the grid word
    // (a sticky bit for levels 0 and 1), rounding up happens exactly when
    // 2 rem + b + (t & 1) > 2^g (above half, or a tie with t odd); then the new
    // residual is 2^g - rem - b with the opposite sign.
    // levels 0, 1: grid 2^(32 + gh) units, gh = 11 / 10 and 3 / 2
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        if (r == 1) {
            const unsigned long long cur = ((unsigned long long)H << 32) | L;
            m1 = cur > m1 ? cur : m1;
        }
        constexpr uint32_t kG[2] = {1u << 11, 1u << 3};
        const uint32_t grid = kG[r] - sg * (kG[r] >> 1);
        const uint32_t t = H >> ((11 - 8 * r) - (int)sg);
        const uint32_t rh = H - t * grid;
        const uint32_t lnz = min(L, 1u);
        const uint32_t lsb = t & 1u;
        const int32_t d = (int32_t)(grid - 2u * rh - lnz - lsb);
        const uint32_t up = (uint32_t)d >> 31;
        s[r] = slice_word(t + up, sg, P[r]);
        H = rh + up * ((uint32_t)d + lsb);
        L = L * (1u - 2u * up);
        sg ^= up;
    }
    // level 2: |X| < 2^35, grid 2^27 / 2^26
    uint32_t Y;
    {
        const unsigned long long cur = ((unsigned long long)H << 32) | L;
        m2 = cur > m2 ? cur : m2;
        const uint32_t grid = (1u << 27) - sg * (1u << 26);
        const uint32_t t = __funnelshift_r(L, H, 27 - (int)sg);
        const uint32_t rem = L - t * grid;
        const uint32_t lsb = t & 1u;
        const int32_t d = (int32_t)(grid - 2u * rem - lsb);
        const uint32_t up = (uint32_t)d >> 31;
        s[2] = slice_word(t + up, sg, P[2]);
        Y = rem + up * ((uint32_t)d + lsb);
        sg ^= up;
    }
    if constexpr (NLEV <= 3) return;                   // levels from NLEV on are not wanted
    // level 3: |X| <= 2^26, grid 2^19 / 2^18
    {
        m[0] = Y > m[0] ? Y : m[0];
        const uint32_t grid = (1u << 19) - sg * (1u << 18);
        const uint32_t t = Y >> (19 - (int)sg);
        const uint32_t rem = Y - t * grid;
        const uint32_t lsb = t & 1u;
        const int32_t d = (int32_t)(grid - 2u * rem - lsb);
        const uint32_t up = (uint32_t)d >> 31;
        s[3] = slice_word(t + up, sg, P[3]);
        Y = rem + up * ((uint32_t)d + lsb);
        sg ^= up;
    }
    if constexpr (NLEV <= 4) return;
    // levels 4, 5: |X| <= 2^18, exact in FP32; the add-subtract projection
    // with C = 1.5 * 2^(23 + g) rounds to the grid 2^g to nearest, ties to even
    float y = __fsub_rn(__uint_as_float(0x4B000000u | Y), 8388608.0f);
    y = sg ? -y : y;
#pragma unroll
    for (int r = 4; r < 6; ++r) {
        if (r >= NLEV) break;
        const float ay = fabsf(y);
        m[r - 3] = max(m[r - 3], (uint32_t)ay);                   // exact: an integer below 2^24
        const float C = (y < 0.0f) ? (r == 4 ? 12884901888.0f : 50331648.0f)      // 1.5 * 2^33, 1.5 * 2^25
                                   : (r == 4 ? 25769803776.0f : 100663296.0f);    // 1.5 * 2^34, 1.5 * 2^26
        const float z = __fsub_rn(__fadd_rn(y, C), C);
        s[r] = slice_word_scaled(z, r == 4 ? 0.00048828125f : 0.125f, P[r]);     // 2^-11, 2^-3
        y = __fsub_rn(y, z);
    }
}

// Per-thread state of the speculative pass: level maxima in units of 2^F.
struct SpecState {
    unsigned long long m1 = 0, m2 = 0;
    uint32_t m[3] = {0, 0, 0};
    uint32_t badmask = 0;
};

// Slices 0 .. NLEV-1 of one entry (NLEV = 3..6; later ones are not formed).
template <int NLEV = 6>
__device__ __forceinline__ void spec_element(double x, int v0, bool fast, const float (&P)[6], uint32_t (&s)[6],
                                             SpecState &st)
{
    if (v0 == kZeroLevel) {
#pragma unroll
        for (int r = 0; r < 6; ++r) s[r] = 0;
    } else if (fast) {
        spec_levels_fast<NLEV>(x, v0 - 50, P, s, st.badmask, st.m1, st.m2, st.m);
    } else {                                          // tiny matrices: the checked general form
        uint16_t t[6];
        unsigned long long mx[5] = {st.m1, st.m2, st.m[0], st.m[1], st.m[2]};
        spec_levels(x, v0, t, st.badmask, mx);
        st.m1 = mx[0]; st.m2 = mx[1];
        st.m[0] = (uint32_t)mx[2]; st.m[1] = (uint32_t)mx[3]; st.m[2] = (uint32_t)mx[4];
#pragma unroll
        for (int r = 0; r < 6; ++r) s[r] = (uint32_t)t[r] << 16;
    }
}

// Plane word of two slice words (element e in the lower half, e + 1 in the upper).
__device__ __forceinline__ uint32_t pack2(uint32_t lo, uint32_t hi) { return __byte_perm(lo, hi, 0x7632); }

// Block-wide publication of the slice flags and the level maxima (as FP64
// bit patterns of |A^(r)|, r = 1..5).  Every thread of the block calls it.
__device__ __forceinline__ void spec_publish(const SpecState &st, int v0, WsHeader *ws, int slot, unsigned long long *red)
{
    const uint32_t bm = __reduce_or_sync(0xFFFFFFFFu, st.badmask);
    if (bm && lane_id() == 0) atomicOr(&ws->slice_bad[slot], bm);
    // maxima in units (integers, so the reduction needs no conversion); one
    // thread converts the block's five maxima to FP64 bit patterns
    unsigned long long mm[5] = {st.m1, st.m2, st.m[0], st.m[1], st.m[2]};
    const int w = threadIdx.x >> 5;
#pragma unroll
    for (int r = 0; r < 5; ++r) {
        mm[r] = warp_max(mm[r]);
        if (lane_id() == 0) red[r * (kThreads / 32) + w] = mm[r];
    }
    __syncthreads();
    if (threadIdx.x < 5) {
        const int r = threadIdx.x;
        unsigned long long m = 0;
        for (int i = 0; i < kThreads / 32; ++i) m = red[r * (kThreads / 32) + i] > m ? red[r * (kThreads / 32) + i] : m;
        if (m) {
            const int F = (v0 == kZeroLevel) ? 0 : v0 - 50;
            const double v = (double)m * pow2_d(F);                   // exact: below 2^53 units
            atomicMax(&ws->maxbits[slot][r + 1], (unsigned long long)__double_as_longlong(v));
        }
    }
}

__device__ __forceinline__ int spec_v0(const WsHeader *ws, int slot)
{
    const unsigned long long m0 = ws->maxbits[slot][0];
    return m0 ? ceil_log2_bits(m0) : kZeroLevel;
}

constexpr size_t kSpecTransposeSmem = 6 * kTile * (kTile / 2) * sizeof(uint32_t);

size_t smem_bytes(int ns) { return (size_t)ns * kTile * kSRow * sizeof(uint16_t); }

int grid_for(int64_t work_items, int max_blocks)
{
    int64_t g = work_items < 1 ? 1 : work_items;
    return (int)(g < max_blocks ? g : max_blocks);
}

}  // namespace

}  // namespace emu
