// Device helpers of the FP64-mode product-sums (Eq. (fp64reconstruction),
// Algorithm 2): register reallocation between warpgroups, exact FP32 -> FP64
// widening, the bound below which a plain FP32 addition of chunk partials is
// exact, TMEM loads and stores of a thread's columns, and Knuth's TwoSum.
#pragma once

#include "gemm_common.cuh"
#include "pair_common.cuh"

namespace emu {

template <uint32_t R> __device__ __forceinline__ void regs_dec() { asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(R)); }
template <uint32_t R> __device__ __forceinline__ void regs_inc() { asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(R)); }

// Exact FP32 -> FP64 widening by integer operations only (on GB300 a
// conversion instruction would occupy the FP64 pipe, which the fold's adds
// need): rebias the exponent and shift the significand of a normal value;
// normalise a subnormal by its leading bit; keep zeros, infinities and NaN
// payloads.
__device__ __forceinline__ double widen_exact(float x)
{
    const uint32_t u = __float_as_uint(x);
    const uint32_t sign = u & 0x80000000u, ex = (u >> 23) & 0xFFu, m = u & 0x7FFFFFu;
    uint32_t e = ex + 896u, f = m;                     // normal: exponent rebased from bias 127 to 1023
    if (ex == 0xFFu) e = 0x7FFu;                       // infinity / NaN
    if (ex == 0u) {
        if (m == 0u) { e = 0u; }                       // zero
        else {                                         // subnormal: m * 2^-149, leading bit at p
            const int p = 31 - __clz(m);
            e = (uint32_t)(p + 874);                   // p - 149 + 1023
            f = (m << (23 - p)) & 0x7FFFFFu;
        }
    }
    return __hiloint2double((int)(sign | (e << 20) | (f >> 3)), (int)(f << 29));
}


// The same widening for a zero or normal FP32 value only (five integer
// operations): rebias the exponent field by 1023 - 127 and move the
// significand's low three bits into the low word.  Not for subnormals,
// infinities or NaNs.
__device__ __forceinline__ double widen_normal(float x)
{
    const uint32_t u = __float_as_uint(x), a = u & 0x7FFFFFFFu;
    const uint32_t hi = (u & 0x80000000u) | (a ? (a >> 3) + 0x38000000u : 0u);
    return __hiloint2double((int)hi, (int)(u << 29));
}

// Largest running-sum magnitude below which adding a chunk partial of product
// (i, j) in FP32 is provably exact: every partial is an integer multiple of the
// unit u = 2^(vA_i + vB_j - 16), so any sum of magnitude below 2^24 u is
// representable, and rounding is monotone, so a rounded sum below 2^24 u was
// exact.  0 (always take the error-free path, renormalising every time) when
// the levels are unknown or the bound is not a normal float; +inf for a
// product of an all-zero slice.
__device__ __forceinline__ float bound_of_levels(int a, int b)
{
    if (a == kZeroLevel || b == kZeroLevel) return __int_as_float(0x7F800000);
    const int e = a + b + 8;                          // 2^24 * 2^(a + b - 16)
    if (e < -126 || e > 127) return 0.0f;
    return __int_as_float((e + 127) << 23);
}

__device__ __forceinline__ float exact_bound(const int32_t *vA, const int32_t *vB, int i, int j)
{
    if (!vA) return 0.0f;
    return bound_of_levels(vA[i], vB[j]);
}

// The same bound with levels per row of A (vA[6][M]) and per column of B
// (vB[6][N]), the vector scaling of Eq. (ozakiscaled): element (row, col) has
// unit 2^(vA_i[row] + vB_j[col] - 16), so a thread summing columns col0 ..
// col0 + ncols - 1 of one row may add plainly below 2^24 of the smallest of
// its units (a column or row whose slice is all zero contributes nothing).
__device__ __forceinline__ float exact_bound_rowcol(const int32_t *vA, const int32_t *vB, int M, int N, int i, int j,
                                                    int row, int col0, int ncols)
{
    const int a = row < M ? vA[(int64_t)i * M + row] : kZeroLevel;
    if (a == kZeroLevel) return __int_as_float(0x7F800000);
    int bmin = 0x7FFFFFFF;
    for (int c = 0; c < ncols; ++c) {
        const int col = col0 + c;
        if (col < N) {
            const int b = vB[(int64_t)j * N + col];
            if (b != kZeroLevel) bmin = b < bmin ? b : bmin;
        }
    }
    if (bmin == 0x7FFFFFFF) return __int_as_float(0x7F800000);
    return bound_of_levels(a, bmin);
}

// 16 consecutive 32-bit TMEM columns of this thread's lane: load / store.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
          "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

__device__ __forceinline__ uint32_t tmem_ld1(uint32_t taddr)
{
    uint32_t r;
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(r) : "r"(taddr) : "memory");
    return r;
}

__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&r)[8])
{
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr)
                 : "memory");
}

__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }


// Error-free sum of two FP32 values (Knuth's TwoSum): s = fl(a + b), a + b = s + e.
__device__ __forceinline__ float two_sum(float a, float b, float &e)
{
    const float s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
    return s;
}

}  // namespace emu
