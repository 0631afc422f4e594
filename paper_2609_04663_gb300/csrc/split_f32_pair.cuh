// Per-element arithmetic of the FP32 three-slice split, Eq. (fp32split),
// shared by the split kernels and the GEMM that splits inside its producer,
// so that both form identical slices.
#pragma once

#include "common.cuh"

namespace emu {

// Eq. (fp32split) on pairs of elements: the hardware conversion
// cvt.rn.bf16x2.f32 rounds two FP32 values to BF16 (round to nearest, ties
// to even, subnormals kept) and packs them into one 32-bit word, low element
// in the low half.  The residual of each is an exact FP32 subtraction of its
// slice, whose FP32 value is the BF16 bits shifted into the upper half.
__device__ __forceinline__ uint32_t bf16x2_rn(float lo, float hi)
{
    uint32_t d;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
    return d;
}

// Three slice words (planes 0, 1, 2) of the element pair (x0, x1).
__device__ __forceinline__ void split_pair(float x0, float x1, uint32_t &w0, uint32_t &w1, uint32_t &w2)
{
    w0 = bf16x2_rn(x0, x1);
    const float r0 = __fsub_rn(x0, __uint_as_float(w0 << 16)), r1 = __fsub_rn(x1, __uint_as_float(w0 & 0xFFFF0000u));
    w1 = bf16x2_rn(r0, r1);
    const float q0 = __fsub_rn(r0, __uint_as_float(w1 << 16)), q1 = __fsub_rn(r1, __uint_as_float(w1 & 0xFFFF0000u));
    w2 = bf16x2_rn(q0, q1);
}

// Largest |x| bit pattern of a pair, folded into a running maximum.
__device__ __forceinline__ uint32_t abs_bits_max(uint32_t amax, float x0, float x1)
{
    return max(amax, max(__float_as_uint(x0) & 0x7FFFFFFFu, __float_as_uint(x1) & 0x7FFFFFFFu));
}

// Flags of Eq. (fp32split)'s domain from the largest |x| bit pattern seen:
// a non-finite input, and a slice that is not finite.  For a finite x the
// only non-finite slice is slice 0 rounding up to infinity, which happens
// exactly when |x| >= 0x7F7F8000 (half a BF16 ulp above the largest BF16).
// Called by all 32 lanes of a warp.
__device__ __forceinline__ void publish_f32_flags(uint32_t amax, uint32_t *flags)
{
    uint32_t f = (amax >= 0x7F800000u ? (uint32_t)EMU_FLAG_NONFINITE : 0u) |
                 (amax >= 0x7F7F8000u ? (uint32_t)EMU_FLAG_SLICE : 0u);
    f = __reduce_or_sync(0xFFFFFFFFu, f);
    if (f && lane_id() == 0) atomicOr(flags, f);
}

}  // namespace emu
