// Pieces shared by the FP32-mode product-sum kernels (the TMA-fed one and the
// one that splits inside its producer): tile configuration, the MMA issue
// loop of Eq. (fp32reuseorder) over a ring of stages (the epilogue is
// store_tile of gemm_common.cuh).
#pragma once

#include "gemm_common.cuh"

namespace emu {

namespace {

// FP32 chain, Eq. (fp32reuseorder): A1B1 A1B0 A2B0 A0B0 A0B1 A0B2.
__constant__ int8_t kChain[6][2] = {{1, 1}, {1, 0}, {2, 0}, {0, 0}, {0, 1}, {0, 2}};

// ===================================================================== FP32
template <int BN, int KB, int STAGES>
struct F32Cfg {
    static constexpr int A_TILE = kBM * KB * 2;
    static constexpr int B_TILE = BN * KB * 2;
    static constexpr int STAGE = 3 * A_TILE + 3 * B_TILE;
    static constexpr uint32_t SWZ = (KB == 64) ? 2u : 4u;       // 128-byte or 64-byte swizzle
    static constexpr uint32_t SBO = 8u * KB * 2u;               // bytes between 8-row groups
    static constexpr int BAR_OFF = STAGES * STAGE;
    static constexpr int SMEM = BAR_OFF + 256 + 1024;           // + barriers + alignment slack
    static constexpr int THREADS = 192;
    static_assert(KB == 32 || KB == 64, "K-block must fill one 64 B or 128 B swizzle row");
    static_assert(BN % 32 == 0 && BN >= 32 && BN <= 256, "UMMA N");
};

// MMA issuer (one thread): for every K-block, wait for its stage, issue the
// six products of Eq. (fp32reuseorder) from it into the one TMEM accumulator,
// and release the stage when those MMAs finish.  Then wait for all MMAs.
template <int BN, int KB, int STAGES>
__device__ __forceinline__ void mma_loop(uint32_t tmem, uint32_t base, uint32_t full0, uint32_t empty0,
                                         uint32_t accum_bar, int nkb, uint32_t *flags)
{
    using Cfg = F32Cfg<BN, KB, STAGES>;
    constexpr uint32_t idesc = make_idesc_bf16(kBM, BN);
    for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % STAGES;
        if (!mbar_wait(full0 + 8u * s, (kb / STAGES) & 1, flags)) break;
        tc_fence_after();
        const uint32_t st = base + (uint32_t)(s * Cfg::STAGE);
#pragma unroll
        for (int kk = 0; kk < KB / 16; ++kk) {
#pragma unroll
            for (int q = 0; q < 6; ++q) {
                const uint64_t ad = make_sdesc(st + kChain[q][0] * Cfg::A_TILE + kk * 32, Cfg::SBO, Cfg::SWZ);
                const uint64_t bd = make_sdesc(st + 3 * Cfg::A_TILE + kChain[q][1] * Cfg::B_TILE + kk * 32, Cfg::SBO, Cfg::SWZ);
                mma_bf16(tmem, ad, bd, idesc, (kb | kk | q) != 0);
            }
        }
        mma_commit(empty0 + 8u * s);         // stage reusable once these MMAs finish
    }
    mma_commit(accum_bar);                   // all MMAs issued so far are done
    (void)mbar_wait(accum_bar, 0, flags);
}

}  // namespace

}  // namespace emu
