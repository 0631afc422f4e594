// FP32-mode tensor-core product-sum (sm_103a: TMA -> shared memory ->
// tcgen05 BF16 MMAs with the FP32 accumulator in tensor memory), Eq. (fp32six)
// and the FP32 reconstruction of Section 6.3.
//
// One CTA owns a 128 x BN tile of C.  Each pipeline stage holds the three A
// slices and the three B slices of one K-block; the six retained products of
// that K-block are issued back to back from the same stage (one load of every
// slice serves all products that use it) into ONE FP32 accumulator in TMEM, in
// the operand-reuse order of Eq. (fp32reuseorder).  The accumulator is read
// once at the end.  Warp roles: warp 0 lane 0 issues TMA loads, warp 1 owns
// TMEM and lane 0 issues the MMAs, warps 2-5 run the epilogue.  Every wait is
// bounded and reports EMU_FLAG_TIMEOUT instead of hanging.
#include <cstdlib>

#include "gemm_common.cuh"
#include "launchers.cuh"

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

template <int BN, int KB, int STAGES>
__global__ void __launch_bounds__(192, 1)
prodsum_f32_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   int M, int N, int K, float *__restrict__ C, int64_t ldc, uint32_t *flags)
{
    using Cfg = F32Cfg<BN, KB, STAGES>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *base_ptr = smem_raw + (base - raw);
    const uint32_t full0 = base + Cfg::BAR_OFF, empty0 = full0 + 8u * STAGES;
    const uint32_t accum_bar = empty0 + 8u * STAGES;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(base_ptr + Cfg::BAR_OFF + 16 * STAGES + 8);

    const int warp = threadIdx.x >> 5, lane = lane_id();
    const int tiles_m = (M + kBM - 1) / kBM, tiles_n = (N + BN - 1) / BN;
    int tm, tn;
    tile_coords(blockIdx.x, tiles_m, tiles_n, tm, tn);
    const int m0 = tm * kBM, n0 = tn * BN;
    const int nkb = (K + KB - 1) / KB;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) { mbar_init(full0 + 8u * s, 1); mbar_init(empty0 + 8u * s, 1); }
        mbar_init(accum_bar, 1);
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    if (warp == 1) { tmem_alloc(smem_u32((const void *)tmem_slot), BN); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        long issued = 0;
        bool ok = true;
        for (int kb = 0; kb < nkb && ok; ++kb) {
            const int s = kb % STAGES;
            if (!(ok = mbar_wait(empty0 + 8u * s, ((kb / STAGES) & 1) ^ 1, flags))) break;
            const uint32_t st = base + (uint32_t)(s * Cfg::STAGE), fb = full0 + 8u * s;
            mbar_arrive_expect_tx(fb, Cfg::STAGE);
#pragma unroll
            for (int r = 0; r < 3; ++r) tma_load_3d(st + r * Cfg::A_TILE, &tmA, fb, kb * KB, m0, r);
#pragma unroll
            for (int r = 0; r < 3; ++r) tma_load_3d(st + 3 * Cfg::A_TILE + r * Cfg::B_TILE, &tmB, fb, kb * KB, n0, r);
            ++issued;
        }
        if (!ok) drain_inflight(full0, STAGES, issued, flags);
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
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
    } else if (warp >= 2) {
        // ---------------- epilogue: TMEM -> registers -> C
        const int quarter = warp & 3;
        const int row = m0 + quarter * 32 + lane;
        const bool ok = mbar_wait(accum_bar, 0, flags);
        __syncwarp();
        if (ok) {
            tc_fence_after();
            float *crow = C + (int64_t)row * ldc;
            const bool vec = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15u) == 0);
#pragma unroll 1
            for (int c = 0; c < BN; c += 32) {
                uint32_t v[32];
                tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c, v);
                tmem_ld_wait();
                const int col = n0 + c;
                if (row < M) {
                    if (vec && col + 32 <= N) {
#pragma unroll
                        for (int j = 0; j < 32; j += 4)
                            *reinterpret_cast<float4 *>(crow + col + j) =
                                make_float4(__uint_as_float(v[j]), __uint_as_float(v[j + 1]),
                                            __uint_as_float(v[j + 2]), __uint_as_float(v[j + 3]));
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (col + j < N) crow[col + j] = __uint_as_float(v[j]);
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, BN);
    }
}

template <int BN, int KB, int STAGES>
cudaError_t run_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                    float *C, int64_t ldc, uint32_t *flags, cudaStream_t st, int64_t a_plane, int64_t b_plane)
{
    using Cfg = F32Cfg<BN, KB, STAGES>;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, 3, ldcomp, KB, kBM, a_plane) ||
        !make_plane_map(&tb, Bp, K, N, 3, ldcomp, KB, BN, b_plane))
        return cudaErrorInvalidValue;
    auto kern = prodsum_f32_kernel<BN, KB, STAGES>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int64_t tiles = ((M + kBM - 1) / kBM) * ((N + BN - 1) / BN);
    kern<<<(unsigned)tiles, Cfg::THREADS, Cfg::SMEM, st>>>(ta, tb, (int)M, (int)N, (int)K, C, ldc, flags);
    return cudaGetLastError();
}

}  // namespace

// FP32 tile shape: 128 x 256 with 32-wide K-blocks (64-byte swizzle, 3 stages)
// by default; EMU_F32_TILE=128x128 selects 128 x 128 with 64-wide K-blocks
// (128-byte swizzle, 2 stages).
cudaError_t launch_prodsum_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                               int64_t ldcomp, float *C, int64_t ldc, uint32_t *flags, cudaStream_t st,
                               int64_t a_plane, int64_t b_plane)
{
    static const bool narrow = [] {
        const char *e = std::getenv("EMU_F32_TILE");
        return e && e[0] == '1' && e[1] == '2' && e[2] == '8' && e[3] == 'x' && e[4] == '1';
    }();
    if (narrow) return run_f32<128, 64, 2>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st, a_plane, b_plane);
    return run_f32<256, 32, 3>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st, a_plane, b_plane);
}

}  // namespace emu
