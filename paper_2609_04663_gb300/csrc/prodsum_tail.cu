// Merged tail of the FP64 mode (an extension of Algorithm 2): the products
// (i, j) with L <= i + j < d are not summed exactly one by one; their sum
// T = sum A_i B_j is accumulated in ONE FP32 tensor-memory accumulator over all
// of K, and the FP64 product-sum adds T once after its last product
// (C = fl64(C_head + T)).  The tail products are at most 2^-8L of the leading
// one, but their FP32 sum runs over all of K: at 4096^3 with 21 products and
// the tail from diagonal 4, e_F against a double-double reference is 1.2e-14
// against 6.3e-15 for Algorithm 2 (and 1.5e-12 with 15 products).  In
// exchange the operand traffic drops: one stage holds slices 0 .. d-1 of A
// and of B and every tail product is issued from it, where the exact path
// streams both operands of every product separately.
//
// One CTA owns a 128 x 128 tile of T.  Stages hold d A tiles and d B tiles of
// one 32-wide K-block (64-byte swizzle, 8 KB each): 96 KB at d = 6, two
// stages.  Warp 0 lane 0 issues TMA loads, warp 1 owns TMEM and lane 0 issues
// the MMAs, warps 2-5 store T.  Every wait is bounded and reports
// EMU_FLAG_TIMEOUT.
//
// What bounds it: with two stages, about one stage of copies is in flight
// while the other is multiplied, and at the loaded L2 latency (about 1.4 us)
// that keeps the tensor pipe about 63 % busy at 11 products per 12 tiles.  Wider tiles need 16-wide K-blocks to fit three
// stages, and TMA copies of 32-byte rows were slower still (measured).
#include "gemm_common.cuh"
#include "launchers.cuh"

namespace emu {

namespace {

struct TailCfg {
    static constexpr int BN = 128, KB = 32, STAGES = 2;
    static constexpr int A_TILE = kBM * KB * 2, B_TILE = BN * KB * 2;   // one slice, one K-block
    static constexpr uint32_t SWZ = 4u, SBO = 8u * KB * 2u;    // 64-byte swizzle
    static constexpr int THREADS = 192;
    __host__ __device__ static constexpr int stage_bytes(int d) { return d * (A_TILE + B_TILE); }
    __host__ __device__ static constexpr int bar_off(int d) { return STAGES * stage_bytes(d); }
    __host__ __device__ static constexpr int smem(int d) { return bar_off(d) + 256 + 1024; }
};
static_assert(TailCfg::smem(6) <= 232448, "shared memory per CTA");

template <int L, int D>
__global__ void __launch_bounds__(TailCfg::THREADS, 1)
prodsum_tail_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, int M, int N,
                    int K, float *__restrict__ T, int64_t ldt, uint32_t *flags)
{
    using Cfg = TailCfg;
    static_assert(3 <= L && L < D && D <= 6, "tail diagonals");
    constexpr int Q0 = L * (L + 1) / 2, Q1 = D * (D + 1) / 2;   // kDiag[Q0 .. Q1) is the tail
    constexpr int STAGE = Cfg::stage_bytes(D), BAR_OFF = Cfg::bar_off(D);
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *base_ptr = smem_raw + (base - raw);
    const uint32_t full0 = base + BAR_OFF, empty0 = full0 + 8u * Cfg::STAGES;
    const uint32_t accum_bar = empty0 + 8u * Cfg::STAGES;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(base_ptr + BAR_OFF + 16 * Cfg::STAGES + 8);

    const int warp = threadIdx.x >> 5, lane = lane_id();
    const int tiles_m = (M + kBM - 1) / kBM, tiles_n = (N + Cfg::BN - 1) / Cfg::BN;
    int tm, tn;
    tile_coords(blockIdx.x, tiles_m, tiles_n, tm, tn);
    const int m0 = tm * kBM, n0 = tn * Cfg::BN;
    const int nkb = (K + Cfg::KB - 1) / Cfg::KB;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) { mbar_init(full0 + 8u * s, 1); mbar_init(empty0 + 8u * s, 1); }
        mbar_init(accum_bar, 1);
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    if (warp == 1) { tmem_alloc(smem_u32((const void *)tmem_slot), Cfg::BN); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: slices 0 .. D-1 of A, then of B
        long issued = 0;
        bool ok = true;
        for (int kb = 0; kb < nkb && ok; ++kb) {
            const int s = kb % Cfg::STAGES;
            if (!(ok = mbar_wait(empty0 + 8u * s, ((kb / Cfg::STAGES) & 1) ^ 1, flags))) break;
            const uint32_t st = base + (uint32_t)(s * STAGE), fb = full0 + 8u * s;
            mbar_arrive_expect_tx(fb, STAGE);
#pragma unroll
            for (int r = 0; r < D; ++r) tma_load_3d(st + r * Cfg::A_TILE, &tmA, fb, kb * Cfg::KB, m0, r);
#pragma unroll
            for (int r = 0; r < D; ++r)
                tma_load_3d(st + D * Cfg::A_TILE + r * Cfg::B_TILE, &tmB, fb, kb * Cfg::KB, n0, r);
            ++issued;
        }
        if (!ok) drain_inflight(full0, Cfg::STAGES, issued, flags);
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: every tail product of the K-block into one accumulator
        constexpr uint32_t idesc = make_idesc_bf16(kBM, Cfg::BN);
        for (int kb = 0; kb < nkb; ++kb) {
            const int s = kb % Cfg::STAGES;
            if (!mbar_wait(full0 + 8u * s, (kb / Cfg::STAGES) & 1, flags)) break;
            tc_fence_after();
            const uint32_t st = base + (uint32_t)(s * STAGE);
#pragma unroll
            for (int kk = 0; kk < Cfg::KB / 16; ++kk) {
#pragma unroll
                for (int q = Q0; q < Q1; ++q) {
                    const uint64_t ad = make_sdesc(st + kDiag[q][0] * Cfg::A_TILE + kk * 32, Cfg::SBO, Cfg::SWZ);
                    const uint64_t bd = make_sdesc(st + D * Cfg::A_TILE + kDiag[q][1] * Cfg::B_TILE + kk * 32,
                                                   Cfg::SBO, Cfg::SWZ);
                    mma_bf16(tmem, ad, bd, idesc, (kb | kk | (q - Q0)) != 0);
                }
            }
            mma_commit(empty0 + 8u * s);
        }
        mma_commit(accum_bar);
        (void)mbar_wait(accum_bar, 0, flags);
    } else if (warp >= 2) {
        // ---------------- epilogue: TMEM -> T
        const bool ok = mbar_wait(accum_bar, 0, flags);
        __syncwarp();
        if (ok) store_tile(tmem, warp & 3, 0, Cfg::BN, m0, n0, M, N, T, ldt);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, Cfg::BN);
    }
}

template <int L, int D>
cudaError_t run_tail(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                     float *T, int64_t ldt, uint32_t *flags, cudaStream_t st)
{
    using Cfg = TailCfg;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, 6, ldcomp, Cfg::KB, kBM) || !make_plane_map(&tb, Bp, K, N, 6, ldcomp, Cfg::KB, Cfg::BN))
        return cudaErrorInvalidValue;
    auto kern = prodsum_tail_kernel<L, D>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::smem(D));
    if (e != cudaSuccess) return e;
    const int64_t tiles = ((M + kBM - 1) / kBM) * ((N + Cfg::BN - 1) / Cfg::BN);
    kern<<<(unsigned)tiles, Cfg::THREADS, Cfg::smem(D), st>>>(ta, tb, (int)M, (int)N, (int)K, T, ldt, flags);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prodsum_tail(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                                int64_t ldcomp, int L, int d, float *T, int64_t ldt, uint32_t *flags,
                                cudaStream_t st)
{
    switch (10 * L + d) {
    case 34: return run_tail<3, 4>(M, N, K, Ap, Bp, ldcomp, T, ldt, flags, st);
    case 35: return run_tail<3, 5>(M, N, K, Ap, Bp, ldcomp, T, ldt, flags, st);
    case 36: return run_tail<3, 6>(M, N, K, Ap, Bp, ldcomp, T, ldt, flags, st);
    case 45: return run_tail<4, 5>(M, N, K, Ap, Bp, ldcomp, T, ldt, flags, st);
    case 46: return run_tail<4, 6>(M, N, K, Ap, Bp, ldcomp, T, ldt, flags, st);
    case 56: return run_tail<5, 6>(M, N, K, Ap, Bp, ldcomp, T, ldt, flags, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace emu
