// FP64-mode tensor-core product-sum, Eq. (fp64reconstruction) / Algorithm 2.
#include "gemm_common.cuh"

namespace emu {

namespace {

// FP64 diagonal order (Algorithm 2): diagonal l = 0..5, i ascending, j = l - i.
// The first 6 / 10 / 15 / 21 entries are the sets S_3 .. S_6.
__constant__ int8_t kDiag[21][2] = {{0, 0}, {0, 1}, {1, 0}, {0, 2}, {1, 1}, {2, 0}, {0, 3},
                                    {1, 2}, {2, 1}, {3, 0}, {0, 4}, {1, 3}, {2, 2}, {3, 1},
                                    {4, 0}, {0, 5}, {1, 4}, {2, 3}, {3, 2}, {4, 1}, {5, 0}};

// ===================================================================== FP64
struct F64Cfg {
    static constexpr int BN = 128, KB = 64, STAGES = 6, NBUF = 4;
    static constexpr int A_TILE = kBM * KB * 2, B_TILE = BN * KB * 2;
    static constexpr int STAGE = A_TILE + B_TILE;
    static constexpr uint32_t SWZ = 2u, SBO = 1024u;
    static constexpr int BAR_OFF = STAGES * STAGE;
    static constexpr int SMEM = BAR_OFF + 256 + 1024;
    static constexpr int DRAIN_WARPS = 8, THREADS = 32 * (2 + DRAIN_WARPS);
    static constexpr int COLS_PER_WARP = BN / (DRAIN_WARPS / 4);   // 64
};

template <int NPROD>
__global__ void __launch_bounds__(F64Cfg::THREADS, 1)
prodsum_f64_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   int M, int N, int K, double *__restrict__ C, int64_t ldc, uint32_t *flags)
{
    using Cfg = F64Cfg;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *base_ptr = smem_raw + (base - raw);
    const uint32_t full0 = base + Cfg::BAR_OFF, empty0 = full0 + 8u * Cfg::STAGES;
    const uint32_t tfull0 = empty0 + 8u * Cfg::STAGES, tempty0 = tfull0 + 8u * Cfg::NBUF;
    const uint32_t done_bar = tempty0 + 8u * Cfg::NBUF;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(
        base_ptr + Cfg::BAR_OFF + 16 * Cfg::STAGES + 16 * Cfg::NBUF + 8);

    const int warp = threadIdx.x >> 5, lane = lane_id();
    const int tiles_m = (M + kBM - 1) / kBM, tiles_n = (N + Cfg::BN - 1) / Cfg::BN;
    int tm, tn;
    tile_coords(blockIdx.x, tiles_m, tiles_n, tm, tn);
    const int m0 = tm * kBM, n0 = tn * Cfg::BN;
    const int nch = (K + kKChunk - 1) / kKChunk;
    const int nt = nch * NPROD;                   // (chunk, pair) partials of this tile

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) { mbar_init(full0 + 8u * s, 1); mbar_init(empty0 + 8u * s, 1); }
        for (int b = 0; b < Cfg::NBUF; ++b) { mbar_init(tfull0 + 8u * b, 1); mbar_init(tempty0 + 8u * b, Cfg::DRAIN_WARPS); }
        mbar_init(done_bar, 1);
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    if (warp == 1) { tmem_alloc(smem_u32((const void *)tmem_slot), 512); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: for chunk, for pair, for K-block
        long L = 0;
        bool ok = true;
        for (int t = 0; t < nt && ok; ++t) {
            const int c = t / NPROD, q = t % NPROD;
            const int kbn = min(kKChunk / Cfg::KB, (K - c * kKChunk + Cfg::KB - 1) / Cfg::KB);
            for (int kb = 0; kb < kbn; ++kb, ++L) {
                const int s = (int)(L % Cfg::STAGES);
                if (!(ok = mbar_wait(empty0 + 8u * s, (uint32_t)(((L / Cfg::STAGES) & 1) ^ 1), flags))) break;
                const uint32_t st = base + (uint32_t)(s * Cfg::STAGE), fb = full0 + 8u * s;
                const int k0 = c * kKChunk + kb * Cfg::KB;
                mbar_arrive_expect_tx(fb, Cfg::STAGE);
                tma_load_3d(st, &tmA, fb, k0, m0, kDiag[q][0]);
                tma_load_3d(st + Cfg::A_TILE, &tmB, fb, k0, n0, kDiag[q][1]);
            }
        }
        if (!ok) drain_inflight(full0, Cfg::STAGES, L, flags);
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: one partial per (chunk, pair) into buffer t % NBUF
        constexpr uint32_t idesc = make_idesc_bf16(kBM, Cfg::BN);
        long L = 0;
        bool ok = true;
        for (int t = 0; t < nt && ok; ++t) {
            const int c = t / NPROD, b = t % Cfg::NBUF;
            const int kbn = min(kKChunk / Cfg::KB, (K - c * kKChunk + Cfg::KB - 1) / Cfg::KB);
            if (!(ok = mbar_wait(tempty0 + 8u * b, (uint32_t)(((t / Cfg::NBUF) & 1) ^ 1), flags))) break;
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(b * Cfg::BN);
            for (int kb = 0; kb < kbn; ++kb, ++L) {
                const int s = (int)(L % Cfg::STAGES);
                if (!(ok = mbar_wait(full0 + 8u * s, (uint32_t)((L / Cfg::STAGES) & 1), flags))) break;
                tc_fence_after();
                const uint32_t st = base + (uint32_t)(s * Cfg::STAGE);
#pragma unroll
                for (int kk = 0; kk < Cfg::KB / 16; ++kk) {
                    const uint64_t ad = make_sdesc(st + kk * 32, Cfg::SBO, Cfg::SWZ);
                    const uint64_t bd = make_sdesc(st + Cfg::A_TILE + kk * 32, Cfg::SBO, Cfg::SWZ);
                    mma_bf16(d, ad, bd, idesc, (kb | kk) != 0);
                }
                mma_commit(empty0 + 8u * s);
            }
            if (ok) mma_commit(tfull0 + 8u * b);
        }
        mma_commit(done_bar);
        (void)mbar_wait(done_bar, 0, flags);
    } else if (warp >= 2) {
        // ---------------- drain: widen each exact FP32 partial, add in FP64
        const int quarter = warp & 3;                       // TMEM lanes 32*quarter ..
        const int colh = ((warp - 2) >> 2) * Cfg::COLS_PER_WARP;
        const uint32_t lane_base = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)colh;
        double acc[Cfg::COLS_PER_WARP];
#pragma unroll
        for (int j = 0; j < Cfg::COLS_PER_WARP; ++j) acc[j] = 0.0;
        bool ok = true;
        for (int t = 0; t < nt; ++t) {
            const int b = t % Cfg::NBUF;
            ok = mbar_wait(tfull0 + 8u * b, (uint32_t)((t / Cfg::NBUF) & 1), flags);
            __syncwarp();
            if (!ok) break;
            tc_fence_after();
#pragma unroll
            for (int h = 0; h < Cfg::COLS_PER_WARP; h += 32) {
                uint32_t v[32];
                tmem_ld32(lane_base + (uint32_t)(b * Cfg::BN + h), v);
                tmem_ld_wait();
#pragma unroll
                for (int j = 0; j < 32; ++j) acc[h + j] = __dadd_rn(acc[h + j], (double)__uint_as_float(v[j]));
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty0 + 8u * b);
        }
        const int row = m0 + quarter * 32 + lane;
        if (ok && row < M) {
            double *crow = C + (int64_t)row * ldc + n0 + colh;
            const int lim = N - (n0 + colh);
            if (lim >= Cfg::COLS_PER_WARP && ((ldc & 1) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15u) == 0)) {
#pragma unroll
                for (int j = 0; j < Cfg::COLS_PER_WARP; j += 2)
                    *reinterpret_cast<double2 *>(crow + j) = make_double2(acc[j], acc[j + 1]);
            } else {
#pragma unroll
                for (int j = 0; j < Cfg::COLS_PER_WARP; ++j)
                    if (j < lim) crow[j] = acc[j];
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

template <int NPROD>
cudaError_t run_f64(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                    double *C, int64_t ldc, uint32_t *flags, cudaStream_t st)
{
    using Cfg = F64Cfg;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, 6, ldcomp, Cfg::KB, kBM) || !make_plane_map(&tb, Bp, K, N, 6, ldcomp, Cfg::KB, Cfg::BN))
        return cudaErrorInvalidValue;
    auto kern = prodsum_f64_kernel<NPROD>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int64_t tiles = ((M + kBM - 1) / kBM) * ((N + Cfg::BN - 1) / Cfg::BN);
    kern<<<(unsigned)tiles, Cfg::THREADS, Cfg::SMEM, st>>>(ta, tb, (int)M, (int)N, (int)K, C, ldc, flags);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prodsum_f64(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                               int64_t ldcomp, int nprod, double *C, int64_t ldc, uint32_t *flags, cudaStream_t st)
{
    switch (nprod) {
    case 6: return run_f64<6>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st);
    case 10: return run_f64<10>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st);
    case 15: return run_f64<15>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st);
    case 21: return run_f64<21>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace emu
