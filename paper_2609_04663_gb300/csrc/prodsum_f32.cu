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
// bounded and reports EMU_FLAG_TIMEOUT instead of hanging.  The 128 x 256
// plan runs on CTA pairs (prodsum_f32_pair_kernel: 256 x 256 tiles, the same
// MMAs per output element).
#include <cstdlib>

#include "launchers.cuh"
#include "pair_common.cuh"
#include "prodsum_f32_common.cuh"

namespace emu {

namespace {

// Epilogue of one warp for a product-sum split along K: accumulator columns
// [c0, c1) of the warp's TMEM lane quarter added into C (which starts at zero)
// by FP32 reductions in L2.  With two K-parts the sum is the same in either
// order of arrival (0 + a, then a + b, rounded once; FP32 reductions flush
// subnormal inputs and results to zero).
__device__ __forceinline__ void reduce_tile(uint32_t tmem, int quarter, int c0, int c1, int m0, int n0, int M, int N,
                                            float *__restrict__ C, int64_t ldc)
{
    tc_fence_after();
    const int row = m0 + quarter * 32 + lane_id();
    float *crow = C + (int64_t)row * ldc;
    const bool vec = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15u) == 0);
#pragma unroll 1
    for (int c = c0; c < c1; c += 32) {
        uint32_t v[32];
        tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c, v);
        tmem_ld_wait();
        const int col = n0 + c;
        if (row < M) {
            if (vec && col + 32 <= N) {
#pragma unroll
                for (int j = 0; j < 32; j += 4)
                    asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(crow + col + j),
                                 "f"(__uint_as_float(v[j])), "f"(__uint_as_float(v[j + 1])),
                                 "f"(__uint_as_float(v[j + 2])), "f"(__uint_as_float(v[j + 3])) : "memory");
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (col + j < N)
                        asm volatile("red.global.add.f32 [%0], %1;" ::"l"(crow + col + j), "f"(__uint_as_float(v[j]))
                                     : "memory");
            }
        }
    }
}

// Epilogue of one warp through the TMA engine, for a C that a tensor map can
// describe: each 32 x 32 piece of the warp's 32 rows is staged in shared
// memory (stage memory, free once every MMA has completed: 4 KB per piece,
// BN / 8 KB per warp) in the 128-byte-swizzled layout of the C map and
// written by one bulk tensor store, or with REDUCE added into C by one bulk
// tensor reduction (the FP32 additions are the L2's, as with red.global).
// L2 then receives whole 128-byte row segments: a warp's st.global.v4 or
// red.global.add.v4 in store_tile / reduce_tile touches 32 cache lines, one
// per row, and those epilogues took 4.7 us per 128 x 256 tile and 2.0 us per
// 128 x 128 tile on GB300.
template <bool REDUCE>
__device__ __forceinline__ void epilogue_tma(uint32_t tmem, int quarter, int ncols, int m0, int n0, int M, int N,
                                             const CUtensorMap *cmap, uint32_t stage)
{
    tc_fence_after();
    const uint32_t lane = lane_id();
    const uint32_t slots = stage + (uint32_t)(quarter * ncols) * 128u;     // 32 rows x 4 bytes per column
    // pieces wholly past the last row or column are neither staged nor copied
    const int cols = m0 + quarter * 32 < M ? min(ncols, N - n0) : 0;
#pragma unroll 1
    for (int c = 0; c < cols; c += 32) {
        uint32_t v[32];
        tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c, v);
        tmem_ld_wait();
        // row `lane` of the piece: 16-byte chunk j at chunk j ^ (lane % 8), conflict-free
        const uint32_t buf = slots + (uint32_t)c * 128u, row = buf + lane * 128u;
#pragma unroll
        for (int j = 0; j < 8; ++j)
            st_shared_v4(row + ((uint32_t)(j ^ (int)(lane & 7u)) << 4), v[4 * j], v[4 * j + 1], v[4 * j + 2],
                         v[4 * j + 3]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            if (REDUCE) tma_reduce_add_2d(cmap, buf, n0 + c, m0 + quarter * 32);
            else tma_store_2d(cmap, buf, n0 + c, m0 + quarter * 32);
        }
    }
    // the CTA may exit once the copies have read shared memory; their writes
    // to C complete before the kernel does
    if (lane == 0) {
        bulk_commit();
        bulk_wait_read<0>();
    }
    __syncwarp();
}

// SPLIT > 1: the grid holds SPLIT CTAs per output tile, each over its own
// contiguous range of K-blocks, which add their FP32 accumulators into C (set
// to zero beforehand) instead of storing them.  c_tma: C is written through
// the tensor map tmC.  pair_first >= 0 (BN = 128): CTA b computes quarter
// b % 4 of 256 x 256 tile pair_first + b / 4 in the raster order of
// prodsum_f32_pair_kernel, which ran the tiles before it.
template <int BN, int KB, int STAGES, int SPLIT>
__global__ void __launch_bounds__(192, 1)
prodsum_f32_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, int c_tma, int M, int N, int K, float *__restrict__ C,
                   int64_t ldc, uint32_t *flags, int pair_first)
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
    const int tiles = tiles_m * tiles_n, part = pair_first >= 0 ? 0 : (int)blockIdx.x / tiles;
    if (pair_first >= 0) {
        int tp, tq;
        tile_coords(pair_first + (int)(blockIdx.x >> 2), (tiles_m + 1) / 2, (N + 255) / 256, tp, tq);
        tm = 2 * tp + (int)(blockIdx.x & 1);
        tn = 2 * tq + (int)((blockIdx.x >> 1) & 1);
    } else {
        tile_coords((int)blockIdx.x % tiles, tiles_m, tiles_n, tm, tn);
    }
    const int m0 = tm * kBM, n0 = tn * BN;
    const int nkb_all = (K + KB - 1) / KB, per = (nkb_all + SPLIT - 1) / SPLIT;
    const int kb0 = min(nkb_all, part * per);
    const int nkb = min(nkb_all, kb0 + per) - kb0;     // K-blocks of this CTA

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
    // set-up above overlaps the end of the kernel that wrote the planes (and
    // cleared C) when this one is launched as its programmatic dependent
    griddep_wait();

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
            for (int r = 0; r < 3; ++r) tma_load_3d(st + r * Cfg::A_TILE, &tmA, fb, (kb0 + kb) * KB, m0, r);
#pragma unroll
            for (int r = 0; r < 3; ++r)
                tma_load_3d(st + 3 * Cfg::A_TILE + r * Cfg::B_TILE, &tmB, fb, (kb0 + kb) * KB, n0, r);
            ++issued;
        }
        if (!ok) drain_inflight(full0, STAGES, issued, flags);
    } else if (warp == 1 && lane == 0) {
        mma_loop<BN, KB, STAGES>(tmem, base, full0, empty0, accum_bar, nkb, flags);
    } else if (warp >= 2) {
        // ---------------- epilogue: TMEM -> registers -> C (tcgen05.ld needs the
        // whole warp, so a timeout in any lane skips the warp's epilogue)
        const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait(accum_bar, 0, flags));
        if (ok && SPLIT == 1 && c_tma) epilogue_tma<false>(tmem, warp & 3, BN, m0, n0, M, N, &tmC, base);
        else if (ok && SPLIT == 1) store_tile(tmem, warp & 3, 0, BN, m0, n0, M, N, C, ldc);
        else if (ok && nkb > 0 && c_tma) epilogue_tma<true>(tmem, warp & 3, BN, m0, n0, M, N, &tmC, base);
        else if (ok && nkb > 0) reduce_tile(tmem, warp & 3, 0, BN, m0, n0, M, N, C, ldc);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, BN);
    }
}

// The FP32 product-sum on CTA pairs: a cluster of two CTAs on one TPC computes
// a 256 x BN tile with tcgen05 cta_group::2 MMAs (M = 256) issued by the
// leader (cluster rank 0).  Each CTA stages its 128 rows of the three A
// slices and its BN / 2-row half of the three B slices, both CTAs' copies
// counted on the leader's stage barrier; the MMA commits arrive on both CTAs'
// barriers, and each CTA's TMEM receives its 128 x BN part of the
// accumulator, which its own epilogue warps write into C.  An SM then takes
// in 128 + BN / 2 rows of operands per K-block for 128 x BN results instead
// of 128 + BN: with BN = 256 a third fewer bytes cross from L2 into shared
// memory, which at 16384^3 (a step held by the power cap) took the
// product-sum from 26.6 to 25.0 ms.  The MMAs and their order per output
// element are those of prodsum_f32_kernel; C is bit-identical to it.
// Timeouts: a peer whose wait gave up cannot see the leader's barriers, so
// it lets its copies land for 200 us before winding down.
template <int BN, int KB, int STAGES>
struct F32PairCfg {
    static constexpr int BH = BN / 2;                          // B rows staged by each CTA
    static constexpr int A_TILE = kBM * KB * 2;
    static constexpr int B_TILE = BH * KB * 2;
    static constexpr int STAGE = 3 * A_TILE + 3 * B_TILE;
    static constexpr uint32_t SWZ = (KB == 64) ? 2u : 4u;
    static constexpr uint32_t SBO = 8u * KB * 2u;
    static constexpr int BAR_OFF = STAGES * STAGE;
    static constexpr int SMEM = BAR_OFF + 256 + 1024;
    static_assert(KB == 32 || KB == 64, "K-block must fill one 64 B or 128 B swizzle row");
    static_assert(BN % 32 == 0 && BN >= 64 && BN <= 256, "UMMA N of a pair");
    static_assert(SMEM <= 232448, "shared memory per CTA");
};

template <int BN, int KB, int STAGES, int SPLIT>
__global__ void __launch_bounds__(192, 1)
prodsum_f32_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                        const __grid_constant__ CUtensorMap tmC, int c_tma, int M, int N, int K,
                        float *__restrict__ C, int64_t ldc, uint32_t *flags)
{
    using Cfg = F32PairCfg<BN, KB, STAGES>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *base_ptr = smem_raw + (base - raw);
    const uint32_t full0 = base + Cfg::BAR_OFF, empty0 = full0 + 8u * STAGES;
    const uint32_t accum_bar = empty0 + 8u * STAGES;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(base_ptr + Cfg::BAR_OFF + 16 * STAGES + 8);
    const int warp = threadIdx.x >> 5, lane = lane_id();
    const uint32_t rank = cluster_rank();
    const int pm = ((M + kBM - 1) / kBM + 1) / 2, tiles_n = (N + BN - 1) / BN;   // pair tile rows, tile columns
    const int ptiles = pm * tiles_n, cl = (int)(blockIdx.x >> 1), part = cl / ptiles;
    int tp, tn;
    tile_coords(cl % ptiles, pm, tiles_n, tp, tn);
    const int m0 = (2 * tp + (int)rank) * kBM, n0 = tn * BN;   // this CTA's 128 rows of the pair's 256
    const int nkb_all = (K + KB - 1) / KB, per = (nkb_all + SPLIT - 1) / SPLIT;
    const int kb0 = min(nkb_all, part * per);
    const int nkb = min(nkb_all, kb0 + per) - kb0;     // K-blocks of this pair

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) { mbar_init(full0 + 8u * s, 1); mbar_init(empty0 + 8u * s, 1); }
        mbar_init(accum_bar, 1);
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    __syncthreads();
    cluster_sync();                                   // both CTAs' barriers initialised
    if (warp == 1) tmem_alloc_pair(smem_u32((const void *)tmem_slot), BN);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // set-up above overlaps the end of the kernel that wrote the planes when
    // this one is launched as its programmatic dependent
    griddep_wait();

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer of this CTA: its A rows and its half of B,
        // counted on the leader's full barrier
        long issued = 0;
        bool ok = true;
        for (int kb = 0; kb < nkb && ok; ++kb) {
            const int s = kb % STAGES;
            if (!(ok = mbar_wait(empty0 + 8u * s, ((kb / STAGES) & 1) ^ 1, flags))) break;
            const uint32_t st = base + (uint32_t)(s * Cfg::STAGE), fb = full0 + 8u * s, fl = peer_addr(fb, 0);
            if (rank == 0) mbar_arrive_expect_tx(fb, 2 * Cfg::STAGE);
            const int k0 = (kb0 + kb) * KB;
#pragma unroll
            for (int r = 0; r < 3; ++r) tma_load_3d_pair(st + r * Cfg::A_TILE, &tmA, fl, k0, m0, r);
#pragma unroll
            for (int r = 0; r < 3; ++r)
                tma_load_3d_pair(st + 3 * Cfg::A_TILE + r * Cfg::B_TILE, &tmB, fl, k0, n0 + (int)rank * Cfg::BH, r);
            ++issued;
        }
        if (!ok) {
            if (rank == 0) {
                drain_inflight(full0, STAGES, issued, flags);
            } else {
                const unsigned long long t0 = globaltimer_ns();
                while (globaltimer_ns() - t0 < 200000ull) {}
            }
        }
    } else if (warp == 1 && lane == 0 && rank == 0) {
        // ---------------- MMA issuer (the leader): the six products of Eq.
        // (fp32reuseorder) per 16-wide K step, M = 256 over the pair
        constexpr uint32_t idesc = make_idesc_bf16(2 * kBM, BN);
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
                    const uint64_t bd = make_sdesc(st + 3 * Cfg::A_TILE + kChain[q][1] * Cfg::B_TILE + kk * 32,
                                                   Cfg::SBO, Cfg::SWZ);
                    mma_bf16_pair(tmem, ad, bd, idesc, (kb | kk | q) != 0);
                }
            }
            mma_commit_pair(empty0 + 8u * s);         // both CTAs' stages reusable once these finish
        }
        mma_commit_pair(accum_bar);                   // both CTAs' accumulator parts complete
    } else if (warp >= 2) {
        // ---------------- epilogue of this CTA's 128 rows (tcgen05.ld needs the
        // whole warp, so a timeout in any lane skips the warp's epilogue)
        const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait(accum_bar, 0, flags));
        if (ok && SPLIT == 1 && c_tma) epilogue_tma<false>(tmem, warp & 3, BN, m0, n0, M, N, &tmC, base);
        else if (ok && SPLIT == 1) store_tile(tmem, warp & 3, 0, BN, m0, n0, M, N, C, ldc);
        else if (ok && nkb > 0 && c_tma) epilogue_tma<true>(tmem, warp & 3, BN, m0, n0, M, N, &tmC, base);
        else if (ok && nkb > 0) reduce_tile(tmem, warp & 3, 0, BN, m0, n0, M, N, C, ldc);
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();                                   // the leader's MMAs are done with both CTAs
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc_pair(tmem, BN);
    }
}

// Per-SM rates of the narrower tiles relative to 128 x 256 (measured at 8192^3:
// 274 and 164 against 316 TFLOP/s for the whole GEMM).
constexpr double kRate128 = 0.87, kRate64 = 0.52;
// Cost of splitting K in two (clearing C, adding the halves in L2) as a
// factor on the per-SM rate.
constexpr double kSplitCost = 0.95;

template <int BN, int KB, int STAGES, int SPLIT = 1>
cudaError_t run_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                    float *C, int64_t ldc, uint32_t *flags, cudaStream_t st, int64_t a_plane, int64_t b_plane,
                    int pair_first = -1, int64_t pair_tiles = 0)
{
    using Cfg = F32Cfg<BN, KB, STAGES>;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, 3, ldcomp, KB, kBM, a_plane) ||
        !make_plane_map(&tb, Bp, K, N, 3, ldcomp, KB, BN, b_plane))
        return cudaErrorInvalidValue;
    // the epilogue writes (or adds) C through a C tensor map when one exists
    static_assert(4 * BN * 128 <= STAGES * Cfg::STAGE, "TMA epilogue staging exceeds the stage memory");
    CUtensorMap tc = {};
    const int c_tma = make_c_map_f32(&tc, C, M, N, ldc) ? 1 : 0;
    auto kern = prodsum_f32_kernel<BN, KB, STAGES, SPLIT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int64_t tiles = pair_first >= 0 ? 4 * pair_tiles : ((M + kBM - 1) / kBM) * ((N + BN - 1) / BN) * SPLIT;
    // launched as a programmatic dependent of the previous kernel in the
    // stream: its set-up overlaps that kernel's tail (griddep_wait orders the
    // rest after it)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)tiles);
    cfg.blockDim = dim3(Cfg::THREADS);
    cfg.dynamicSmemBytes = Cfg::SMEM;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, c_tma, (int)M, (int)N, (int)K, C, ldc, flags, pair_first);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

template <int BN, int KB, int STAGES, int SPLIT>
cudaError_t run_f32_pair(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                         float *C, int64_t ldc, uint32_t *flags, cudaStream_t st, int64_t a_plane, int64_t b_plane,
                         int64_t pair_tiles)
{
    using Cfg = F32PairCfg<BN, KB, STAGES>;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, 3, ldcomp, KB, kBM, a_plane) ||
        !make_plane_map(&tb, Bp, K, N, 3, ldcomp, KB, Cfg::BH, b_plane))
        return cudaErrorInvalidValue;
    static_assert(4 * BN * 128 <= STAGES * Cfg::STAGE, "TMA epilogue staging exceeds the stage memory");
    CUtensorMap tc = {};
    const int c_tma = make_c_map_f32(&tc, C, M, N, ldc) ? 1 : 0;
    auto kern = prodsum_f32_pair_kernel<BN, KB, STAGES, SPLIT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int64_t pairs = pair_tiles * SPLIT;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(2 * pairs));
    cfg.blockDim = dim3(192);
    cfg.dynamicSmemBytes = Cfg::SMEM;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, c_tma, (int)M, (int)N, (int)K, C, ldc, flags);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

// FP32 tile plan.  128 x 256 with 32-wide K-blocks (64-byte swizzle, three
// stages) is the fastest per SM; 128 x 128 (64-wide K-blocks, 128-byte
// swizzle, two stages) and 128 x 64 (64-wide K-blocks, three stages) reach
// smaller fractions of it but give more CTAs, which pays when there are too
// few 128 x 256 tiles to fill the GPU.  The choice maximises (SMs kept busy
// over the waves) x (relative per-SM rate).  Every shape issues the same MMAs
// in the same order for each output element, so C does not depend on it.
// EMU_F32_TILE=128x256 / 128x128 / 128x64 forces one.  The 128 x 256 plan
// runs on CTA pairs where it can (f32_pair_plan below).
void f32_tile_plan(int64_t M, int64_t N, int64_t K, bool split_ok, int &bn, int &parts)
{
    static const int forced = [] {
        const char *e = std::getenv("EMU_F32_TILE");
        if (!e || e[0] != '1' || e[1] != '2' || e[2] != '8' || e[3] != 'x') return 0;
        return (e[4] == '2' && e[5] == '5' && e[6] == '6') ? 256 : (e[4] == '1' && e[5] == '2' && e[6] == '8') ? 128
               : (e[4] == '6' && e[5] == '4') ? 64 : 0;
    }();
    bn = forced;
    parts = 1;
    if (bn != 0) return;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        sms = 152;
    // (width, K-parts, relative per-SM rate); the split plan needs C cleared
    // beforehand and at least two 64-wide K-blocks per part
    const int widths[4] = {256, 128, 64, 128}, nparts[4] = {1, 1, 1, 2};
    const double rate[4] = {1.0, kRate128, kRate64, kRate128 * kSplitCost};
    const int options = (split_ok && K >= 4 * 64) ? 4 : 3;
    double best = -1.0;
    for (int i = 0; i < options; ++i) {
        const int64_t ctas = ((M + kBM - 1) / kBM) * ((N + widths[i] - 1) / widths[i]) * nparts[i];
        const int64_t waves = (ctas + sms - 1) / sms;
        const double score = rate[i] * (double)ctas / (double)(waves * sms);
        if (score > best * 1.02) { best = score; bn = widths[i]; parts = nparts[i]; }   // earlier options win near ties
    }
}

// Per-SM rate of a 128 x 128 tile relative to the 256 x 256 tiles on pairs.
constexpr double kRateQuarter = 0.85;

static bool f32_pair_ok()
{
    static const bool ok = [] {
        const char *e = std::getenv("EMU_F32_PAIR");
        return !(e && e[0] == '0');
    }();
    return ok;
}

// Schedule of the 128 x 256 plan: 256 x 256 tiles on CTA pairs wherever there
// are two or more 128-row tile rows (EMU_F32_PAIR=0 keeps one CTA per tile).
// When the pair tiles leave the last wave partly empty and its tiles fit one
// wave as 128 x 128 quarters, those run in a second launch of the one-CTA
// kernel if that is estimated at least 2 % faster (a quarter takes
// 0.5 / kRateQuarter of a pair wave).  pairs: pair tiles in the first launch;
// rest: pair tiles left to the quarters launch (0: none).  false: no pairs.
static bool f32_pair_plan(int64_t M, int64_t N, int64_t &pairs, int64_t &rest)
{
    if (!f32_pair_ok() || M <= kBM) return false;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 2)
        sms = 152;
    const int64_t total = (((M + kBM - 1) / kBM + 1) / 2) * ((N + 255) / 256), per_wave = sms / 2;
    const int64_t full = total / per_wave, left = total % per_wave;
    pairs = total;
    rest = 0;
    if (full >= 1 && left > 0 && 4 * left <= sms &&
        (double)full + 0.5 / kRateQuarter <= 0.98 * (double)(full + 1)) {
        pairs = total - left;
        rest = left;
    }
    return true;
}

int f32_prodsum_launches(int64_t M, int64_t N)
{
    int bn, parts;
    f32_tile_plan(M, N, 0, false, bn, parts);
    int64_t pairs, rest;
    return (bn == 256 && f32_pair_plan(M, N, pairs, rest) && rest > 0) ? 2 : 1;
}

int f32_tile_rows(int64_t M, int64_t N)
{
    int bn, parts;
    f32_tile_plan(M, N, 0, false, bn, parts);
    int64_t pairs, rest;
    return (bn == 256 && f32_pair_plan(M, N, pairs, rest)) ? 256 : 128;
}

int f32_tile_columns(int64_t M, int64_t N)
{
    int bn, parts;
    f32_tile_plan(M, N, 0, false, bn, parts);
    return bn;
}

int f32_split_parts(int64_t M, int64_t N, int64_t K)
{
    int bn, parts;
    f32_tile_plan(M, N, K, true, bn, parts);
    return parts;
}

cudaError_t launch_prodsum_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                               int64_t ldcomp, float *C, int64_t ldc, uint32_t *flags, cudaStream_t st,
                               int64_t a_plane, int64_t b_plane, bool c_zeroed)
{
    int bn, parts;
    f32_tile_plan(M, N, K, c_zeroed, bn, parts);
    // 128 x 256 tiles run as 256 x 256 tiles on CTA pairs (64-wide K-blocks,
    // two 96 KB stages: at 16384^3 25.0 ms against 25.5 with 32-wide K-blocks
    // in four stages), the last partial wave possibly as 128 x 128 quarters
    int64_t pairs, rest;
    if (bn == 256 && parts == 1 && f32_pair_plan(M, N, pairs, rest)) {
        cudaError_t e = run_f32_pair<256, 64, 2, 1>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st, a_plane, b_plane,
                                                    pairs);
        if (e == cudaSuccess && rest > 0)
            e = run_f32<128, 64, 2>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st, a_plane, b_plane, (int)pairs, rest);
        return e;
    }
    if (parts == 2) return run_f32<128, 64, 2, 2>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st, a_plane, b_plane);
    if (bn == 128) return run_f32<128, 64, 2>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st, a_plane, b_plane);
    if (bn == 64) return run_f32<64, 64, 3>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st, a_plane, b_plane);
    return run_f32<256, 32, 3>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st, a_plane, b_plane);
}

}  // namespace emu
