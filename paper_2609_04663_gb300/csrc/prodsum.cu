// Tensor-core product-sum kernels (sm_103a: TMA -> shared memory -> tcgen05
// BF16 MMAs with FP32 accumulators in tensor memory).
//
// FP32 mode, Eq. (fp32six) / Section 5.3: one CTA owns a 128 x BN tile of C.
// Each pipeline stage holds the three A slices and the three B slices of one
// K-block; the six retained products of that K-block are issued back to back
// from the same stage (one load of every slice serves all products that use
// it) into ONE FP32 accumulator in TMEM, in the operand-reuse order of
// Eq. (fp32reuseorder).  The accumulator is read once at the end.
//
// FP64 mode, Eq. (fp64reconstruction) / Algorithm 2: for every K-chunk of 256
// and every retained pair (i, j) in diagonal order the chunk partial
// fl32(A_i B_j) is formed in its own TMEM buffer (4 rotating buffers of 128
// columns), then eight drain warps widen it to FP64 and add it into FP64
// register accumulators while the tensor cores already form the next
// partials.  The drain adds the partials in exactly the oracle's order
// (chunk outer, pair inner); every partial is exact (BF16 slices on the grid
// of Eq. (fp64split), 256-long chunks), so the FP64 result is bit-identical
// to the oracle.
//
// Warp roles: warp 0 lane 0 issues TMA loads, warp 1 owns TMEM and lane 0
// issues the MMAs, the remaining warps read TMEM.  Every wait is bounded and
// reports EMU_FLAG_TIMEOUT instead of hanging.
#include <cstdlib>
#include <mutex>

#include "common.cuh"

namespace emu {

namespace {

// FP32 chain, Eq. (fp32reuseorder): A1B1 A1B0 A2B0 A0B0 A0B1 A0B2.
__constant__ int8_t kChain[6][2] = {{1, 1}, {1, 0}, {2, 0}, {0, 0}, {0, 1}, {0, 2}};
// FP64 diagonal order (Algorithm 2): diagonal l = 0..5, i ascending, j = l - i.
// The first 6 / 10 / 15 / 21 entries are the sets S_3 .. S_6.
__constant__ int8_t kDiag[21][2] = {{0, 0}, {0, 1}, {1, 0}, {0, 2}, {1, 1}, {2, 0}, {0, 3},
                                    {1, 2}, {2, 1}, {3, 0}, {0, 4}, {1, 3}, {2, 2}, {3, 1},
                                    {4, 0}, {0, 5}, {1, 4}, {2, 3}, {3, 2}, {4, 1}, {5, 0}};

constexpr int kBM = 128;
constexpr int kGroupM = 8;       // rasterisation: 8 tile rows walk the N tiles together

__device__ __forceinline__ void tile_coords(int tile, int tiles_m, int tiles_n, int &tm, int &tn)
{
    const int group_size = kGroupM * tiles_n;
    const int first_m = (tile / group_size) * kGroupM;
    const int gm = min(tiles_m - first_m, kGroupM);
    const int local = tile % group_size;
    tm = first_m + local % gm;
    tn = local / gm;
}

// Wait (bounded) for the TMA loads the producer issued that the MMA warp may
// not have consumed: used only when a wait already timed out, so that no
// copy into shared memory is left in flight when the CTA exits.
__device__ __forceinline__ void drain_inflight(uint32_t full0, int stages, long issued, uint32_t *flags)
{
    for (long L = issued - stages < 0 ? 0 : issued - stages; L < issued; ++L)
        (void)mbar_wait(full0 + 8u * (uint32_t)(L % stages), (uint32_t)((L / stages) & 1), flags, 100000000ull);
}

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

// ============================================================ host helpers
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                   CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                   CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = []() -> EncodeTiledFn {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return nullptr;
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

// Tensor map over a plane set [S][rows][ldcomp] of BF16: dims (K, rows, S),
// box (kb, box_rows, 1), swizzle matching a kb * 2-byte row.  Out-of-range
// boxes (ragged M, N, K) read zeros.
bool make_plane_map(CUtensorMap *map, const uint16_t *planes, int64_t K, int64_t rows, int S, int64_t ldcomp,
                    int kb, int box_rows)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)rows, (cuuint64_t)S};
    cuuint64_t strides[2] = {(cuuint64_t)ldcomp * 2, (cuuint64_t)rows * ldcomp * 2};
    cuuint32_t box[3] = {(cuuint32_t)kb, (cuuint32_t)box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    const CUtensorMapSwizzle swz = (kb == 64) ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<uint16_t *>(planes), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int KB, int STAGES>
cudaError_t run_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                    float *C, int64_t ldc, uint32_t *flags, cudaStream_t st)
{
    using Cfg = F32Cfg<BN, KB, STAGES>;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, 3, ldcomp, KB, kBM) || !make_plane_map(&tb, Bp, K, N, 3, ldcomp, KB, BN))
        return cudaErrorInvalidValue;
    auto kern = prodsum_f32_kernel<BN, KB, STAGES>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int64_t tiles = ((M + kBM - 1) / kBM) * ((N + BN - 1) / BN);
    kern<<<(unsigned)tiles, Cfg::THREADS, Cfg::SMEM, st>>>(ta, tb, (int)M, (int)N, (int)K, C, ldc, flags);
    return cudaGetLastError();
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

// FP32 tile shape: 128 x 256 with 32-wide K-blocks (64-byte swizzle, 3 stages)
// by default; EMU_F32_TILE=128x128 selects 128 x 128 with 64-wide K-blocks
// (128-byte swizzle, 2 stages).
cudaError_t launch_prodsum_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                               int64_t ldcomp, float *C, int64_t ldc, uint32_t *flags, cudaStream_t st)
{
    static const bool narrow = [] {
        const char *e = std::getenv("EMU_F32_TILE");
        return e && e[0] == '1' && e[1] == '2' && e[2] == '8' && e[3] == 'x' && e[4] == '1';
    }();
    if (narrow) return run_f32<128, 64, 2>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st);
    return run_f32<256, 32, 3>(M, N, K, Ap, Bp, ldcomp, C, ldc, flags, st);
}

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

// ------------------------------------------------------- watchdog self-test
namespace {
__global__ void timeout_selftest_kernel(uint32_t *flags, unsigned long long limit_ns)
{
    __shared__ __align__(8) uint64_t bar;
    const uint32_t b = smem_u32(&bar);
    if (threadIdx.x == 0) { mbar_init(b, 1); fence_mbar_init(); }
    __syncthreads();
    if (threadIdx.x == 0) (void)mbar_wait(b, 0, flags, limit_ns);   // nothing ever arrives
    __syncthreads();
}
}  // namespace

cudaError_t launch_timeout_selftest(uint32_t *flags, uint32_t timeout_us, cudaStream_t st)
{
    timeout_selftest_kernel<<<1, 32, 0, st>>>(flags, 1000ull * timeout_us);
    return cudaGetLastError();
}

}  // namespace emu
