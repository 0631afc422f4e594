// FP32-mode GEMM in one kernel: the split of Eq. (fp32split) inside the
// tensor-core product-sum of Eq. (fp32six).
#include "launchers.cuh"
#include "prodsum_f32_common.cuh"
#include "split_f32_pair.cuh"

namespace emu {

namespace {

// The FP32-mode GEMM in one kernel: the split of Eq. (fp32split) runs inside
// the product-sum's producer, on the tiles each CTA is about to multiply (the
// streamed-slice variant of Section 6.2, which the AMX design sets aside
// because every panel re-splits its slices).  Tile, stage layout, MMA order and
// accumulator are those of prodsum_f32_kernel<256, 32, 3>, and the slices are
// formed by the same pair arithmetic as the split kernels, so C is
// bit-identical to split + product-sum.
//
// Warp 0 owns TMEM and its lane 0 issues the MMAs.  CONV converter threads
// (warps 1 ..) load the FP32 tiles of A (128 x 32) and B (32 x 256) one K-block
// ahead with coalesced loads, prefetch four K-blocks ahead into L2, split in
// registers and store the slices into the stage in the 64-byte-swizzled
// K-major layout that a TMA copy of the planes would have produced (16-byte
// chunk c of row r at chunk c ^ ((r >> 1) & 3)); each warp then signals the
// stage once.  After the last K-block they run the epilogue.  A converter
// thread takes float4 number ct % 8 of A rows ct / 8 + (CONV / 8) i (a warp
// reads four whole 128-byte rows per load) and column ct % 256 of B over
// 32 * 256 / CONV consecutive K rows (a warp reads 128 contiguous bytes per
// K row), which form part of row ct % 256 of the transposed B slices.  Both
// store patterns are free of bank conflicts, and the shared-memory traffic
// equals that of the TMA-fed kernel.
//
// Cost: a CTA splits every tile it multiplies, so each element of A is split
// once per 256-column tile of C and each element of B once per 128-row tile
// (32 and 64 times at 8192^3).  With 16 converter warps this kernel is
// slower than split + product-sum (4.1 against 3.45 ms at 8192^3): the
// repeated split arithmetic and the loads keep the schedulers two-thirds busy
// and leave the tensor pipe idle 28 % of the time.
constexpr int kFusedPrefetch = 4;        // K-blocks between the L2 prefetch and the loads

__device__ __forceinline__ void prefetch_l2(const void *p)
{
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// What one of CONV converter threads holds of a 128 x 32 A tile and a 32 x BN
// B tile: float4 number ct % 8 of A rows ct / 8 + (CONV / 8) i, and B column
// ct % BN over the K rows KPT (ct / BN) .. + KPT - 1 (KPT >= 8, so that a
// thread fills whole 16-byte chunks of its transposed B row).
template <int BN, int CONV>
struct FusedTiles {
    static constexpr int NA = 1024 / CONV, KPT = 32 * BN / CONV;
    static_assert(KPT >= 8 && KPT % 8 == 0 && CONV % BN == 0, "converter mapping of the B tile");
    float a[NA][4];
    float b[KPT];
};

template <int BN, int KB, int STAGES, int CONV>
__global__ void __launch_bounds__(32 + CONV, 1)
gemm_f32_fused_kernel(const float *__restrict__ A, int64_t lda, const float *__restrict__ B, int64_t ldb, int M,
                      int N, int K, float *__restrict__ C, int64_t ldc, uint32_t *flags)
{
    using Cfg = F32Cfg<BN, KB, STAGES>;
    static_assert(KB == 32 && (CONV == 256 || CONV == 512), "converter mapping");
    using Tiles = FusedTiles<BN, CONV>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *base_ptr = smem_raw + (base - raw);
    const uint32_t full0 = base + Cfg::BAR_OFF, empty0 = full0 + 8u * STAGES;
    const uint32_t accum_bar = empty0 + 8u * STAGES;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(base_ptr + Cfg::BAR_OFF + 16 * STAGES + 8);

    const int warp = threadIdx.x >> 5;
    const int tiles_m = (M + kBM - 1) / kBM, tiles_n = (N + BN - 1) / BN;
    int tm, tn;
    tile_coords(blockIdx.x, tiles_m, tiles_n, tm, tn);
    const int m0 = tm * kBM, n0 = tn * BN;
    const int nkb = (K + KB - 1) / KB;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) { mbar_init(full0 + 8u * s, CONV / 32); mbar_init(empty0 + 8u * s, 1); }
        mbar_init(accum_bar, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(smem_u32((const void *)tmem_slot), BN); tmem_relinquish(); }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane_id() == 0) mma_loop<BN, KB, STAGES>(tmem, base, full0, empty0, accum_bar, nkb, flags);
    } else {
        const int ct = threadIdx.x - 32;
        const int a_c4 = ct & 7, a_r0 = ct >> 3;
        const int b_col = ct % BN, b_k0 = (ct / BN) * Tiles::KPT;
        const int bn = n0 + b_col;
        const bool avec = ((lda & 3) == 0) && ((reinterpret_cast<uintptr_t>(A) & 15u) == 0);

        auto load = [&](int kb, Tiles &t) {
            const int k0 = kb * KB;
#pragma unroll
            for (int i = 0; i < Tiles::NA; ++i) {
                const int m = m0 + a_r0 + (CONV / 8) * i, k = k0 + 4 * a_c4;
                const float *src = A + (int64_t)(m < M ? m : 0) * lda + k;
                if (m < M && avec && k + 4 <= K) {
                    const float4 v = __ldg(reinterpret_cast<const float4 *>(src));
                    t.a[i][0] = v.x; t.a[i][1] = v.y; t.a[i][2] = v.z; t.a[i][3] = v.w;
                } else {
#pragma unroll
                    for (int e = 0; e < 4; ++e) t.a[i][e] = (m < M && k + e < K) ? __ldg(src + e) : 0.0f;
                }
            }
            const int kb0 = k0 + b_k0;
            const float *bsrc = B + (int64_t)kb0 * ldb + (bn < N ? bn : 0);
            if (bn < N && kb0 + Tiles::KPT <= K) {
#pragma unroll
                for (int k = 0; k < Tiles::KPT; ++k) t.b[k] = __ldg(bsrc + (int64_t)k * ldb);
            } else {
#pragma unroll
                for (int k = 0; k < Tiles::KPT; ++k)
                    t.b[k] = (bn < N && kb0 + k < K) ? __ldg(bsrc + (int64_t)k * ldb) : 0.0f;
            }
        };
        // one 128-byte line per thread and operand: A row ct, B K row ct / L segment ct % L
        // (L = BN / 32 lines per K row of the B tile)
        auto prefetch = [&](int kb) {
            constexpr int L = BN / 32;
            const int k0 = kb * KB;
            if (ct < kBM && m0 + ct < M) prefetch_l2(A + (int64_t)(m0 + ct) * lda + k0);
            const int k = k0 + ct / L, n = n0 + 32 * (ct % L);
            if (ct < 32 * L && k < K && n < N) prefetch_l2(B + (int64_t)k * ldb + n);
        };
        uint32_t amax = 0;
        auto store = [&](uint32_t st, const Tiles &t) {
#pragma unroll
            for (int i = 0; i < Tiles::NA; ++i) {
                const int r = a_r0 + (CONV / 8) * i;
                uint32_t w[3][2];
                amax = abs_bits_max(abs_bits_max(amax, t.a[i][0], t.a[i][1]), t.a[i][2], t.a[i][3]);
                split_pair(t.a[i][0], t.a[i][1], w[0][0], w[1][0], w[2][0]);
                split_pair(t.a[i][2], t.a[i][3], w[0][1], w[1][1], w[2][1]);
                const uint32_t off = (uint32_t)r * 64u + ((uint32_t)((a_c4 >> 1) ^ ((r >> 1) & 3)) << 4) +
                                     ((uint32_t)(a_c4 & 1) << 3);
#pragma unroll
                for (int p = 0; p < 3; ++p) st_shared_v2(st + p * Cfg::A_TILE + off, w[p][0], w[p][1]);
            }
#pragma unroll
            for (int cc = 0; cc < Tiles::KPT / 8; ++cc) {
                const int c = b_k0 / 8 + cc;        // 16-byte chunk of the transposed row
                uint32_t w[3][4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    amax = abs_bits_max(amax, t.b[8 * cc + 2 * e], t.b[8 * cc + 2 * e + 1]);
                    split_pair(t.b[8 * cc + 2 * e], t.b[8 * cc + 2 * e + 1], w[0][e], w[1][e], w[2][e]);
                }
                const uint32_t off = (uint32_t)b_col * 64u + ((uint32_t)(c ^ ((b_col >> 1) & 3)) << 4);
#pragma unroll
                for (int p = 0; p < 3; ++p)
                    st_shared_v4(st + 3 * Cfg::A_TILE + p * Cfg::B_TILE + off, w[p][0], w[p][1], w[p][2], w[p][3]);
            }
        };
        // K-block kb from `cur` while `nxt` receives kb + 1; false after a timeout
        auto step = [&](int kb, const Tiles &cur, Tiles &nxt) -> bool {
            const int s = kb % STAGES;
            if (kb + 1 < nkb) load(kb + 1, nxt);
            if (kb + 1 + kFusedPrefetch < nkb) prefetch(kb + 1 + kFusedPrefetch);
            if (!mbar_wait(empty0 + 8u * s, ((kb / STAGES) & 1) ^ 1, flags)) return false;
            store(base + (uint32_t)(s * Cfg::STAGE), cur);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane_id() == 0) mbar_arrive(full0 + 8u * s);     // one arrival per converter warp
            return true;
        };
        Tiles t0, t1;
        for (int p = 1; p <= kFusedPrefetch && p < nkb; ++p) prefetch(p);
        if (nkb > 0) load(0, t0);
#pragma unroll 1
        for (int kb = 0; kb < nkb; kb += 2) {
            if (!step(kb, t0, t1)) break;
            if (kb + 1 < nkb && !step(kb + 1, t1, t0)) break;
        }
        publish_f32_flags(amax, flags);
        // epilogue: CONV / 128 warps per TMEM lane quarter, an equal share of the columns each
        constexpr int kPart = BN / (CONV / 128);
        static_assert(kPart % 32 == 0, "epilogue columns come in groups of 32");
        const bool ok = mbar_wait(accum_bar, 0, flags);
        __syncwarp();
        const int part = (warp - 1) >> 2;
        if (ok) store_tile(tmem, warp & 3, part * kPart, (part + 1) * kPart, m0, n0, M, N, C, ldc);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, BN);
    }
}

}  // namespace

template <int BN, int STAGES, int CONV>
cudaError_t run_fused(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda, const float *B, int64_t ldb,
                      float *C, int64_t ldc, uint32_t *flags, cudaStream_t st)
{
    using Cfg = F32Cfg<BN, 32, STAGES>;
    auto kern = gemm_f32_fused_kernel<BN, 32, STAGES, CONV>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int64_t tiles = ((M + kBM - 1) / kBM) * ((N + BN - 1) / BN);
    kern<<<(unsigned)tiles, 32 + CONV, Cfg::SMEM, st>>>(A, lda, B, ldb, (int)M, (int)N, (int)K, C, ldc, flags);
    return cudaGetLastError();
}

// FP32-mode GEMM with the split in the producer (gemm_f32_fused_kernel), on
// the tile width the product-sum would take for this result size (128 x 256,
// 128 x 128 or 128 x 64): every width issues the same MMAs in the same order
// for each output element, so C does not depend on it.
cudaError_t launch_gemm_f32_fused(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda, const float *B,
                                  int64_t ldb, float *C, int64_t ldc, uint32_t *flags, cudaStream_t st)
{
    switch (f32_tile_columns(M, N)) {
    case 64: return run_fused<64, 4, 256>(M, N, K, A, lda, B, ldb, C, ldc, flags, st);
    case 128: return run_fused<128, 4, 256>(M, N, K, A, lda, B, ldb, C, ldc, flags, st);
    default: return run_fused<256, 3, 512>(M, N, K, A, lda, B, ldb, C, ldc, flags, st);
    }
}

}  // namespace emu
