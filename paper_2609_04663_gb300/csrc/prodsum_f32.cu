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
#include "split_f32_pair.cuh"

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

// Epilogue of one warp: accumulator columns [c0, c1) of the warp's TMEM lane
// quarter (tile rows quarter * 32 ..) -> C.
__device__ __forceinline__ void store_tile(uint32_t tmem, int quarter, int c0, int c1, int m0, int n0, int M, int N,
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
        mma_loop<BN, KB, STAGES>(tmem, base, full0, empty0, accum_bar, nkb, flags);
    } else if (warp >= 2) {
        // ---------------- epilogue: TMEM -> registers -> C
        const bool ok = mbar_wait(accum_bar, 0, flags);
        __syncwarp();
        if (ok) store_tile(tmem, warp & 3, 0, BN, m0, n0, M, N, C, ldc);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, BN);
    }
}

// ------------------------------------------------- split fused into the producer
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

__device__ __forceinline__ void st_shared_v2(uint32_t addr, uint32_t a, uint32_t b)
{
    asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr), "r"(a), "r"(b) : "memory");
}
__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d)
{
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
// Makes this thread's shared-memory stores visible to the tensor cores
// (async proxy) before it signals the stage as full.
__device__ __forceinline__ void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void prefetch_l2(const void *p)
{
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// What one of CONV converter threads holds of a 128 x 32 A tile and a 32 x 256
// B tile: float4 number ct % 8 of A rows ct / 8 + (CONV / 8) i, and B column
// ct % 256 over the K rows KPT (ct / 256) .. + KPT - 1.
template <int CONV>
struct FusedTiles {
    static constexpr int NA = 1024 / CONV, KPT = 32 * 256 / CONV;
    float a[NA][4];
    float b[KPT];
};

template <int BN, int KB, int STAGES, int CONV>
__global__ void __launch_bounds__(32 + CONV, 1)
gemm_f32_fused_kernel(const float *__restrict__ A, int64_t lda, const float *__restrict__ B, int64_t ldb, int M,
                      int N, int K, float *__restrict__ C, int64_t ldc, uint32_t *flags)
{
    using Cfg = F32Cfg<BN, KB, STAGES>;
    static_assert(BN == 256 && KB == 32 && (CONV == 256 || CONV == 512), "converter mapping");
    using Tiles = FusedTiles<CONV>;
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
        const int b_col = ct & 255, b_k0 = (ct >> 8) * Tiles::KPT;
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
        // one 128-byte line per thread and operand: A row ct, B K row ct / 8 segment ct % 8
        auto prefetch = [&](int kb) {
            const int k0 = kb * KB;
            if (ct < kBM && m0 + ct < M) prefetch_l2(A + (int64_t)(m0 + ct) * lda + k0);
            const int k = k0 + (ct >> 3), n = n0 + 32 * (ct & 7);
            if (ct < 256 && k < K && n < N) prefetch_l2(B + (int64_t)k * ldb + n);
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

// FP32-mode GEMM with the split in the producer (gemm_f32_fused_kernel).
cudaError_t launch_gemm_f32_fused(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda, const float *B,
                                  int64_t ldb, float *C, int64_t ldc, uint32_t *flags, cudaStream_t st)
{
    constexpr int kConv = 512;
    using Cfg = F32Cfg<256, 32, 3>;
    auto kern = gemm_f32_fused_kernel<256, 32, 3, kConv>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int64_t tiles = ((M + kBM - 1) / kBM) * ((N + 255) / 256);
    kern<<<(unsigned)tiles, 32 + kConv, Cfg::SMEM, st>>>(A, lda, B, ldb, (int)M, (int)N, (int)K, C, ldc,
                                                               flags);
    return cudaGetLastError();
}

}  // namespace emu
