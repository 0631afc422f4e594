// FP64-mode tensor-core product-sum on 256-column output tiles, Eq.
// (fp64reconstruction) / Algorithm 2: the same arithmetic as the 128 x 128
// kernel (prodsum_f64.cu), bit for bit, with twice the output columns per CTA,
// and optionally (PAIR) twice the rows per MMA on a pair of SMs.
//
// Why wider: every MMA brings its A and B operands into the SM through shared
// memory, and for one product at a time nothing is reused across MMAs.  A
// 128 x 256 x 16 MMA takes in 12 KB of operands for 2^20 FLOP, a 128 x 128 x 16
// one 8 KB for 2^19, so this tile moves 0.75x the bytes per FLOP, the quantity
// that bounds the narrower kernel.  With PAIR a cluster of two CTAs on one TPC
// computes a 256 x 256 tile with cta_group::2 MMAs (M = 256): each CTA stages
// its 128 rows of the A slice and half of the B slice's 256 rows, the leader
// (cluster rank 0) issues the MMAs for both, and each CTA's TMEM receives its
// 128 x 256 part of the partials; per SM that is 8 KB of operands per 2^20
// FLOP.  Both CTAs' copies complete on the leader's stage barriers, the MMA
// commits arrive on both CTAs' barriers (multicast), and both CTAs' drain
// warps release a TMEM buffer on the leader's barrier.
//
// Products are taken in Algorithm 2's diagonal order (outer loop); for each
// product K is walked in chunks of 256 (B_K of Section 6.1), every chunk
// partial fl32(A_i B_j) formed on the tensor cores in one of two 256-column
// TMEM buffers (all 512 columns).  Partials are exact: slice entries are
// integers times 2^(v-8) of magnitude <= 256, so a chunk partial is an
// integer of at most 2^24 units u = 2^(vA_i + vB_j - 16).
//
// Sixteen drain warps (four per TMEM lane quarter, 64 columns each) sum a
// product's partials exactly in FP32 registers, as the narrow kernel does:
// plain additions while the running sum stays below 2^24 u; past that either
// a carry of the coarse part (multiples of 2^12 u) into a low word kept in C,
// or TwoSums whose errors are summed into that low word.
//
// Exact running sums for 128 x 256 elements take 64 registers in each of the
// 512 drain threads, which leaves no registers for fold warps.  So at the end
// of product q each drain thread hands its 64 exact sums (hi + lo, exact in
// FP64) to the L2 as FP64 reductions into the tile's accumulator in the
// workspace (red.global.add.f64, round to nearest even): the L2 performs
// Algorithm 2's step C <- fl64(C + A_i B_j) while the thread goes on with
// product q+1, and the SM's FP64 pipe, which on GB300 competes with the
// tensor cores, is not used at all.  Reductions of one thread to one address
// take effect in program order, so every element sees its products added in
// Algorithm 2's diagonal order.  Product 0 is stored rather than added (the
// accumulator need not be cleared); after the last product each thread reads
// its accumulator back (bypassing L1) and writes C.  The accumulator is
// column-major within the tile, so a warp's 32 rows of one column are 256
// contiguous bytes.  The result is bit-identical to the oracle in its
// product-outer order.
//
// Warp roles: warp 0 lane 0 issues TMA loads (four 48 KB stages, one 64-wide
// K-block of the A slice and the B slice each; PAIR: six 32 KB stages), warp
// 1 owns TMEM and lane 0 issues the MMAs (M = 128, N = 256; PAIR: the
// leader's, M = 256), warps 4-19 drain and reduce.  Every wait is bounded and
// reports EMU_FLAG_TIMEOUT instead of hanging.
#include "launchers.cuh"
#include "prodsum_f64_common.cuh"

namespace emu {

namespace {

// PAIR: a cluster of two CTAs computes a 256 x 256 tile with cta_group::2
// MMAs (M = 256); each CTA stages its 128 rows of the A slice and its 128-row
// half of the B slice and holds its 128 x 256 part of the partials, so a CTA
// takes in 8 KB of operands per 2^20 FLOP instead of 12 KB.
template <bool PAIR>
struct F64WCfgT {
    static constexpr int BN = 256, KB = 64, NBUF = 2;
    static constexpr int BH = PAIR ? BN / 2 : BN;                       // B rows staged by this CTA
    static constexpr int STAGES = PAIR ? 6 : 4;
    static constexpr int A_TILE = kBM * KB * 2, B_TILE = BH * KB * 2;   // 16 KB + 32 KB (pair: 16 KB)
    static constexpr int STAGE = A_TILE + B_TILE;
    static constexpr uint32_t SWZ = 2u, SBO = 1024u;                     // 128-byte swizzle
    static constexpr int BAR_OFF = STAGES * STAGE + (PAIR ? 16384 : 0);
    // barriers: full/empty per stage, tfull/tempty per buffer, done; then the TMEM address slot
    static constexpr int NBARS = 2 * STAGES + 2 * NBUF + 1;
    static constexpr int SMEM = BAR_OFF + 256 + 1024;
    // warpgroup 0: TMA producer (warp 0), MMA issuer + TMEM owner (warp 1), two
    // idle warps; warpgroups 1-4: sixteen drain warps
    static constexpr int FIRST_DRAIN = 4, DRAIN_WARPS = 16, THREADS = 20 * 32;
    static constexpr int COLS = BN / (DRAIN_WARPS / 4);                 // 64 columns per drain thread
    // Register split: the launch reserves 640 x 96; 128 x 32 (control) +
    // 512 x 112 (drain) = 61440 = 640 x 96.
    static constexpr int REG_CTRL = 32, REG_DRAIN = 112, REG_LAUNCH = 96;
    static constexpr int TILE_ELEMS = kBM * BN;
    static_assert(NBUF * BN == 512, "TMEM budget: two 256-column partial buffers");
    static_assert(kKChunk % KB == 0, "a K-chunk is a whole number of stages");
    static_assert(8 * NBARS + 8 <= 256, "barrier area");
    static_assert(SMEM <= 232448, "shared memory per CTA");
    static_assert(128 * REG_CTRL + 512 * REG_DRAIN <= THREADS * REG_LAUNCH,
                  "setmaxnreg split exceeds the registers reserved at launch");
    static_assert(COLS % 16 == 0, "drain columns come in groups of 16");
};
using F64WCfg = F64WCfgT<false>;

// FP64 reduction in L2: *p <- fl64(*p + x), round to nearest even.
__device__ __forceinline__ void red_add_f64(double *p, double x)
{
    asm volatile("red.global.add.f64 [%0], %1;" ::"l"(p), "d"(x) : "memory");
}

__device__ __forceinline__ double ld_cg_f64(const double *p)
{
    double x;
    asm volatile("ld.global.cg.f64 %0, [%1];" : "=d"(x) : "l"(p) : "memory");
    return x;
}

// TAIL: add the merged tail T (an M x N FP32 matrix) once after the last product.
template <int NPROD, bool ROWCOL, bool TAIL, bool PAIR>
__global__ void __launch_bounds__(F64WCfg::THREADS, 1)
prodsum_f64w_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmC, int c_tma, int M, int N, int K,
                    const int32_t *__restrict__ vA, const int32_t *__restrict__ vB, double *__restrict__ C,
                    int64_t ldc, double *__restrict__ acc, uint32_t *flags, const float *__restrict__ T, int64_t ldt)
{
    using Cfg = F64WCfgT<PAIR>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *base_ptr = smem_raw + (base - raw);
    const uint32_t full0 = base + Cfg::BAR_OFF, empty0 = full0 + 8u * Cfg::STAGES;
    const uint32_t tfull0 = empty0 + 8u * Cfg::STAGES, tempty0 = tfull0 + 8u * Cfg::NBUF;
    const uint32_t done_bar = tempty0 + 8u * Cfg::NBUF;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(base_ptr + Cfg::BAR_OFF + 8 * Cfg::NBARS);

    const int warp = threadIdx.x >> 5, lane = lane_id();
    const uint32_t rank = PAIR ? cluster_rank() : 0u;
    const int tiles_n = (N + Cfg::BN - 1) / Cfg::BN;
    int tm, tn;
    if constexpr (PAIR) {                             // the pair's 256 rows: this CTA takes half `rank`
        int tp;
        tile_coords((int)(blockIdx.x >> 1), (M + 2 * kBM - 1) / (2 * kBM), tiles_n, tp, tn);
        tm = 2 * tp + (int)rank;
    } else {
        tile_coords(blockIdx.x, (M + kBM - 1) / kBM, tiles_n, tm, tn);
    }
    const int m0 = tm * kBM, n0 = tn * Cfg::BN;
    const int nch = (K + kKChunk - 1) / kKChunk;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) { mbar_init(full0 + 8u * s, 1); mbar_init(empty0 + 8u * s, 1); }
        // a pair's TMEM buffers are released by the drain warps of both CTAs,
        // on the leader's barriers
        for (int b = 0; b < Cfg::NBUF; ++b) {
            mbar_init(tfull0 + 8u * b, 1);
            mbar_init(tempty0 + 8u * b, (PAIR ? 2 : 1) * Cfg::DRAIN_WARPS);
        }
        mbar_init(done_bar, 1);
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    if constexpr (PAIR) {
        __syncthreads();
        cluster_sync();                               // both CTAs' barriers initialised
        if (warp == 1) tmem_alloc_pair(smem_u32((const void *)tmem_slot), 512);
    } else {
        if (warp == 1) { tmem_alloc(smem_u32((const void *)tmem_slot), 512); tmem_relinquish(); }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp < Cfg::FIRST_DRAIN) {
      regs_dec<Cfg::REG_CTRL>();
      if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: for product, for chunk, for 64-wide K-block of the chunk
        int L = 0, s = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int q = 0; q < NPROD && ok; ++q) {
            const int ia = kDiag[q][0], jb = kDiag[q][1];
            for (int c = 0; c < nch && ok; ++c) {
                const int kbs = min(kKChunk / Cfg::KB, (K - c * kKChunk + Cfg::KB - 1) / Cfg::KB);
                for (int u = 0; u < kbs; ++u, ++L) {
                    if (!(ok = mbar_wait(empty0 + 8u * s, ph ^ 1u, flags))) break;
                    const uint32_t st = base + (uint32_t)(s * Cfg::STAGE), fb = full0 + 8u * s;
                    const int k0 = c * kKChunk + u * Cfg::KB;
                    if constexpr (PAIR) {
                        // both CTAs' copies are counted on the leader's full barrier
                        const uint32_t fl = peer_addr(fb, 0);
                        if (rank == 0) mbar_arrive_expect_tx(fb, 2 * Cfg::STAGE);
                        tma_load_3d_pair(st, &tmA, fl, k0, m0, ia);
                        tma_load_3d_pair(st + Cfg::A_TILE, &tmB, fl, k0, n0 + (int)rank * Cfg::BH, jb);
                    } else {
                        mbar_arrive_expect_tx(fb, Cfg::STAGE);
                        tma_load_3d(st, &tmA, fb, k0, m0, ia);
                        tma_load_3d(st + Cfg::A_TILE, &tmB, fb, k0, n0, jb);
                    }
                    if (++s == Cfg::STAGES) { s = 0; ph ^= 1u; }
                }
            }
        }
        if (!ok) {
            if (rank == 0) {
                drain_inflight(full0, Cfg::STAGES, L, flags);
            } else {
                // the peer's copies complete on the leader's barriers, which it
                // cannot observe: give them 200 us before the CTA winds down
                const unsigned long long t0 = globaltimer_ns();
                while (globaltimer_ns() - t0 < 200000ull) {}
            }
        }
      } else if (warp == 1 && lane == 0 && rank == 0) {
        // ---------------- MMA issuer (a pair's leader): one chunk partial into buffer t % NBUF
        constexpr uint32_t idesc = make_idesc_bf16(PAIR ? 2 * kBM : kBM, Cfg::BN);
        int s = 0, b = 0;
        uint32_t ph = 0, tph = 0;
        bool ok = true;
        for (int t = 0; t < NPROD * nch && ok; ++t) {
            const int c = t % nch;
            const int kbs = min(kKChunk / Cfg::KB, (K - c * kKChunk + Cfg::KB - 1) / Cfg::KB);
            if (!(ok = mbar_wait(tempty0 + 8u * b, tph ^ 1u, flags))) break;
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(b * Cfg::BN);
            for (int u = 0; u < kbs; ++u) {
                if (!(ok = mbar_wait(full0 + 8u * s, ph, flags))) break;
                tc_fence_after();
                const uint32_t st = base + (uint32_t)(s * Cfg::STAGE);
#pragma unroll
                for (int kk = 0; kk < Cfg::KB / 16; ++kk) {
                    const uint64_t ad = make_sdesc(st + kk * 32, Cfg::SBO, Cfg::SWZ);
                    const uint64_t bd = make_sdesc(st + Cfg::A_TILE + kk * 32, Cfg::SBO, Cfg::SWZ);
                    if constexpr (PAIR) mma_bf16_pair(d, ad, bd, idesc, (u | kk) != 0);
                    else mma_bf16(d, ad, bd, idesc, (u | kk) != 0);
                }
                if constexpr (PAIR) mma_commit_pair(empty0 + 8u * s);
                else mma_commit(empty0 + 8u * s);
                if (++s == Cfg::STAGES) { s = 0; ph ^= 1u; }
            }
            if (ok) {
                if constexpr (PAIR) mma_commit_pair(tfull0 + 8u * b);
                else mma_commit(tfull0 + 8u * b);
            }
            if (++b == Cfg::NBUF) { b = 0; tph ^= 1u; }
        }
        if constexpr (PAIR) mma_commit_pair(done_bar);
        else mma_commit(done_bar);
        (void)mbar_wait(done_bar, 0, flags);
      }
    } else {
        regs_inc<Cfg::REG_DRAIN>();
        // ---------------- drain: exact per-product sums, reduced into the accumulator in L2
        const int quarter = warp & 3;                                    // TMEM lanes 32*quarter ..
        const int cq = (warp - Cfg::FIRST_DRAIN) >> 2;                   // column quarter
        const int r = quarter * 32 + lane;                               // tile row of this thread
        const uint32_t tcol = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(cq * Cfg::COLS);
        const int row = m0 + r;
        double *crow = C + (int64_t)row * ldc + n0 + cq * Cfg::COLS;
        const int lim = row < M ? N - (n0 + cq * Cfg::COLS) : 0;        // valid columns of this thread
        // this thread's elements of the tile's accumulator (column-major)
        double *tacc = acc + ((size_t)tm * tiles_n + tn) * Cfg::TILE_ELEMS + (size_t)(cq * Cfg::COLS) * kBM + r;
        // a pair's second CTA may lie wholly below the last row, past the
        // accumulator's tiles: its threads touch neither the accumulator nor C
        const bool live = !PAIR || row < M;
        // the low words live in one half of this thread's C words until their product is reduced
        float *lrow = reinterpret_cast<float *>(crow);
        float hi[Cfg::COLS];
        bool ok = true;
        for (int q = 0; q < NPROD && ok; ++q) {
#pragma unroll
            for (int j = 0; j < Cfg::COLS; ++j) hi[j] = 0.0f;
            uint32_t dirty = 0;                           // 16-column groups whose low part lives in C
            const float bound = ROWCOL ? exact_bound_rowcol(vA, vB, M, N, kDiag[q][0], kDiag[q][1], row,
                                                            n0 + cq * Cfg::COLS, Cfg::COLS)
                                       : exact_bound(vA, vB, kDiag[q][0], kDiag[q][1]);
            // Carry instead of TwoSums when all elements share the unit u = 2^-24 bound
            // (levels per matrix) and the split constant 1.5 * 2^35 u is finite.  A
            // carry splits the running sum and the partial (each at most 2^24 u) at
            // multiples of 2^12 u and moves both coarse parts (together at most
            // 2^25 u) to the low word in C, which stays exact below 2^36 u, i.e. for
            // up to 2^11 carries.
            const bool carry = !ROWCOL && bound > 0.0f && bound <= 0x1p116f && nch <= 2048;
            const int a_row = (ROWCOL && row < M) ? vA[(int64_t)kDiag[q][0] * M + row] : kZeroLevel;
            for (int c = 0; c < nch; ++c) {
                const int t = q * nch + c, b = t % Cfg::NBUF;
                ok = mbar_wait(tfull0 + 8u * b, (uint32_t)((t / Cfg::NBUF) & 1), flags);
                __syncwarp();
                if (!ok) break;
                tc_fence_after();
#pragma unroll
                for (int h = 0; h < Cfg::COLS; h += 16) {
                    const uint32_t taddr = tcol + (uint32_t)(b * Cfg::BN + h);
                    uint32_t v[16];                           // the partials, then the sums
                    tmem_ld16(taddr, v);
                    tmem_ld_wait();
                    bool big = false;
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const float sm = __fadd_rn(hi[h + j], __uint_as_float(v[j]));
                        big |= !(fabsf(sm) < bound);
                        v[j] = __float_as_uint(sm);
                    }
                    if (!__any_sync(0xFFFFFFFFu, big)) {
#pragma unroll
                        for (int j = 0; j < 16; ++j) hi[h + j] = __uint_as_float(v[j]);
                    } else if (carry) {
                        // rare: some sum would reach 2^24 u.  Split the running sum and
                        // the partial (read again from TMEM: the buffer is not yet
                        // released) at multiples of 2^12 u by the add-subtract
                        // projection; the coarse parts go to the low word in C, the
                        // remainders (below 2^12 u) restart the running sum.  All exact.
                        const bool was = (dirty >> (h / 16)) & 1u;
                        dirty |= 1u << (h / 16);
                        const float cm = 3072.0f * bound;         // 1.5 * 2^35 u
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj) {
                            const int j = h + jj;
                            const float p = __uint_as_float(tmem_ld1(taddr + (uint32_t)jj));
                            tmem_ld_wait();
                            const float h1 = __fsub_rn(__fadd_rn(hi[j], cm), cm), l1 = __fsub_rn(hi[j], h1);
                            const float h2 = __fsub_rn(__fadd_rn(p, cm), cm), l2 = __fsub_rn(p, h2);
                            const bool mine = j < lim;
                            const float s2 = __fadd_rn((was && mine) ? lrow[2 * j] : 0.0f, __fadd_rn(h1, h2));
                            hi[j] = __fadd_rn(l1, l2);
                            if (mine) lrow[2 * j] = s2;
                        }
                    } else {
                        // rare: redo the 16 additions as TwoSums, the errors summed
                        // exactly into the low part; with levels per row / column an
                        // element whose own unit allows it takes the carry instead
                        // (its own split constant).
                        const bool was = (dirty >> (h / 16)) & 1u;
                        dirty |= 1u << (h / 16);
                        const float renorm = 0.5f * bound;        // lo is kept below 2^23 u
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj) {
                            const int j = h + jj;
                            const float p = __uint_as_float(tmem_ld1(taddr + (uint32_t)jj));
                            tmem_ld_wait();
                            const bool mine = j < lim;
                            float be = 0.0f;
                            if (ROWCOL && mine && nch <= 2048)
                                be = bound_of_levels(a_row, vB[(int64_t)kDiag[q][1] * N + n0 + cq * Cfg::COLS + j]);
                            if (be > 0.0f && be <= 0x1p116f) {
                                const float cm = 3072.0f * be;
                                const float h1 = __fsub_rn(__fadd_rn(hi[j], cm), cm), l1 = __fsub_rn(hi[j], h1);
                                const float h2 = __fsub_rn(__fadd_rn(p, cm), cm), l2 = __fsub_rn(p, h2);
                                lrow[2 * j] = __fadd_rn(was ? lrow[2 * j] : 0.0f, __fadd_rn(h1, h2));
                                hi[j] = __fadd_rn(l1, l2);
                            } else {
                                float e, lo;
                                const float sm = two_sum(hi[j], p, e);
                                lo = __fadd_rn((was && mine) ? lrow[2 * j] : 0.0f, e);
                                hi[j] = (fabsf(lo) < renorm) ? sm : two_sum(sm, lo, lo);   // renormalise (hi, lo)
                                if (mine) lrow[2 * j] = lo;
                            }
                        }
                    }
                    if (h + 16 == Cfg::COLS) {                   // buffer free: all values are in registers
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) {
                            if constexpr (PAIR) mbar_arrive_peer(peer_addr(tempty0 + 8u * b, 0));
                            else mbar_arrive(tempty0 + 8u * b);
                        }
                    }
                }
            }
            if (!ok) break;
            // C <- fl64(C + (hi + lo)) in L2, column by column (product 0: a plain store).
            // The sums are integer multiples of the smallest unit of this thread's
            // elements, 2^-24 bound; when that unit is a normal FP32 number so is
            // every nonzero sum, and the short widening is exact.
            // The common case (no low words, normal unit) is a branch of its own
            // with integer widening only: written as selects, the rare path's
            // FP64 additions and general widening would run for every element
            // (GB300's FP64 pipe does about one warp-wide add per 32 clocks per
            // SM sub-partition).
            const bool normal_sums = bound >= 0x1p-102f;
            if (live && dirty == 0 && normal_sums) {
                if (q == 0) {
#pragma unroll
                    for (int j = 0; j < Cfg::COLS; ++j) tacc[j * kBM] = widen_normal(hi[j]);
                } else {
#pragma unroll
                    for (int j = 0; j < Cfg::COLS; ++j) red_add_f64(tacc + j * kBM, widen_normal(hi[j]));
                }
            } else if (live) {
#pragma unroll
                for (int j = 0; j < Cfg::COLS; ++j) {
                    double sq = normal_sums ? widen_normal(hi[j]) : widen_exact(hi[j]);
                    if (((dirty >> (j >> 4)) & 1u) && j < lim) sq = __dadd_rn(sq, widen_exact(lrow[2 * j]));   // exact
                    if (q == 0) tacc[j * kBM] = sq;
                    else red_add_f64(tacc + j * kBM, sq);
                }
            }
        }
        // The warp takes the bulk-copy branch together (its __syncwarp and the
        // copies lane 0 issues need every lane) when no lane's wait timed out and
        // one of its rows is live (a pair's second CTA may reach past the last
        // row).  Lanes of rows past M read their accumulator elements (inside the
        // tile, never written) and the copies leave those rows out.
        const bool warp_ok = __all_sync(0xFFFFFFFFu, ok), warp_live = __any_sync(0xFFFFFFFFu, live);
        if (warp_ok && warp_live && c_tma && !TAIL) {
            // the accumulator holds every product now (this thread's own reductions,
            // same addresses, so they precede these loads): C <- acc through the TMA
            // engine.  Each 32 x 16 piece of the warp's rows (4 KB, two alternating
            // buffers per warp in the stage memory, which every MMA has finished
            // reading) is staged in the 128-byte-swizzled layout of the C map and
            // written by one bulk tensor store: whole 128-byte row segments, where
            // the per-lane stores below touch one cache line per row and lane.
            const uint32_t bufs = base + (uint32_t)(warp - Cfg::FIRST_DRAIN) * 8192u;
            fence_proxy_async_global();       // this thread's low-word writes to C precede the copies
            __syncwarp();
#pragma unroll 1
            // pieces wholly past the last column are neither staged nor copied
            for (int j0 = 0, g = 0; j0 < Cfg::COLS && n0 + cq * Cfg::COLS + j0 < N; j0 += 16, ++g) {
                const uint32_t buf = bufs + (uint32_t)(g & 1) * 4096u;
                if (g >= 2) {                 // the copy that last read this buffer
                    if (lane == 0) bulk_wait_read<1>();
                    __syncwarp();
                }
                const uint32_t srow = buf + (uint32_t)lane * 128u;
#pragma unroll
                for (int h = 0; h < 16; h += 8) {         // eight columns at a time: few live registers
                    double out[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) out[j] = ld_cg_f64(tacc + (j0 + h + j) * kBM);
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const unsigned long long a = (unsigned long long)__double_as_longlong(out[2 * k]);
                        const unsigned long long b = (unsigned long long)__double_as_longlong(out[2 * k + 1]);
                        st_shared_v4(srow + ((uint32_t)((h / 2 + k) ^ (lane & 7)) << 4), (uint32_t)a,
                                     (uint32_t)(a >> 32), (uint32_t)b, (uint32_t)(b >> 32));
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&tmC, buf, n0 + cq * Cfg::COLS + j0, m0 + quarter * 32);
                    bulk_commit();
                }
            }
            if (lane == 0) bulk_wait_read<0>();
            __syncwarp();
        } else if (ok && live && !(c_tma && !TAIL)) {
            // the accumulator holds every product now (this thread's own reductions,
            // same addresses, so they precede these loads): C <- acc (+ the merged tail)
            const float *trow = TAIL ? T + (int64_t)(row < M ? row : 0) * ldt + n0 + cq * Cfg::COLS : nullptr;
            const bool vec = ((ldc & 1) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15u) == 0);
#pragma unroll 1
            for (int j0 = 0; j0 < Cfg::COLS; j0 += 8) {
                double out[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) out[j] = ld_cg_f64(tacc + (j0 + j) * kBM);
                if (TAIL) {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        if (j0 + j < lim) out[j] = __dadd_rn(out[j], widen_exact(trow[j0 + j]));
                }
                if (vec && lim >= j0 + 8) {
#pragma unroll
                    for (int j = 0; j < 8; j += 2)
                        *reinterpret_cast<double2 *>(crow + j0 + j) = make_double2(out[j], out[j + 1]);
                } else {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        if (j0 + j < lim) crow[j0 + j] = out[j];
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if constexpr (PAIR) cluster_sync();               // the leader's MMAs are done with both CTAs
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        if constexpr (PAIR) tmem_dealloc_pair(tmem, 512);
        else tmem_dealloc(tmem, 512);
    }
}

// tiles: the first `tiles` tiles in raster order (all of them, or the full
// waves when the narrow kernel takes the rest): 128 x 256 tiles, one CTA
// each, or with PAIR 256 x 256 tiles, one cluster of two CTAs each.
template <int NPROD, bool ROWCOL, bool TAIL, bool PAIR>
cudaError_t run_f64w(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                     const int32_t *vA, const int32_t *vB, double *C, int64_t ldc, double *acc, uint32_t *flags,
                     cudaStream_t st, int64_t a_plane, const float *T, int64_t ldt, int64_t tiles)
{
    using Cfg = F64WCfgT<PAIR>;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, 6, ldcomp, Cfg::KB, kBM, a_plane) ||
        !make_plane_map(&tb, Bp, K, N, 6, ldcomp, Cfg::KB, Cfg::BH))
        return cudaErrorInvalidValue;
    static_assert(Cfg::DRAIN_WARPS * 8192 <= Cfg::STAGES * Cfg::STAGE, "TMA epilogue staging exceeds the stages");
    CUtensorMap tc = {};
    const int c_tma = make_c_map_f64(&tc, C, M, N, ldc) ? 1 : 0;
    auto kern = prodsum_f64w_kernel<NPROD, ROWCOL, TAIL, PAIR>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((PAIR ? 2 : 1) * tiles));
    cfg.blockDim = dim3(Cfg::THREADS);
    cfg.dynamicSmemBytes = Cfg::SMEM;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = PAIR ? 2 : 1;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = PAIR ? 1 : 0;
    e = cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, c_tma, (int)M, (int)N, (int)K, vA, vB, C, ldc, acc, flags, T, ldt);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

template <bool PAIR>
cudaError_t dispatch_f64w(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                          const int32_t *vA, const int32_t *vB, int nprod, double *C, int64_t ldc, double *acc,
                          uint32_t *flags, cudaStream_t st, int64_t a_plane, bool rowcol, const float *T, int64_t ldt,
                          int64_t tiles)
{
#define EMU_F64W(NP, RC, TL) \
    run_f64w<NP, RC, TL, PAIR>(M, N, K, Ap, Bp, ldcomp, vA, vB, C, ldc, acc, flags, st, a_plane, T, ldt, tiles)
    if (T) {                                          // merged tail: whole-matrix levels only
        if (rowcol) return cudaErrorInvalidValue;
        switch (nprod) {
        case 6: return EMU_F64W(6, false, true);
        case 10: return EMU_F64W(10, false, true);
        case 15: return EMU_F64W(15, false, true);
        default: return cudaErrorInvalidValue;
        }
    }
    switch (nprod) {
    case 6: return rowcol ? EMU_F64W(6, true, false) : EMU_F64W(6, false, false);
    case 10: return rowcol ? EMU_F64W(10, true, false) : EMU_F64W(10, false, false);
    case 15: return rowcol ? EMU_F64W(15, true, false) : EMU_F64W(15, false, false);
    case 21: return rowcol ? EMU_F64W(21, true, false) : EMU_F64W(21, false, false);
    default: return cudaErrorInvalidValue;
    }
#undef EMU_F64W
}

}  // namespace

cudaError_t launch_prodsum_f64_wide(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                                    int64_t ldcomp, const int32_t *vA, const int32_t *vB, int nprod, double *C,
                                    int64_t ldc, double *acc, uint32_t *flags, cudaStream_t st, int64_t a_plane,
                                    bool rowcol, const float *T, int64_t ldt, int64_t tiles, bool pair)
{
    return pair ? dispatch_f64w<true>(M, N, K, Ap, Bp, ldcomp, vA, vB, nprod, C, ldc, acc, flags, st, a_plane, rowcol,
                                      T, ldt, tiles)
                : dispatch_f64w<false>(M, N, K, Ap, Bp, ldcomp, vA, vB, nprod, C, ldc, acc, flags, st, a_plane, rowcol,
                                       T, ldt, tiles);
}

}  // namespace emu
