// FP64-mode tensor-core product-sum, Eq. (fp64reconstruction) / Algorithm 2.
//
// Products are taken in Algorithm 2's diagonal order (outer loop); for each
// product the K dimension is walked in chunks of 256 (B_K of Section 6.1).
// Every chunk partial fl32(A_i B_j) is formed on the tensor cores in its own
// TMEM buffer (two rotating 128-column buffers).  The partials are exact:
// slice entries are integers times 2^(v-8) of magnitude <= 256, so a chunk
// partial is an integer of at most 2^24 units u = 2^(vA_i + vB_j - 16).
//
// Sixteen drain warps sum the partials of one product exactly in FP32
// registers: while the running sum hi stays below 2^24 u (known from the
// split's level exponents) a plain FP32 addition is exact.  Past that bound
// the error of each addition is recovered with Knuth's TwoSum and summed into
// a low part lo, an FP32 word kept in the output buffer C (free scratch until
// the last product; even products use one half of each C word, odd products
// the other); (hi, lo) is renormalised by another TwoSum whenever lo reaches
// 2^23 u, so the additions into lo are exact for any K.
//
// A finished product's sums go through a 128-column TMEM hand-off area to
// four fold warps, which add hi + lo (exact in FP64) once into the FP64
// accumulator: C <- fl64(C + fl32(A_i B_j)), Algorithm 2's step.  GB300's
// FP64 pipe does two adds per clock per SM, so a product's 128 x 128 FP64
// adds take as long as several chunk partials; with the fold in its own warps
// the drain warps go straight on to the next product and the tensor cores
// keep running.  The FP64 accumulator lives in a workspace buffer (tile by
// tile, 128 KB per CTA, L2-resident while the tile runs), which leaves TMEM
// for three partial buffers and the hand-off and shared memory for three
// 64 KB operand stages.  The result is bit-identical to the oracle in its
// product-outer order.
//
// Warp roles: warp 0 lane 0 issues TMA loads, warp 1 owns TMEM and lane 0
// issues the MMAs, warps 4-19 drain (four per TMEM lane quarter, 32 columns
// each), warps 20-23 fold (one per lane quarter, 128 columns each).
// setmaxnreg moves registers between the warpgroups.  Every wait is bounded
// and reports EMU_FLAG_TIMEOUT instead of hanging.
#include <cstdlib>
#include <cstring>

#include "launchers.cuh"
#include "prodsum_f64_common.cuh"

namespace emu {

namespace {

struct F64Cfg {
    // A stage holds SUB K-blocks of 64 (one 128-byte swizzle row each) of the
    // A slice and of the B slice.
    static constexpr int BN = 128, KB = 64, SUB = 2, STAGES = 3, NBUF = 3;
    static constexpr int KSPAN = KB * SUB;                          // K per stage
    static constexpr int A_SUB = kBM * KB * 2, B_SUB = BN * KB * 2; // one 64-wide K-block tile
    static constexpr int A_TILE = A_SUB * SUB, B_TILE = B_SUB * SUB;
    static constexpr int STAGE = A_TILE + B_TILE;
    static constexpr uint32_t SWZ = 2u, SBO = 1024u;              // 128-byte swizzle
    // one low-part mask byte per (row, drain column quarter) of the product
    // being handed off
    static constexpr int MASK_OFF = STAGES * STAGE;
    static constexpr int BAR_OFF = MASK_OFF + kBM * 4;
    // barriers: full/empty per stage, tfull/tempty per buffer, hand-off
    // full/empty, done; then the TMEM address slot
    static constexpr int NBARS = 2 * STAGES + 2 * NBUF + 2 + 1;
    static constexpr int SMEM = BAR_OFF + 256 + 1024;
    // warpgroup 0: TMA producer (warp 0), MMA issuer + TMEM owner (warp 1),
    // two idle warps; warpgroups 1-4: sixteen drain warps; warpgroup 5: fold
    static constexpr int FIRST_DRAIN = 4, DRAIN_WARPS = 16, FIRST_FOLD = 20, THREADS = 24 * 32;
    static constexpr int COLS = BN / (DRAIN_WARPS / 4);            // 32 columns per drain thread
    // Register split: the launch reserves 768 x 80 (six warps per SMSP);
    // 128 x 32 (control) + 512 x 96 (drain) + 128 x 64 (fold) = 61440 = 768 x 80.
    static constexpr int REG_CTRL = 32, REG_DRAIN = 96, REG_FOLD = 64, REG_LAUNCH = 80;
    static constexpr uint32_t HP_COL = NBUF * BN;                  // hand-off area: one FP32 word per column
};
static_assert(F64Cfg::HP_COL + F64Cfg::BN == 512, "TMEM budget: 3 partial buffers + hand-off area");
static_assert(kBM == 128 && F64Cfg::BN == 128, "f64_acc_bytes assumes 128 x 128 tiles");
static_assert(kKChunk % F64Cfg::KSPAN == 0, "a K-chunk is a whole number of stages");
static_assert(8 * F64Cfg::NBARS + 8 <= 256, "barrier area");
static_assert(F64Cfg::SMEM <= 232448, "shared memory per CTA");
static_assert(128 * F64Cfg::REG_CTRL + 512 * F64Cfg::REG_DRAIN + 128 * F64Cfg::REG_FOLD <=
                  F64Cfg::THREADS * F64Cfg::REG_LAUNCH,
              "setmaxnreg split exceeds the registers reserved at launch");

// TAIL: add the merged tail T (an M x N FP32 matrix) once after the last product.
template <int NPROD, bool ROWCOL, bool TAIL>
__global__ void __launch_bounds__(F64Cfg::THREADS, 1)
prodsum_f64_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   int M, int N, int K, const int32_t *__restrict__ vA, const int32_t *__restrict__ vB,
                   double *__restrict__ C, int64_t ldc, double *__restrict__ acc, uint32_t *flags,
                   const float *__restrict__ T, int64_t ldt, int wide_first, int wide_rows)
{
    using Cfg = F64Cfg;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *base_ptr = smem_raw + (base - raw);
    const uint32_t full0 = base + Cfg::BAR_OFF, empty0 = full0 + 8u * Cfg::STAGES;
    const uint32_t tfull0 = empty0 + 8u * Cfg::STAGES, tempty0 = tfull0 + 8u * Cfg::NBUF;
    const uint32_t hfull = tempty0 + 8u * Cfg::NBUF, hempty = hfull + 8u, done_bar = hempty + 8u;
    const uint32_t hmask = base + Cfg::MASK_OFF;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(base_ptr + Cfg::BAR_OFF + 8 * Cfg::NBARS);

    const int warp = threadIdx.x >> 5, lane = lane_id();
    const int tiles_m = (M + kBM - 1) / kBM, tiles_n = (N + Cfg::BN - 1) / Cfg::BN;
    int tm, tn;
    if (wide_first < 0) {
        tile_coords(blockIdx.x, tiles_m, tiles_n, tm, tn);
    } else {
        // the 128 x 128 parts of the (128 * wide_rows) x 256 tiles from raster
        // index wide_first on, which the wide kernel's last, partial wave
        // would have taken: two column halves per 128-row tile row
        const int per = 2 * wide_rows;
        int tw, tnw;
        tile_coords(wide_first + (int)(blockIdx.x / per), (tiles_m + wide_rows - 1) / wide_rows, (N + 255) / 256,
                    tw, tnw);
        const int sub = (int)(blockIdx.x % per);
        tm = tw * wide_rows + (sub >> 1);
        tn = 2 * tnw + (sub & 1);
        if (tm >= tiles_m || tn >= tiles_n) return;   // a part past the last row or column
    }
    const int m0 = tm * kBM, n0 = tn * Cfg::BN;
    const int nch = (K + kKChunk - 1) / kKChunk;

    if (threadIdx.x == 0) {
        for (int s = 0; s < Cfg::STAGES; ++s) { mbar_init(full0 + 8u * s, 1); mbar_init(empty0 + 8u * s, 1); }
        for (int b = 0; b < Cfg::NBUF; ++b) { mbar_init(tfull0 + 8u * b, 1); mbar_init(tempty0 + 8u * b, Cfg::DRAIN_WARPS); }
        mbar_init(hfull, Cfg::DRAIN_WARPS);
        mbar_init(hempty, 4);
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

    if (warp < Cfg::FIRST_DRAIN) {
      regs_dec<Cfg::REG_CTRL>();
      if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: for product, for chunk, for K-span of the chunk
        int L = 0, s = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int q = 0; q < NPROD && ok; ++q) {
            const int ia = kDiag[q][0], jb = kDiag[q][1];
            for (int c = 0; c < nch && ok; ++c) {
                const int kspans = min(kKChunk / Cfg::KSPAN, (K - c * kKChunk + Cfg::KSPAN - 1) / Cfg::KSPAN);
                for (int u = 0; u < kspans; ++u, ++L) {
                    if (!(ok = mbar_wait(empty0 + 8u * s, ph ^ 1u, flags))) break;
                    const uint32_t st = base + (uint32_t)(s * Cfg::STAGE), fb = full0 + 8u * s;
                    const int k0 = c * kKChunk + u * Cfg::KSPAN;
                    mbar_arrive_expect_tx(fb, Cfg::STAGE);
#pragma unroll
                    for (int h = 0; h < Cfg::SUB; ++h) {
                        tma_load_3d(st + h * Cfg::A_SUB, &tmA, fb, k0 + h * Cfg::KB, m0, ia);
                        tma_load_3d(st + Cfg::A_TILE + h * Cfg::B_SUB, &tmB, fb, k0 + h * Cfg::KB, n0, jb);
                    }
                    if (++s == Cfg::STAGES) { s = 0; ph ^= 1u; }
                }
            }
        }
        if (!ok) drain_inflight(full0, Cfg::STAGES, L, flags);
      } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: one chunk partial into buffer t % NBUF
        constexpr uint32_t idesc = make_idesc_bf16(kBM, Cfg::BN);
        int s = 0, b = 0;
        uint32_t ph = 0, tph = 0;
        bool ok = true;
        for (int t = 0; t < NPROD * nch && ok; ++t) {
            const int c = t % nch;
            const int kspans = min(kKChunk / Cfg::KSPAN, (K - c * kKChunk + Cfg::KSPAN - 1) / Cfg::KSPAN);
            if (!(ok = mbar_wait(tempty0 + 8u * b, tph ^ 1u, flags))) break;
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(b * Cfg::BN);
            for (int u = 0; u < kspans; ++u) {
                if (!(ok = mbar_wait(full0 + 8u * s, ph, flags))) break;
                tc_fence_after();
                const uint32_t st = base + (uint32_t)(s * Cfg::STAGE);
#pragma unroll
                for (int h = 0; h < Cfg::SUB; ++h) {
#pragma unroll
                    for (int kk = 0; kk < Cfg::KB / 16; ++kk) {
                        const uint64_t ad = make_sdesc(st + h * Cfg::A_SUB + kk * 32, Cfg::SBO, Cfg::SWZ);
                        const uint64_t bd = make_sdesc(st + Cfg::A_TILE + h * Cfg::B_SUB + kk * 32, Cfg::SBO, Cfg::SWZ);
                        mma_bf16(d, ad, bd, idesc, (u | h | kk) != 0);
                    }
                }
                mma_commit(empty0 + 8u * s);
                if (++s == Cfg::STAGES) { s = 0; ph ^= 1u; }
            }
            if (ok) mma_commit(tfull0 + 8u * b);
            if (++b == Cfg::NBUF) { b = 0; tph ^= 1u; }
        }
        mma_commit(done_bar);
        (void)mbar_wait(done_bar, 0, flags);
      }
    } else if (warp < Cfg::FIRST_FOLD) {
        regs_inc<Cfg::REG_DRAIN>();
        // ---------------- drain: exact per-product sum of the partials
        const int quarter = warp & 3;                                    // TMEM lanes 32*quarter ..
        const int cq = (warp - Cfg::FIRST_DRAIN) >> 2;                   // column quarter
        const int r = quarter * 32 + lane;                               // tile row of this thread
        const uint32_t tcol = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(cq * Cfg::COLS);
        const uint32_t thp = tcol + Cfg::HP_COL;                         // this thread's hand-off columns
        const int row = m0 + r;
        double *crow = C + (int64_t)row * ldc + n0 + cq * Cfg::COLS;
        const int lim = row < M ? N - (n0 + cq * Cfg::COLS) : 0;        // valid columns of this thread
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
            // this thread's row level of slice i (levels per row / column only)
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
                        float *lrow = reinterpret_cast<float *>(crow) + (q & 1);
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
                        // exactly into the low part; the partials are read again from
                        // TMEM (the buffer is not yet released).  With levels per row /
                        // column an element whose own unit allows it takes the carry
                        // above instead (its own split constant).
                        const bool was = (dirty >> (h / 16)) & 1u;
                        dirty |= 1u << (h / 16);
                        const float renorm = 0.5f * bound;        // lo is kept below 2^23 u
                        float *lrow = reinterpret_cast<float *>(crow) + (q & 1);
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
                        if (lane == 0) mbar_arrive(tempty0 + 8u * b);
                    }
                }
            }
            if (!ok) break;
            // hand the sums over once the fold warps have taken the previous product's
            if (q > 0) {
                ok = mbar_wait(hempty, (uint32_t)((q - 1) & 1), flags);
                __syncwarp();
                if (!ok) break;
            }
#pragma unroll
            for (int h = 0; h < Cfg::COLS; h += 16) {
                uint32_t w[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) w[j] = __float_as_uint(hi[h + j]);
                tmem_st16(thp + (uint32_t)h, w);
            }
            tmem_st_wait();
            asm volatile("st.shared.u8 [%0], %1;" ::"r"(hmask + (uint32_t)(r * 4 + cq)), "r"(dirty) : "memory");
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(hfull);
        }
    } else {
        regs_dec<Cfg::REG_FOLD>();
        // ---------------- fold: C <- fl64(C + (hi + lo)) per product, in product order
        const int quarter = warp & 3;
        const int r = quarter * 32 + lane;
        const uint32_t thp = tmem + ((uint32_t)(quarter * 32) << 16) + Cfg::HP_COL;
        const int row = m0 + r;
        double *crow = C + (int64_t)row * ldc + n0;
        // this tile's accumulator, column-major: a warp's 32 rows of a column are contiguous
        double *tacc = acc + ((size_t)tm * tiles_n + tn) * (size_t)(kBM * Cfg::BN) + r;
        const int lim = row < M ? N - n0 : 0;
        const bool vec = ((ldc & 1) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15u) == 0);
        // merged tail: one more addition after the last product
        const float *trow = TAIL ? T + (int64_t)(row < M ? row : 0) * ldt + n0 : nullptr;
        for (int q = 0; q < NPROD; ++q) {
            const bool ok = mbar_wait(hfull, (uint32_t)(q & 1), flags);
            __syncwarp();
            if (!ok) break;
            tc_fence_after();
            const bool first = (q == 0), last = (q == NPROD - 1);
            const float *lrow = reinterpret_cast<const float *>(crow) + (q & 1);
            double nxt[8];                                   // accumulator of the next 8 columns (prefetched)
            if (!first) {
#pragma unroll
                for (int j = 0; j < 8; ++j) nxt[j] = tacc[j * kBM];
            }
#pragma unroll 1
            for (int col = 0; col < Cfg::BN; col += 8) {
                double cur[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) cur[j] = nxt[j];
                if (!first && col + 8 < Cfg::BN) {
#pragma unroll
                    for (int j = 0; j < 8; ++j) nxt[j] = tacc[(col + 8 + j) * kBM];
                }
                uint32_t hv[8];
                tmem_ld8(thp + (uint32_t)col, hv);
                uint32_t mask;
                asm volatile("ld.shared.u8 %0, [%1];" : "=r"(mask) : "r"(hmask + (uint32_t)(r * 4 + (col >> 5))) : "memory");
                const bool dg = (mask >> ((col >> 4) & 1)) & 1u;   // 16-column group of these 8 columns
                tmem_ld_wait();
                // the common case (no low words, not the first product) is a
                // branch of its own: written as selects, the rare cases' FP64
                // additions would run for every element (GB300's FP64 pipe does
                // about one warp-wide add per 32 clocks per sub-partition)
                double out[8];
                if (!dg && !first) {
#pragma unroll
                    for (int j = 0; j < 8; ++j) out[j] = __dadd_rn(cur[j], widen_exact(__uint_as_float(hv[j])));
                } else {
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        double sq = widen_exact(__uint_as_float(hv[j]));
                        if (dg && col + j < lim) sq = __dadd_rn(sq, widen_exact(lrow[2 * (col + j)]));   // exact
                        out[j] = first ? sq : __dadd_rn(cur[j], sq);
                    }
                }
                if (TAIL && last) {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        if (col + j < lim) out[j] = __dadd_rn(out[j], widen_exact(trow[col + j]));
                }
                if (!last) {
#pragma unroll
                    for (int j = 0; j < 8; ++j) tacc[(col + j) * kBM] = out[j];
                } else if (vec && lim >= col + 8) {
#pragma unroll
                    for (int j = 0; j < 8; j += 2)
                        *reinterpret_cast<double2 *>(crow + col + j) = make_double2(out[j], out[j + 1]);
                } else {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        if (col + j < lim) crow[col + j] = out[j];
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(hempty);
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

// Per-SM rate of the 128 x 128 kernel relative to the 128 x 256 one (measured
// at 8192^3 with 21 products: 1128 against 1437 TFLOP/s executed, with 27 and
// 14 waves of CTAs).
constexpr double kF64RateNarrow = 0.76;

template <int NPROD, bool ROWCOL, bool TAIL = false>
cudaError_t run_f64(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp, int64_t ldcomp,
                    const int32_t *vA, const int32_t *vB, double *C, int64_t ldc, double *acc, uint32_t *flags,
                    cudaStream_t st, int64_t a_plane, const float *T, int64_t ldt, int wide_first, int wide_rows,
                    int64_t ctas)
{
    using Cfg = F64Cfg;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, 6, ldcomp, Cfg::KB, kBM, a_plane) || !make_plane_map(&tb, Bp, K, N, 6, ldcomp, Cfg::KB, Cfg::BN))
        return cudaErrorInvalidValue;
    auto kern = prodsum_f64_kernel<NPROD, ROWCOL, TAIL>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM);
    if (e != cudaSuccess) return e;
    const int64_t tiles = wide_first < 0 ? ((M + kBM - 1) / kBM) * ((N + Cfg::BN - 1) / Cfg::BN) : ctas;
    kern<<<(unsigned)tiles, Cfg::THREADS, Cfg::SMEM, st>>>(ta, tb, (int)M, (int)N, (int)K, vA, vB, C, ldc, acc, flags,
                                                           T, ldt, wide_first, wide_rows);
    return cudaGetLastError();
}

}  // namespace

static cudaError_t launch_prodsum_f64_narrow(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                               int64_t ldcomp, const int32_t *vA, const int32_t *vB, int nprod, double *C,
                               int64_t ldc, double *acc, uint32_t *flags, cudaStream_t st, int64_t a_plane,
                               bool rowcol, const float *T, int64_t ldt, int wide_first = -1, int wide_rows = 1,
                               int64_t ctas = 0)
{
#define EMU_F64N(NP, RC, TL) \
    run_f64<NP, RC, TL>(M, N, K, Ap, Bp, ldcomp, vA, vB, C, ldc, acc, flags, st, a_plane, T, ldt, wide_first, \
                        wide_rows, ctas)
    if (T) {                                          // merged tail: whole-matrix levels only
        if (rowcol) return cudaErrorInvalidValue;
        switch (nprod) {
        case 6: return EMU_F64N(6, false, true);
        case 10: return EMU_F64N(10, false, true);
        case 15: return EMU_F64N(15, false, true);
        default: return cudaErrorInvalidValue;
        }
    }
    switch (nprod) {
    case 6: return rowcol ? EMU_F64N(6, true, false) : EMU_F64N(6, false, false);
    case 10: return rowcol ? EMU_F64N(10, true, false) : EMU_F64N(10, false, false);
    case 15: return rowcol ? EMU_F64N(15, true, false) : EMU_F64N(15, false, false);
    case 21: return rowcol ? EMU_F64N(21, true, false) : EMU_F64N(21, false, false);
    default: return cudaErrorInvalidValue;
    }
#undef EMU_F64N
}

// Tile shape of the FP64 product-sum.  Every shape forms the same exact
// per-product sums and folds them in the same order, so C does not depend on
// the choice.
// - 128 x 256 tiles (prodsum_f64w.cu) take in 0.75x the operand bytes per FLOP
//   of 128 x 128 and are faster per SM, but give half as many CTAs; the width
//   maximises (SMs kept busy over the waves) x (relative per-SM rate), as for
//   the FP32 product-sum.
// - With two or more 128-row tile rows, the 256-column tiles run as 256 x 256
//   tiles on CTA pairs (the same kernel with cta_group::2 MMAs): each SM then
//   stages 8 KB of operands per 2^20 FLOP instead of 12 KB.
// - When those tiles leave the last wave partly empty, the full waves run as
//   such and the narrow kernel, launched after them, takes the remaining
//   tiles as 128 x 128 parts, if that is estimated faster (a part takes
//   0.5 / kF64RateNarrow of a 128 x 256 tile's time).  The two kernels run one
//   after the other, so the accumulator tiles they index differently never
//   overlap in time.
// EMU_F64_TILE=128x128 / 128x256 / 256x256 forces one shape for every result
// (and no mixed last wave).
static int f64_tile_forced()
{
    static const int forced = [] {
        const char *e = std::getenv("EMU_F64_TILE");
        if (!e) return 0;
        if (std::strcmp(e, "128x128") == 0) return 1;
        if (std::strcmp(e, "128x256") == 0) return 2;
        if (std::strcmp(e, "256x256") == 0) return 3;
        return 0;
    }();
    return forced;
}

static int device_sms()
{
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 2)
        sms = 152;
    return sms;
}

F64Plan f64_plan(int64_t M, int64_t N)
{
    F64Plan p;
    if (M < 1 || N < 1) return p;
    const int forced = f64_tile_forced();
    const int sms = device_sms();
    const int64_t tiles_m = (M + kBM - 1) / kBM;
    int cols = forced == 1 ? 128 : forced >= 2 ? 256 : 0;
    if (cols == 0) {
        const int widths[2] = {256, 128};
        const double rate[2] = {1.0, kF64RateNarrow};
        double best = -1.0;
        for (int i = 0; i < 2; ++i) {
            const int64_t tiles = tiles_m * ((N + widths[i] - 1) / widths[i]);
            const int64_t waves = (tiles + sms - 1) / sms;
            const double score = rate[i] * (double)tiles / (double)(waves * sms);
            if (score > best * 1.02) { best = score; cols = widths[i]; }   // prefer the wider tile on near ties
        }
    }
    p.cols = cols;
    p.rows = kBM;
    p.launches = 1;
    if (cols == 128) {
        p.tiles = tiles_m * ((N + 127) / 128);
        return p;
    }
    const bool pair = forced == 3 || (forced == 0 && tiles_m >= 2);
    const int rows_per = pair ? 2 : 1, slots = pair ? sms / 2 : sms;
    p.rows = kBM * rows_per;
    const int64_t tiles = ((tiles_m + rows_per - 1) / rows_per) * ((N + 255) / 256);
    const int64_t full = (tiles / slots) * slots, rem = tiles - full;
    const double t_wide = (double)((tiles + slots - 1) / slots);
    const double t_mixed = (double)(full / slots) + (0.5 / kF64RateNarrow) * (double)((2 * rows_per * rem + sms - 1) / sms);
    p.tiles = tiles;
    if (forced == 0 && full > 0 && rem > 0 && t_mixed < 0.97 * t_wide) {
        p.tiles = full;
        p.rest = 2 * rows_per * rem;
        p.launches = 2;
    }
    return p;
}

int f64_tile_columns(int64_t M, int64_t N)
{
    return f64_plan(M, N).cols;
}

cudaError_t launch_prodsum_f64(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                               int64_t ldcomp, const int32_t *vA, const int32_t *vB, int nprod, double *C,
                               int64_t ldc, double *acc, uint32_t *flags, cudaStream_t st, int64_t a_plane,
                               bool rowcol, const float *T, int64_t ldt)
{
    const F64Plan p = f64_plan(M, N);
    if (p.cols == 128)
        return launch_prodsum_f64_narrow(M, N, K, Ap, Bp, ldcomp, vA, vB, nprod, C, ldc, acc, flags, st, a_plane,
                                         rowcol, T, ldt);
    const bool pair = p.rows == 2 * kBM;
    cudaError_t e = launch_prodsum_f64_wide(M, N, K, Ap, Bp, ldcomp, vA, vB, nprod, C, ldc, acc, flags, st, a_plane,
                                            rowcol, T, ldt, p.tiles, pair);
    if (e != cudaSuccess || p.rest == 0) return e;
    return launch_prodsum_f64_narrow(M, N, K, Ap, Bp, ldcomp, vA, vB, nprod, C, ldc, acc, flags, st, a_plane, rowcol,
                                     T, ldt, (int)p.tiles, pair ? 2 : 1, p.rest);
}

}  // namespace emu
