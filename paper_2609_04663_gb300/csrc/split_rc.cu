// FP64 six-slice split with level exponents per row of A / per column of B
// (the vector scaling of Eq. (ozakiscaled)): a literal level-0 pass, a
// speculative pass per vector, and one cooperative launch that verifies
// every vector and redoes the literal levels only for the vectors whose
// speculation failed.
#include "split_common.cuh"

namespace emu {

namespace {

// ------------------------------ FP64 split with levels per row / per column
// The vector scaling of Eq. (ozakiscaled): each plane row (an input row, or
// an input column when the planes are transposed) gets its own six levels
// v^(r) = ceil(log2 max |X^(r)|) over that vector.  Literal form: level L's
// maxima come from a pass that recomputes levels 0 .. L-1 from x with the
// vector's final levels; a one-thread-per-vector kernel turns them into
// v[L][vector]; the tile kernel (MODE 3) then writes all six planes.

// Max |X^(L)| per vector.  Not transposed: one warp per row, lanes striding
// along it.  Transposed: one thread per column over a range of rows, the
// block's columns contiguous, maxima merged with atomicMax.  Level 0 also
// checks the input domain of Eq. (bf16rangefp64).
// Maxima of |X^(L)| per vector.  Transposed: work item = (block of 256
// columns, range of rows_per_block rows), column_blocks of them per row range;
// by rows: one warp per row.  Items are spread over nblk blocks.
template <bool TRANSPOSE>
__device__ __forceinline__ void
rc_max_pass(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx, int L,
            const int32_t *__restrict__ vrc, unsigned long long *maxbits, int64_t rows_per_block, WsHeader *ws,
            const int32_t *__restrict__ ff, int64_t bid, int64_t nblk)
{
    constexpr unsigned long long kLo = 0x3810000000000000ull, kHi = 0x47EFE00000000000ull;
    constexpr unsigned long long kInf = 0x7FF0000000000000ull;
    const int64_t nvec = TRANSPOSE ? cols : rows;
    uint32_t flagbits = 0;
    auto take = [&](double R, const int (&v)[6], unsigned long long &m) {
        bool bad = false;
        for (int l = 0; l < L; ++l) (void)f64_level_int(R, v[l], bad);
        const unsigned long long ab = (unsigned long long)__double_as_longlong(R) & 0x7FFFFFFFFFFFFFFFull;
        if (L == 0) {
            if (ab >= kInf) flagbits |= EMU_FLAG_NONFINITE;
            else if (ab != 0 && (ab < kLo || ab > kHi)) flagbits |= EMU_FLAG_RANGE;
            if (ab <= kInf) m = ab > m ? ab : m;                      // NaN never wins
        } else {
            m = ab > m ? ab : m;
        }
    };
    int v[6] = {0, 0, 0, 0, 0, 0};
    if (!TRANSPOSE) {
        const int64_t nwarps = nblk * (kThreads / 32);
        for (int64_t i = bid * (kThreads / 32) + (threadIdx.x >> 5); i < rows; i += nwarps) {
            if (ff && ff[i] >= L) continue;
            for (int l = 0; l < L; ++l) v[l] = vrc[l * nvec + i];
            unsigned long long m = 0;
            for (int64_t j = lane_id(); j < cols; j += 32) take(X[i * ldx + j], v, m);
            m = warp_max(m);
            if (lane_id() == 0) maxbits[i] = m;
        }
    } else {
        const int64_t cblocks = (cols + kThreads - 1) / kThreads;
        const int64_t ranges = (rows + rows_per_block - 1) / rows_per_block;
        for (int64_t it = bid; it < cblocks * ranges; it += nblk) {
            const int64_t j = (it % cblocks) * kThreads + threadIdx.x;
            const int64_t i0 = (it / cblocks) * rows_per_block;
            const int64_t i1 = i0 + rows_per_block < rows ? i0 + rows_per_block : rows;
            if (j < cols && !(ff && ff[j] >= L)) {
                for (int l = 0; l < L; ++l) v[l] = vrc[l * nvec + j];
                unsigned long long m = 0;
                for (int64_t i = i0; i < i1; ++i) take(X[i * ldx + j], v, m);
                if (m) atomicMax(&maxbits[j], m);
            }
        }
    }
    flagbits = __reduce_or_sync(0xFFFFFFFFu, flagbits);
    if (flagbits && lane_id() == 0) atomicOr(&ws->flags, flagbits);
}

// The pass as a kernel: ff (fix passes only): levels <= ff[vector] are final;
// nothing to do for vectors with ff >= L, and nothing at all unless some
// vector failed.
template <bool TRANSPOSE>
__global__ void __launch_bounds__(kThreads)
rc_max_kernel(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx, int L,
              const int32_t *__restrict__ vrc, unsigned long long *maxbits, int64_t rows_per_block, WsHeader *ws,
              const int32_t *__restrict__ ff)
{
    if (ff && ws->fix_any == 0) return;
    rc_max_pass<TRANSPOSE>(X, rows, cols, ldx, L, vrc, maxbits, rows_per_block, ws, ff, blockIdx.x, gridDim.x);
}

// v[L][vector] from the maxima of level L; a vector whose previous level was
// already zero stays zero (Section 4.3's early stop).  Clears the maxima.
__device__ __forceinline__ void rc_levels_pass(int L, unsigned long long *maxbits, int32_t *vrc, int64_t nvec,
                                               const int32_t *ff, int64_t tid, int64_t nthreads)
{
    for (int64_t i = tid; i < nvec; i += nthreads) {
        if (ff && ff[i] >= L) continue;
        const unsigned long long m = maxbits[i];
        int v = m ? ceil_log2_bits(m) : kZeroLevel;
        if (L > 0 && vrc[(L - 1) * nvec + i] == kZeroLevel) v = kZeroLevel;
        vrc[L * nvec + i] = v;
        maxbits[i] = 0;
    }
}

__global__ void rc_levels_kernel(int L, unsigned long long *maxbits, int32_t *vrc, int64_t nvec, const int32_t *ff,
                                 const WsHeader *ws)
{
    if (ff && ws->fix_any == 0) return;
    rc_levels_pass(L, maxbits, vrc, nvec, ff, (int64_t)blockIdx.x * blockDim.x + threadIdx.x,
                   (int64_t)gridDim.x * blockDim.x);
}

// Speculative pass with per-vector levels: each element is split with its
// vector's v0 (level 0 is literal) under the assumption v^(r) = v0 - 8r, as
// in the whole-matrix speculative pass; the magnitudes |X^(r)| before levels
// 1 .. 5 are reduced per vector into vmax[5][vectors] (32-bit: levels 1 and
// 2 in units of 2^(F + 20) with a sticky last bit, levels 3 .. 5 exact in
// units of 2^F, F = v0 - 50).
__device__ __forceinline__ uint32_t jam20(unsigned long long m)
{
    return (uint32_t)(m >> 20) | ((m & 0xFFFFFull) != 0 ? 1u : 0u);
}

__device__ __forceinline__ void spec_element_mags(double x, int v0, const float (&P)[6], uint32_t (&s)[6],
                                                  uint32_t &badmask, uint32_t (&mag)[5])
{
    SpecState st;
    spec_element(x, v0, v0 >= -78, P, s, st);
    badmask |= st.badmask;
    mag[0] = jam20(st.m1);
    mag[1] = jam20(st.m2);
    mag[2] = st.m[0];
    mag[3] = st.m[1];
    mag[4] = st.m[2];
}

// Row-major planes, levels per row: thread = 4 consecutive entries of a row.
__global__ void __launch_bounds__(kThreads)
rc_spec_rows_kernel(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                    uint16_t *__restrict__ comps, int64_t ldcomp, int64_t plane, const int32_t *__restrict__ vrc,
                    uint32_t *vmax, WsHeader *ws, int slot)
{
    const bool vin = ((ldx & 1) == 0) && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0);
    const bool vout = ((ldcomp & 3) == 0) && ((plane & 3) == 0) && ((reinterpret_cast<uintptr_t>(comps) & 7u) == 0);
    const int64_t j0 = ((int64_t)blockIdx.x * kThreads + threadIdx.x) * 4;
    const bool full = j0 + 4 <= cols;
    uint32_t badmask = 0;
    for (int64_t i = blockIdx.y; i < rows; i += gridDim.y) {
        const int v0 = vrc[i];
        uint32_t mx[5] = {0, 0, 0, 0, 0};
        if (j0 < cols) {
            const double *src = X + i * ldx + j0;
            double x[4];
            if (vin && full) {
                const double2 a = reinterpret_cast<const double2 *>(src)[0], c = reinterpret_cast<const double2 *>(src)[1];
                x[0] = a.x; x[1] = a.y; x[2] = c.x; x[3] = c.y;
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) x[e] = (j0 + e < cols) ? src[e] : 0.0;
            }
            float P[6] = {};
            if (v0 >= -78) spec_units(v0 - 50, P);
            uint32_t w[6][2];
#pragma unroll
            for (int e = 0; e < 4; e += 2) {
                uint32_t sa[6], sb[6], ma[5], mb[5];
                spec_element_mags(x[e], v0, P, sa, badmask, ma);
                spec_element_mags(x[e + 1], v0, P, sb, badmask, mb);
#pragma unroll
                for (int r = 0; r < 5; ++r) {
                    const uint32_t mm = ma[r] > mb[r] ? ma[r] : mb[r];
                    mx[r] = mm > mx[r] ? mm : mx[r];
                }
#pragma unroll
                for (int r = 0; r < 6; ++r) w[r][e >> 1] = pack2(sa[r], sb[r]);
            }
            uint16_t *dst = comps + i * ldcomp + j0;
#pragma unroll
            for (int r = 0; r < 6; ++r) {
                if (vout && full) {
                    *reinterpret_cast<uint2 *>(dst + r * plane) = make_uint2(w[r][0], w[r][1]);
                } else {
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (j0 + e < cols) dst[r * plane + e] = (uint16_t)(w[r][e >> 1] >> (16 * (e & 1)));
                }
            }
        }
#pragma unroll
        for (int r = 0; r < 5; ++r) {
            const uint32_t m = __reduce_max_sync(0xFFFFFFFFu, mx[r]);
            if (lane_id() == 0 && m) atomicMax(&vmax[r * rows + i], m);
        }
    }
    badmask = __reduce_or_sync(0xFFFFFFFFu, badmask);
    if (badmask && lane_id() == 0) atomicOr(&ws->slice_bad[slot], badmask);
}

// Transposed planes, levels per column: the 64 x 64 tile of the whole-matrix
// transposed pass; each warp reduces its 8 columns' magnitudes over its 64 rows.
__global__ void __launch_bounds__(kThreads)
rc_spec_transpose_kernel(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                         uint16_t *__restrict__ comps, int64_t ldcomp, int64_t plane,
                         const int32_t *__restrict__ vrc, uint32_t *vmax, WsHeader *ws, int slot)
{
    extern __shared__ __align__(16) uint32_t smw[];                  // [6][kTile][kTile / 2]
    const bool vin = ((ldx & 1) == 0) && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0);
    const bool vout = ((ldcomp & 7) == 0) && ((plane & 7) == 0) && ((reinterpret_cast<uintptr_t>(comps) & 15u) == 0);
    const int q = threadIdx.x >> 5, p = lane_id();
    const int64_t tiles_r = (rows + kTile - 1) / kTile, tiles_c = (cols + kTile - 1) / kTile;
    uint32_t badmask = 0;
    for (int64_t t = blockIdx.x; t < tiles_r * tiles_c; t += gridDim.x) {
        const int64_t r0 = (t / tiles_c) * kTile, c0 = (t % tiles_c) * kTile;
        const int64_t gj = c0 + 8 * q;
        // two adjacent columns per step (one 16-byte load per row), so that
        // the element body appears four times in the loop, not sixteen
#pragma unroll 1
        for (int k = 0; k < 8; k += 2) {
            double x[2][2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int64_t gi = r0 + 2 * p + h;
                const double *src = X + gi * ldx + gj + k;
                if (gi < rows && vin && gj + 8 <= cols) {
                    const double2 a = *reinterpret_cast<const double2 *>(src);
                    x[h][0] = a.x; x[h][1] = a.y;
                } else {
#pragma unroll
                    for (int e = 0; e < 2; ++e) x[h][e] = (gi < rows && gj + k + e < cols) ? src[e] : 0.0;
                }
            }
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int64_t col = gj + k + e;
                const int v0 = col < cols ? vrc[col] : kZeroLevel;
                float P[6] = {};
                if (v0 >= -78) spec_units(v0 - 50, P);
                uint32_t s0[6], s1[6], m0[5], m1[5];
                spec_element_mags(x[0][e], v0, P, s0, badmask, m0);
                spec_element_mags(x[1][e], v0, P, s1, badmask, m1);
#pragma unroll
                for (int r = 0; r < 6; ++r) smw[(r * kTile + 8 * q + k + e) * (kTile / 2) + p] = pack2(s0[r], s1[r]);
#pragma unroll
                for (int r = 0; r < 5; ++r) {
                    const uint32_t m = __reduce_max_sync(0xFFFFFFFFu, m0[r] > m1[r] ? m0[r] : m1[r]);
                    if (p == 0 && m && col < cols) atomicMax(&vmax[r * cols + col], m);
                }
            }
        }
        __syncthreads();
#pragma unroll 4
        for (int it = 0; it < 6 * kTile * 8 / kThreads; ++it) {
            const int c = threadIdx.x + it * kThreads;
            const int r = c >> 9, orow = (c >> 3) & 63, ch = c & 7;
            const int64_t go = c0 + orow, gk = r0 + 8 * ch;
            if (go < cols && gk < rows) {
                const uint4 v = *reinterpret_cast<const uint4 *>(&smw[(r * kTile + orow) * (kTile / 2) + 4 * ch]);
                uint16_t *dst = comps + r * plane + go * ldcomp + gk;
                if (vout && gk + 8 <= rows) {
                    *reinterpret_cast<uint4 *>(dst) = v;
                } else {
                    const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        if (gk + e < rows) dst[e] = (uint16_t)(wv[e >> 1] >> (16 * (e & 1)));
                }
            }
        }
        __syncthreads();
    }
    badmask = __reduce_or_sync(0xFFFFFFFFu, badmask);
    if (badmask && lane_id() == 0) atomicOr(&ws->slice_bad[slot], badmask);
}

__device__ __forceinline__ int ceil_log2_u32(uint32_t m) { return m <= 1u ? 0 : 32 - __clz(m - 1u); }

// One thread per vector: checks its speculative levels in order.  A level
// that matches v0 - 8r is final (the 32-bit maxima decide matches exactly);
// at the first mismatch r the literal passes redo levels r .. 5 (ff = r - 1:
// levels up to ff are final).  A residual that became zero ends the vector
// (literal as long as the levels before were right).  A slice outside the
// BF16 range (or a non-finite input) anywhere in the operand sends every
// vector to the literal passes, which flag such slices as Eq. (fp64split)
// computes them.
__device__ __forceinline__ void rc_verify_pass(const uint32_t *vmax, int32_t *vrc, int32_t *ff, int64_t nvec,
                                               WsHeader *ws, int slot, int64_t tid, int64_t nthreads)
{
    const bool fix_all = (ws->slice_bad[slot] & 0x3Fu) != 0;
    for (int64_t i = tid; i < nvec; i += nthreads) {
        const int v0 = vrc[i];
        int f = 6;
        if (v0 == kZeroLevel) {
            for (int r = 1; r < 6; ++r) vrc[r * nvec + i] = kZeroLevel;
        } else if (fix_all) {
            f = 0;
        } else {
            const int F = v0 - 50;
            bool zero = false;
            for (int r = 1; r < 6; ++r) {
                if (zero) { vrc[r * nvec + i] = kZeroLevel; continue; }
                const uint32_t m = vmax[(r - 1) * nvec + i];
                if (m == 0) { vrc[r * nvec + i] = kZeroLevel; zero = true; continue; }
                const int vr = ceil_log2_u32(m) + F + (r <= 2 ? 20 : 0);
                if (vr != v0 - 8 * r) { f = r - 1; break; }
                vrc[r * nvec + i] = vr;
            }
        }
        ff[i] = f;
        if (f < 6) atomicOr(&ws->fix_any, 1u);
    }
}

// Everything after the per-vector speculative pass, in one cooperative
// launch: every vector is verified; after a grid barrier each block reads
// whether any vector failed (the same answer everywhere) and, if none did --
// the usual case -- the launch ends.  Otherwise levels 1 .. 5 are redone
// literally for the failed vectors (maxima, then levels, the grid
// synchronised between the steps) and their planes rewritten.
template <bool TRANSPOSE>
__global__ void __launch_bounds__(kThreads)
rc_fix_kernel(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx, uint16_t *__restrict__ comps,
              int64_t ldcomp, int64_t plane, const uint32_t *vmax, int32_t *vrc, int32_t *ff,
              unsigned long long *maxbits, int64_t rows_per_block, WsHeader *ws, int slot)
{
    extern __shared__ __align__(16) uint16_t smdyn[];
    const int64_t nvec = TRANSPOSE ? cols : rows;
    const int64_t tid = (int64_t)blockIdx.x * kThreads + threadIdx.x, nthreads = (int64_t)gridDim.x * kThreads;
    rc_verify_pass(vmax, vrc, ff, nvec, ws, slot, tid, nthreads);
    grid_sync(ws, slot);
    if (*reinterpret_cast<volatile uint32_t *>(&ws->fix_any) == 0) return;
    for (int L = 1; L < 6; ++L) {
        rc_max_pass<TRANSPOSE>(X, rows, cols, ldx, L, vrc, maxbits, rows_per_block, ws, ff, blockIdx.x, gridDim.x);
        grid_sync(ws, slot);
        rc_levels_pass(L, maxbits, vrc, nvec, ff, tid, nthreads);
        grid_sync(ws, slot);
    }
    split_tile_pass<double, 3, TRANSPOSE>(X, rows, cols, ldx, comps, ldcomp, plane, ws, slot, vrc, ff, blockIdx.x,
                                          gridDim.x, smdyn);
}

}  // namespace

namespace {

// Cooperative launch of rc_fix_kernel with as many blocks as fit at once
// (at most 152 x 8), found once per device.
template <bool TRANSPOSE>
cudaError_t launch_rc_fix(const double *X, int64_t rows, int64_t cols, int64_t ldx, uint16_t *comps, int64_t ldcomp,
                          int64_t plane, const uint32_t *vmax, int32_t *vrc, int32_t *ff, unsigned long long *maxbits,
                          int64_t rows_per_block, WsHeader *ws, int slot, cudaStream_t st)
{
    constexpr int kMaxDev = 64;
    static int grid_of[kMaxDev] = {};
    const size_t sm = smem_bytes(6);
    auto kern = rc_fix_kernel<TRANSPOSE>;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDev) return cudaErrorInvalidDevice;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    int grid = grid_of[dev];
    if (grid == 0) {
        int sms = 0, per = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, kern, kThreads, sm);
        if (e != cudaSuccess) return e;
        grid = per * sms;
        if (grid > 152 * 8) grid = 152 * 8;
        if (grid < 1) return cudaErrorInvalidConfiguration;
        grid_of[dev] = grid;
    }
    void *args[] = {(void *)&X,    (void *)&rows,  (void *)&cols,    (void *)&ldx,           (void *)&comps,
                    (void *)&ldcomp, (void *)&plane, (void *)&vmax, (void *)&vrc, (void *)&ff,
                    (void *)&maxbits, (void *)&rows_per_block, (void *)&ws, (void *)&slot};
    return cudaLaunchCooperativeKernel((const void *)kern, dim3((unsigned)grid), dim3(kThreads), args, sm, st);
}

}  // namespace

cudaError_t launch_split_f64_rc(const double *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose,
                                uint16_t *comps, int64_t ldcomp, int32_t *v_out, void *scratch, WsHeader *ws,
                                int slot, cudaStream_t st)
{
    const int64_t nvec = transpose ? cols : rows;
    const int64_t plane = nvec * ldcomp;
    // scratch: literal maxima [nvec] u64, speculative maxima [5][nvec] u32, ff [nvec] i32
    auto *maxbits = static_cast<unsigned long long *>(scratch);
    auto *vmax = reinterpret_cast<uint32_t *>(maxbits + nvec);
    int32_t *ff = reinterpret_cast<int32_t *>(vmax + 5 * nvec);
    if (nvec == 0) return cudaSuccess;
    const int lgrid = grid_for((nvec + 255) / 256, 152 * 4);
    cudaError_t e = cudaMemsetAsync(scratch, 0, (size_t)nvec * (8 + 20), st);
    if (rows == 0 || cols == 0) {
        // an empty vector has no nonzero entry: every level is zero
        for (int L = 0; L < 6 && e == cudaSuccess; ++L) {
            rc_levels_kernel<<<lgrid, 256, 0, st>>>(L, maxbits, v_out, nvec, nullptr, ws);
            e = cudaGetLastError();
        }
        return e;
    }
    if (e == cudaSuccess && transpose)
        e = cudaFuncSetAttribute(rc_spec_transpose_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSpecTransposeSmem);
    if (e != cudaSuccess) return e;
    // transposed max passes: work items of 256 columns by rpb rows, one block each
    const int64_t cbx = (cols + kThreads - 1) / kThreads;
    int64_t cby = (152 * 8 + cbx - 1) / cbx;
    cby = cby < rows ? cby : rows;
    cby = cby < 65535 ? cby : 65535;
    const int64_t rpb = (rows + cby - 1) / cby;
    auto max_pass = [&](int L, const int32_t *gate) {
        if (transpose)
            rc_max_kernel<true><<<(unsigned)(cbx * cby), kThreads, 0, st>>>(X, rows, cols, ldx, L, v_out, maxbits, rpb,
                                                                            ws, gate);
        else
            rc_max_kernel<false><<<grid_for((rows + 7) / 8, 152 * 8), kThreads, 0, st>>>(X, rows, cols, ldx, L, v_out,
                                                                                        maxbits, 0, ws, gate);
        rc_levels_kernel<<<lgrid, 256, 0, st>>>(L, maxbits, v_out, nvec, gate, ws);
    };
    // level 0 literally, then all levels speculatively, verified per vector
    max_pass(0, nullptr);
    const int64_t tiles = ((rows + kTile - 1) / kTile) * ((cols + kTile - 1) / kTile);
    const int gt = grid_for(tiles, 152 * 8);
    if (transpose) {
        rc_spec_transpose_kernel<<<gt, kThreads, kSpecTransposeSmem, st>>>(X, rows, cols, ldx, comps, ldcomp, plane,
                                                                          v_out, vmax, ws, slot);
    } else {
        const int64_t bx = (cols + 4 * kThreads - 1) / (4 * kThreads);
        const int64_t want = (152 * 8 + bx - 1) / bx;
        const int64_t by = rows < want ? rows : (want < 65535 ? want : 65535);
        rc_spec_rows_kernel<<<dim3((unsigned)bx, (unsigned)by), kThreads, 0, st>>>(X, rows, cols, ldx, comps, ldcomp,
                                                                                  plane, v_out, vmax, ws, slot);
    }
    // verification and the literal passes for the vectors whose speculation
    // failed, in one cooperative launch
    e = cudaGetLastError();
    if (e == cudaSuccess)
        e = transpose ? launch_rc_fix<true>(X, rows, cols, ldx, comps, ldcomp, plane, vmax, v_out, ff, maxbits, rpb, ws,
                                            slot, st)
                      : launch_rc_fix<false>(X, rows, cols, ldx, comps, ldcomp, plane, vmax, v_out, ff, maxbits, rpb,
                                             ws, slot, st);
    return e;
}


}  // namespace emu
