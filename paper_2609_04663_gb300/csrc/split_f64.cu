// FP64 fixed six-slice simplified Ozaki split, Eq. (fp64split), with one set
// of level exponents per matrix, writing BF16 component planes row-major or
// transposed (K-major for the B operand).
//
// The FP64 split reads a 64 x 64 tile of X with coalesced vector loads,
// splits it in registers, stages it in shared memory and writes 16-byte
// chunks of whole plane rows, so transposed B planes are written as
// coalesced as row-major A planes.
//
// FP64 level exponents need a whole-matrix max per level (v^(r) of
// Eq. (fp64split)), i.e. six dependent grid-wide reductions.  The split does
// them speculatively in one pass: after the exact max of level 0, the fused
// pass assumes v^(r) = v^(0) - 8r (a residual always shrinks by at least 2^-8
// per level, and on full-size dense data by exactly that), writes the planes
// (all six, or only the d a product-sum of d diagonals reads) and records the
// true per-level maxima.  One cooperative launch then checks the assumption
// level by level and, only if it fails, recomputes the remaining levels
// literally.  The result is identical to the literal definition in every
// case.
#include "split_common.cuh"

namespace emu {

namespace {


// Row-major planes: thread = 4 consecutive entries of a row (two 16-byte
// loads, one 8-byte store per plane), rows advancing by the grid's y size.
// Block (bx, by) of a grid with gy rows of blocks; red: 5 * kThreads / 32
// words of shared memory.
template <int NLEV>
__device__ __forceinline__ void f64_spec_rows_body(const double *__restrict__ X, int64_t rows, int64_t cols,
                                                   int64_t ldx, uint16_t *__restrict__ comps, int64_t ldcomp,
                                                   int64_t plane, WsHeader *ws, int slot, int64_t bx, int64_t by,
                                                   int64_t gy, unsigned long long *red)
{
    const int v0 = spec_v0(ws, slot);
    const bool fast = v0 >= -78;
    float P[6] = {};
    if (fast) spec_units(v0 - 50, P);
    const bool vin = ((ldx & 1) == 0) && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0);
    const bool vout = ((ldcomp & 3) == 0) && ((plane & 3) == 0) && ((reinterpret_cast<uintptr_t>(comps) & 7u) == 0);
    const int64_t j0 = (bx * kThreads + threadIdx.x) * 4;
    SpecState st;
    if (j0 < cols) {
        const bool full = j0 + 4 <= cols;
        for (int64_t i = by; i < rows; i += gy) {
            const double *src = X + i * ldx + j0;
            double x[4];
            if (vin && full) {
                const double2 a = reinterpret_cast<const double2 *>(src)[0], c = reinterpret_cast<const double2 *>(src)[1];
                x[0] = a.x; x[1] = a.y; x[2] = c.x; x[3] = c.y;
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) x[e] = (j0 + e < cols) ? src[e] : 0.0;
            }
            uint32_t w[NLEV][2];
#pragma unroll
            for (int e = 0; e < 4; e += 2) {
                uint32_t sa[6], sb[6];
                spec_element<NLEV>(x[e], v0, fast, P, sa, st);
                spec_element<NLEV>(x[e + 1], v0, fast, P, sb, st);
#pragma unroll
                for (int r = 0; r < NLEV; ++r) w[r][e >> 1] = pack2(sa[r], sb[r]);
            }
            uint16_t *dst = comps + i * ldcomp + j0;
#pragma unroll
            for (int r = 0; r < NLEV; ++r) {
                if (vout && full) {
                    *reinterpret_cast<uint2 *>(dst + r * plane) = make_uint2(w[r][0], w[r][1]);
                } else {
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (j0 + e < cols) dst[r * plane + e] = (uint16_t)(w[r][e >> 1] >> (16 * (e & 1)));
                }
            }
        }
    }
    spec_publish(st, v0, ws, slot, red);
}

template <int NLEV>
__global__ void __launch_bounds__(kThreads)
f64_spec_rows_kernel(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                     uint16_t *__restrict__ comps, int64_t ldcomp, int64_t plane, WsHeader *ws, int slot)
{
    __shared__ unsigned long long red[5 * (kThreads / 32)];
    f64_spec_rows_body<NLEV>(X, rows, cols, ldx, comps, ldcomp, plane, ws, slot, blockIdx.x, blockIdx.y, gridDim.y, red);
}

// Transposed (K-major) planes: a 64 x 64 tile; lane p of warp q takes rows
// 2rp and 2rp+1 (rp = 4q + p / 8) and columns 16j + 2(p % 8) + {0, 1},
// j = 0..3, so eight lanes read 128 contiguous bytes of a row.  Each plane
// word packs the two entries adjacent in the transposed row; it is staged
// with each transposed row's 16-byte K-chunks permuted by an XOR with the
// column (a warp's stores hit 32 different banks) and written as 16-byte
// chunks of whole transposed rows.  Shared memory: [6][64][32] words.
// Block bid of nblk (tiles with a stride of nblk); smw: [6][kTile][kTile / 2]
// words, red: 5 * kThreads / 32 words of shared memory.
template <int NLEV>
__device__ __forceinline__ void f64_spec_transpose_body(const double *__restrict__ X, int64_t rows, int64_t cols,
                                                        int64_t ldx, uint16_t *__restrict__ comps, int64_t ldcomp,
                                                        int64_t plane, WsHeader *ws, int slot, int64_t bid,
                                                        int64_t nblk, uint32_t *smw, unsigned long long *red)
{
    const int v0 = spec_v0(ws, slot);
    const bool fast = v0 >= -78;
    float P[6] = {};
    if (fast) spec_units(v0 - 50, P);
    const bool vin = ((ldx & 1) == 0) && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0);
    const bool vout = ((ldcomp & 7) == 0) && ((plane & 7) == 0) && ((reinterpret_cast<uintptr_t>(comps) & 15u) == 0);
    const int q = threadIdx.x >> 5, p = lane_id();
    const int rp = 4 * q + (p >> 3), cg = p & 7;       // rows 2rp, 2rp + 1; columns 16j + 2cg + {0, 1}
    const int64_t tiles_r = (rows + kTile - 1) / kTile, tiles_c = (cols + kTile - 1) / kTile;
    SpecState st;
    // this thread's two entries in step j of tile t: eight lanes read 128
    // contiguous bytes of one row
    auto load = [&](int64_t t, int j, double (&x)[2][2]) {
        const int64_t r0 = (t / tiles_c) * kTile, gj = (t % tiles_c) * kTile + 16 * j + 2 * cg;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int64_t gi = r0 + 2 * rp + h;
            const double *src = X + gi * ldx + gj;
            if (gi < rows && vin && gj + 2 <= cols) {
                const double2 a = *reinterpret_cast<const double2 *>(src);
                x[h][0] = a.x; x[h][1] = a.y;
            } else {
#pragma unroll
                for (int e = 0; e < 2; ++e) x[h][e] = (gi < rows && gj + e < cols) ? src[e] : 0.0;
            }
        }
    };
    double xn[2][2] = {{0.0, 0.0}, {0.0, 0.0}};
    if (bid < tiles_r * tiles_c) load(bid, 0, xn);
    for (int64_t t = bid; t < tiles_r * tiles_c; t += nblk) {
        const int64_t r0 = (t / tiles_c) * kTile, c0 = (t % tiles_c) * kTile;
        // two adjacent columns per step (one 16-byte load per row), so that
        // the element body appears four times in the loop, not sixteen; the
        // next step's entries are loaded before this step is split
#pragma unroll 1
        for (int j = 0; j < 4; ++j) {
            double x[2][2];
#pragma unroll
            for (int h = 0; h < 2; ++h) { x[h][0] = xn[h][0]; x[h][1] = xn[h][1]; }
            if (j + 1 < 4) load(t, j + 1, xn);
            else if (t + nblk < tiles_r * tiles_c) load(t + nblk, 0, xn);
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                uint32_t s0[6], s1[6];
                spec_element<NLEV>(x[0][e], v0, fast, P, s0, st);
                spec_element<NLEV>(x[1][e], v0, fast, P, s1, st);
                // transposed row col, K-chunk rp / 4 stored at chunk (rp / 4) ^ cg: conflict-free
                const int col = 16 * j + 2 * cg + e;
#pragma unroll
                for (int r = 0; r < NLEV; ++r)
                    smw[(r * kTile + col) * (kTile / 2) + (((q ^ cg) << 2) | (p >> 3))] = pack2(s0[r], s1[r]);
            }
        }
        __syncthreads();
        // NLEV planes x 64 transposed rows x 8 chunks (two iterations per plane)
#pragma unroll 4
        for (int it = 0; it < NLEV * kTile * 8 / kThreads; ++it) {
            const int c = threadIdx.x + it * kThreads;
            const int r = c >> 9, orow = (c >> 3) & 63, ch = c & 7;
            const int64_t go = c0 + orow, gk = r0 + 8 * ch;
            if (go < cols && gk < rows) {
                const uint4 v = *reinterpret_cast<const uint4 *>(&smw[(r * kTile + orow) * (kTile / 2) + 4 * (ch ^ ((orow >> 1) & 7))]);
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
    spec_publish(st, v0, ws, slot, red);
}

template <int NLEV>
__global__ void __launch_bounds__(kThreads)
f64_spec_transpose_kernel(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                          uint16_t *__restrict__ comps, int64_t ldcomp, int64_t plane, WsHeader *ws, int slot)
{
    extern __shared__ __align__(16) uint32_t smw[];                  // [6][kTile][kTile / 2]
    __shared__ unsigned long long red[5 * (kThreads / 32)];
    f64_spec_transpose_body<NLEV>(X, rows, cols, ldx, comps, ldcomp, plane, ws, slot, blockIdx.x, gridDim.x, smw, red);
}

// Block b of a launch that holds nA blocks of one kind and nB of another:
// the first 2 min(nA, nB) blocks alternate between the kinds (blocks are
// dispatched roughly in index order, so both kinds run side by side), the
// rest belong to the larger kind.  Returns the block's index within its kind.
__device__ __forceinline__ int64_t pair_block(int64_t b, int64_t nA, int64_t nB, bool &is_a)
{
    const int64_t m = nA < nB ? nA : nB;
    if (b < 2 * m) { is_a = (b & 1) == 0; return b >> 1; }
    is_a = nA > nB;
    return m + (b - 2 * m);
}

// The level-0 maxima of both operands of an FP64 GEMM in one launch: nA
// blocks on A (header slot 0) and nB on B (slot 1), interleaved.
__global__ void __launch_bounds__(kThreads)
f64_max_gemm_kernel(const double *__restrict__ A, int64_t M, int64_t K, int64_t lda, const double *__restrict__ B,
                    int64_t N, int64_t ldb, WsHeader *ws, int64_t nA, int64_t nB)
{
    __shared__ unsigned long long red[kThreads / 32];
    bool is_a;
    const int64_t i = pair_block(blockIdx.x, nA, nB, is_a);
    if (is_a) f64_max_pass<0>(A, M, K, lda, ws, 0, i, nA, red);
    else f64_max_pass<0>(B, K, N, ldb, ws, 1, i, nB, red);
}

// The fused speculative pass for slices 0 .. NLEV-1.
template <int NLEV>
cudaError_t launch_spec(const double *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose, uint16_t *comps,
                        int64_t ldcomp, int64_t plane, WsHeader *ws, int slot, int gt, cudaStream_t st)
{
    if (transpose) {
        cudaError_t e = cudaFuncSetAttribute(f64_spec_transpose_kernel<NLEV>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSpecTransposeSmem);
        if (e != cudaSuccess) return e;
        f64_spec_transpose_kernel<NLEV><<<gt, kThreads, kSpecTransposeSmem, st>>>(X, rows, cols, ldx, comps, ldcomp,
                                                                                  plane, ws, slot);
    } else {
        // about eight blocks per SM, each over several rows
        const int64_t bx = (cols + 4 * kThreads - 1) / (4 * kThreads);
        const int64_t want = (152 * 8 + bx - 1) / bx;
        const int64_t by = rows < want ? rows : (want < 65535 ? want : 65535);
        f64_spec_rows_kernel<NLEV><<<dim3((unsigned)bx, (unsigned)by), kThreads, 0, st>>>(X, rows, cols, ldx, comps,
                                                                                          ldcomp, plane, ws, slot);
    }
    return cudaSuccess;
}

}  // namespace

cudaError_t launch_split_f64(const double *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose,
                             uint16_t *comps, int64_t ldcomp, int32_t *v_out, WsHeader *ws, int slot,
                             cudaStream_t st, int nlev)
{
    if (nlev < 3 || nlev > 6) return cudaErrorInvalidValue;
    const int64_t plane = (transpose ? cols : rows) * ldcomp;
    if (rows > 0 && cols > 0) {
        const int64_t segs = rows * ((cols + 4 * kThreads - 1) / (4 * kThreads));
        const int gmax = grid_for(segs, 152 * 8);
        const int64_t tiles = ((rows + kTile - 1) / kTile) * ((cols + kTile - 1) / kTile);
        const int gt = grid_for(tiles, 152 * 8);
        cudaError_t e = cudaSuccess;
        f64_max_kernel<0><<<gmax, kThreads, 0, st>>>(X, rows, cols, ldx, ws, slot);
        switch (nlev) {
        case 3: e = launch_spec<3>(X, rows, cols, ldx, transpose, comps, ldcomp, plane, ws, slot, gt, st); break;
        case 4: e = launch_spec<4>(X, rows, cols, ldx, transpose, comps, ldcomp, plane, ws, slot, gt, st); break;
        case 5: e = launch_spec<5>(X, rows, cols, ldx, transpose, comps, ldcomp, plane, ws, slot, gt, st); break;
        default: e = launch_spec<6>(X, rows, cols, ldx, transpose, comps, ldcomp, plane, ws, slot, gt, st); break;
        }
        if (e == cudaSuccess) e = cudaGetLastError();
        if (e == cudaSuccess)
            e = launch_f64_fix(X, rows, cols, ldx, transpose, comps, ldcomp, plane, ws, slot, v_out, st, nlev);
        return e;
    }
    // an empty matrix: all levels zero, nothing to fix
    return launch_f64_fix_empty(ws, slot, v_out, st);
}


// Both operands of an FP64 GEMM (A: M x K into row-major planes, B: K x N
// into K-major planes, row pitch ldcomp), with the level maxima of A and B in
// one launch; the speculative passes and verifiers stay one launch per
// operand.  Results are those of launch_split_f64 on A, then B.
cudaError_t launch_split_f64_gemm(const double *A, int64_t M, int64_t K, int64_t lda, const double *B, int64_t N,
                                  int64_t ldb, uint16_t *Ap, uint16_t *Bp, int64_t ldcomp, int32_t *vA_out,
                                  int32_t *vB_out, WsHeader *ws, cudaStream_t st, int nlev)
{
    if (nlev < 3 || nlev > 6) return cudaErrorInvalidValue;
    if (M == 0 || N == 0 || K == 0) {
        cudaError_t e = launch_split_f64(A, M, K, lda, false, Ap, ldcomp, vA_out, ws, 0, st, nlev);
        if (e == cudaSuccess) e = launch_split_f64(B, K, N, ldb, true, Bp, ldcomp, vB_out, ws, 1, st, nlev);
        return e;
    }
    // level-0 maxima: blocks shared in proportion to the entries, at most 152 x 8 in all
    const int64_t segA = M * ((K + 4 * kThreads - 1) / (4 * kThreads)), segB = K * ((N + 4 * kThreads - 1) / (4 * kThreads));
    const double fa = (double)(M * K) / (double)(M * K + K * N);
    int64_t nA = (int64_t)(152 * 8 * fa + 0.5), nB = 152 * 8 - nA;
    nA = nA < 1 ? 1 : (nA > segA ? segA : nA);
    nB = nB < 1 ? 1 : (nB > segB ? segB : nB);
    f64_max_gemm_kernel<<<(unsigned)(nA + nB), kThreads, 0, st>>>(A, M, K, lda, B, N, ldb, ws, nA, nB);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // the speculative passes stay one launch per operand: in one launch the
    // row blocks would reserve the transposed blocks' shared memory (measured
    // 15-25 % slower)
    const int gB = grid_for(((K + kTile - 1) / kTile) * ((N + kTile - 1) / kTile), 152 * 8);
    switch (nlev) {
    case 3:
        e = launch_spec<3>(A, M, K, lda, false, Ap, ldcomp, M * ldcomp, ws, 0, 0, st);
        if (e == cudaSuccess) e = launch_spec<3>(B, K, N, ldb, true, Bp, ldcomp, N * ldcomp, ws, 1, gB, st);
        break;
    case 4:
        e = launch_spec<4>(A, M, K, lda, false, Ap, ldcomp, M * ldcomp, ws, 0, 0, st);
        if (e == cudaSuccess) e = launch_spec<4>(B, K, N, ldb, true, Bp, ldcomp, N * ldcomp, ws, 1, gB, st);
        break;
    case 5:
        e = launch_spec<5>(A, M, K, lda, false, Ap, ldcomp, M * ldcomp, ws, 0, 0, st);
        if (e == cudaSuccess) e = launch_spec<5>(B, K, N, ldb, true, Bp, ldcomp, N * ldcomp, ws, 1, gB, st);
        break;
    default:
        e = launch_spec<6>(A, M, K, lda, false, Ap, ldcomp, M * ldcomp, ws, 0, 0, st);
        if (e == cudaSuccess) e = launch_spec<6>(B, K, N, ldb, true, Bp, ldcomp, N * ldcomp, ws, 1, gB, st);
        break;
    }
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e == cudaSuccess) e = launch_f64_fix(A, M, K, lda, false, Ap, ldcomp, M * ldcomp, ws, 0, vA_out, st, nlev);
    if (e == cudaSuccess) e = launch_f64_fix(B, K, N, ldb, true, Bp, ldcomp, N * ldcomp, ws, 1, vB_out, st, nlev);
    return e;
}

}  // namespace emu
