// FP32 three-slice residual split, Eq. (fp32split): element pairs rounded by
// the hardware BF16x2 conversion; row-major planes straight from registers,
// transposed (K-major) planes through a conflict-free shared-memory tile.
#include "split_common.cuh"
#include "split_f32_pair.cuh"

namespace emu {

namespace {

// ------------------------------------------------------ FP32 split kernels
// Row-major planes: thread = 8 consecutive elements of a row (two 16-byte
// loads, one 16-byte store per plane), no shared memory.  Rows advance by
// the grid's y dimension.
// Block (bx, by) of a grid with gy rows of blocks; returns the block's part of
// the flag check (the largest |x| bit pattern seen), for publish_f32_flags.
__device__ __forceinline__ uint32_t split_f32_rows_body(const float *__restrict__ X, int64_t rows, int64_t cols,
                                                    int64_t ldx, uint16_t *__restrict__ comps, int64_t ldcomp,
                                                    int64_t plane, WsHeader *ws, int64_t bx, int64_t by, int64_t gy)
{
    const bool vin = ((ldx & 3) == 0) && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0);
    const bool vout = ((ldcomp & 7) == 0) && ((plane & 7) == 0) && ((reinterpret_cast<uintptr_t>(comps) & 15u) == 0);
    const int64_t j0 = (bx * kThreads + threadIdx.x) * 8;
    uint32_t amax = 0;
    if (j0 < cols) {
        const bool full = j0 + 8 <= cols;
        for (int64_t i = by; i < rows; i += gy) {
            const float *src = X + i * ldx + j0;
            float x[8];
            if (vin && full) {
                const float4 a = reinterpret_cast<const float4 *>(src)[0], b = reinterpret_cast<const float4 *>(src)[1];
                x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
            } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) x[e] = (j0 + e < cols) ? src[e] : 0.0f;
            }
            uint32_t w[3][4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                amax = abs_bits_max(amax, x[2 * e], x[2 * e + 1]);
                split_pair(x[2 * e], x[2 * e + 1], w[0][e], w[1][e], w[2][e]);
            }
            uint16_t *dst = comps + i * ldcomp + j0;
#pragma unroll
            for (int r = 0; r < 3; ++r) {
                if (vout && full) {
                    *reinterpret_cast<uint4 *>(dst + r * plane) = make_uint4(w[r][0], w[r][1], w[r][2], w[r][3]);
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        if (j0 + e < cols) dst[r * plane + e] = (uint16_t)(w[r][e >> 1] >> (16 * (e & 1)));
                }
            }
        }
    }
    return amax;
}

// Row-major planes by 64 x 64 tiles (the GEMM's one-launch split of A):
// thread t takes rows t / 16 + 16 i (i = 0..3) and columns 4 (t % 16) .. + 3
// of a tile, so a warp reads two whole 256-byte row segments per load and
// writes 128 contiguous bytes of two plane rows per store; the next tile's
// entries are loaded before this tile is split and stored, so every thread
// has four to eight 16-byte loads in flight.  Block bid of nblk (tiles with a
// stride of nblk).  Returns the block's part of the flag check.
__device__ __forceinline__ uint32_t split_f32_rowtile_body(const float *__restrict__ X, int64_t rows, int64_t cols,
                                                       int64_t ldx, uint16_t *__restrict__ comps, int64_t ldcomp,
                                                       int64_t plane, int64_t bid, int64_t nblk)
{
    const bool vin = ((ldx & 3) == 0) && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0);
    const bool vout = ((ldcomp & 3) == 0) && ((plane & 3) == 0) && ((reinterpret_cast<uintptr_t>(comps) & 7u) == 0);
    const int tr = threadIdx.x >> 4, tc = 4 * (threadIdx.x & 15);
    const int64_t tiles_c = (cols + kTile - 1) / kTile, ntiles = ((rows + kTile - 1) / kTile) * tiles_c;
    auto load_tile = [&](int64_t t, float (&x)[4][4]) {
        const int64_t r0 = (t / tiles_c) * kTile, gj = (t % tiles_c) * kTile + tc;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int64_t gi = r0 + tr + 16 * i;
            const float *src = X + gi * ldx + gj;
            if (gi < rows && vin && gj + 4 <= cols) {
                const float4 a = *reinterpret_cast<const float4 *>(src);
                x[i][0] = a.x; x[i][1] = a.y; x[i][2] = a.z; x[i][3] = a.w;
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) x[i][e] = (gi < rows && gj + e < cols) ? src[e] : 0.0f;
            }
        }
    };
    uint32_t amax = 0;
    float x[4][4];
    if (bid < ntiles) load_tile(bid, x);
    for (int64_t t = bid; t < ntiles; t += nblk) {
        float xn[4][4];
        if (t + nblk < ntiles) load_tile(t + nblk, xn);
        const int64_t r0 = (t / tiles_c) * kTile, gj = (t % tiles_c) * kTile + tc;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int64_t gi = r0 + tr + 16 * i;
            uint32_t w[3][2];
            amax = abs_bits_max(abs_bits_max(amax, x[i][0], x[i][1]), x[i][2], x[i][3]);
            split_pair(x[i][0], x[i][1], w[0][0], w[1][0], w[2][0]);
            split_pair(x[i][2], x[i][3], w[0][1], w[1][1], w[2][1]);
            if (gi < rows) {
                uint16_t *dst = comps + gi * ldcomp + gj;
#pragma unroll
                for (int r = 0; r < 3; ++r) {
                    if (vout && gj + 4 <= cols) {
                        *reinterpret_cast<uint2 *>(dst + r * plane) = make_uint2(w[r][0], w[r][1]);
                    } else {
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            if (gj + e < cols) dst[r * plane + e] = (uint16_t)(w[r][e >> 1] >> (16 * (e & 1)));
                    }
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int e = 0; e < 4; ++e) x[i][e] = xn[i][e];
    }
    return amax;
}

__global__ void __launch_bounds__(kThreads)
split_f32_rows_kernel(const float *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                      uint16_t *__restrict__ comps, int64_t ldcomp, int64_t plane, WsHeader *ws)
{
    publish_f32_flags(split_f32_rows_body(X, rows, cols, ldx, comps, ldcomp, plane, ws, blockIdx.x, blockIdx.y,
                                          gridDim.y), &ws->flags);
}

// Transposed (K-major) planes: a 64 x 64 tile of X.  Lane p of warp q takes
// rows 2rp and 2rp+1 (rp = 4q + p / 8) and columns 32j + 4(p % 8) + {0..3},
// j = 0, 1, so eight lanes read 128 contiguous bytes of a row and each slice
// word packs the two elements that are adjacent in the transposed row; the
// words go to shared memory, each transposed row's 16-byte K-chunks permuted
// by an XOR with its column (so a warp's stores hit 32 different banks), and
// leave as 16-byte chunks of whole transposed rows.
// Block bid of nblk blocks (tiles taken with a stride of nblk); sm: the
// block's [3][kTile][kTile / 2] staging words.  Returns the block's part of
// the flag check, as the row body does.
__device__ __forceinline__ uint32_t split_f32_transpose_body(const float *__restrict__ X, int64_t rows, int64_t cols,
                                                         int64_t ldx, uint16_t *__restrict__ comps, int64_t ldcomp,
                                                         int64_t plane, WsHeader *ws, int64_t bid, int64_t nblk,
                                                         uint32_t (*sm)[kTile][kTile / 2])
{
    const bool vin = ((ldx & 3) == 0) && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0);
    const bool vout = ((ldcomp & 7) == 0) && ((plane & 7) == 0) && ((reinterpret_cast<uintptr_t>(comps) & 15u) == 0);
    const int q = threadIdx.x >> 5, p = lane_id();
    const int rp = 4 * q + (p >> 3), cg = p & 7;       // rows 2rp, 2rp + 1; columns 32j + 4cg + {0..3}
    const int64_t tiles_r = (rows + kTile - 1) / kTile, tiles_c = (cols + kTile - 1) / kTile;
    // the next tile's rows are loaded before this tile is split and stored,
    // so that the loads of a block overlap its own stores; eight lanes read
    // 128 contiguous bytes of one row
    auto load_tile = [&](int64_t t, float (&x)[2][8]) {
        const int64_t r0 = (t / tiles_c) * kTile, c0 = (t % tiles_c) * kTile;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int64_t gi = r0 + 2 * rp + h;
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                const int64_t gj = c0 + 32 * j + 4 * cg;
                const float *src = X + gi * ldx + gj;
                if (gi < rows && vin && gj + 4 <= cols) {
                    const float4 a = *reinterpret_cast<const float4 *>(src);
                    x[h][4 * j] = a.x; x[h][4 * j + 1] = a.y; x[h][4 * j + 2] = a.z; x[h][4 * j + 3] = a.w;
                } else {
#pragma unroll
                    for (int e = 0; e < 4; ++e) x[h][4 * j + e] = (gi < rows && gj + e < cols) ? src[e] : 0.0f;
                }
            }
        }
    };
    uint32_t amax = 0;
    float x[2][8];
    if (bid < tiles_r * tiles_c) load_tile(bid, x);
    for (int64_t t = bid; t < tiles_r * tiles_c; t += nblk) {
        const int64_t r0 = (t / tiles_c) * kTile, c0 = (t % tiles_c) * kTile;
        float xn[2][8];
        if (t + nblk < tiles_r * tiles_c) load_tile(t + nblk, xn);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            amax = abs_bits_max(amax, x[0][e], x[1][e]);
            uint32_t w0, w1, w2;
            split_pair(x[0][e], x[1][e], w0, w1, w2);
            // transposed row col, K-chunk rp / 4 stored at chunk (rp / 4) ^ cg: conflict-free
            const int col = 32 * (e >> 2) + 4 * cg + (e & 3), w = ((q ^ cg) << 2) | (p >> 3);
            sm[0][col][w] = w0;
            sm[1][col][w] = w1;
            sm[2][col][w] = w2;
        }
        __syncthreads();
        // 3 planes x 64 transposed rows x 8 chunks of 16 bytes
#pragma unroll
        for (int it = 0; it < 3 * kTile * 8 / kThreads; ++it) {
            const int c = threadIdx.x + it * kThreads;
            const int r = c >> 9, orow = (c >> 3) & 63, ch = c & 7;
            const int64_t go = c0 + orow, gk = r0 + 8 * ch;
            if (go < cols && gk < rows) {
                const uint4 v = *reinterpret_cast<const uint4 *>(&sm[r][orow][4 * (ch ^ ((orow >> 2) & 7))]);
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
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int e = 0; e < 8; ++e) x[h][e] = xn[h][e];
    }
    return amax;
}

__global__ void __launch_bounds__(kThreads)
split_f32_transpose_kernel(const float *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx,
                           uint16_t *__restrict__ comps, int64_t ldcomp, int64_t plane, WsHeader *ws)
{
    __shared__ __align__(16) uint32_t sm[3][kTile][kTile / 2];   // [plane][transposed row][word]
    publish_f32_flags(split_f32_transpose_body(X, rows, cols, ldx, comps, ldcomp, plane, ws, blockIdx.x, gridDim.x, sm),
                      &ws->flags);
}

// Both operands of an FP32 GEMM in one launch: blocks [0, nA) split A into
// row-major planes (by rows on an ax x (nA / ax) grid when ax > 0, else by
// 64 x 64 tiles), blocks [nA, nA + nB) split B into K-major planes, and
// blocks from nA + nB on set the M x N result C to zero (a product-sum that
// adds its K-parts into C needs it cleared).
__global__ void __launch_bounds__(kThreads)
split_f32_gemm_kernel(const float *__restrict__ A, int64_t M, int64_t K, int64_t lda, const float *__restrict__ B,
                      int64_t N, int64_t ldb, uint16_t *__restrict__ Ap, uint16_t *__restrict__ Bp, int64_t ldcomp,
                      WsHeader *ws, int64_t ax, int64_t nA, int64_t nB, float *__restrict__ C, int64_t ldc, int64_t nC)
{
    __shared__ __align__(16) uint32_t sm[3][kTile][kTile / 2];
    // the product-sum launched after this kernel may start its set-up as soon
    // as every block of this one is running (it waits for all of it before
    // reading planes or C)
    griddep_launch_dependents();
    const int64_t b = blockIdx.x;
    if (b < nA + nB) {
        const uint32_t amax =
            b >= nA ? split_f32_transpose_body(B, K, N, ldb, Bp, ldcomp, N * ldcomp, ws, b - nA, nB, sm)
            : ax > 0 ? split_f32_rows_body(A, M, K, lda, Ap, ldcomp, M * ldcomp, ws, b % ax, b / ax, nA / ax)
                     : split_f32_rowtile_body(A, M, K, lda, Ap, ldcomp, M * ldcomp, b, nA);
        // the flag word is cleared by the operation before this launch, which
        // may still be running when this kernel is its programmatic dependent
        griddep_wait();
        publish_f32_flags(amax, &ws->flags);
    } else {
        const int64_t c = b - nA - nB;
        const bool vec = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15u) == 0);
        for (int64_t i = c; i < M; i += nC) {
            float *row = C + i * ldc;
            if (vec) {
                for (int64_t j = 4 * (int64_t)threadIdx.x; j < N; j += 4 * kThreads) {
                    if (j + 4 <= N) *reinterpret_cast<float4 *>(row + j) = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
                    else for (int64_t e = j; e < N; ++e) row[e] = 0.0f;
                }
            } else {
                for (int64_t j = threadIdx.x; j < N; j += kThreads) row[j] = 0.0f;
            }
        }
    }
}

}  // namespace

// ----------------------------------------------------------- host launchers
cudaError_t launch_split_f32(const float *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose,
                             uint16_t *comps, int64_t ldcomp, WsHeader *ws, cudaStream_t st, int64_t plane_stride)
{
    if (rows == 0 || cols == 0) return cudaSuccess;
    const int64_t plane = plane_stride ? plane_stride : (transpose ? cols : rows) * ldcomp;
    if (transpose) {
        const int64_t tiles = ((rows + kTile - 1) / kTile) * ((cols + kTile - 1) / kTile);
        split_f32_transpose_kernel<<<grid_for(tiles, 152 * 8), kThreads, 0, st>>>(X, rows, cols, ldx, comps, ldcomp,
                                                                                   plane, ws);
    } else {
        const int64_t bx = (cols + 8 * kThreads - 1) / (8 * kThreads);
        const int64_t by = rows < 4096 ? rows : 4096;
        split_f32_rows_kernel<<<dim3((unsigned)bx, (unsigned)by), kThreads, 0, st>>>(X, rows, cols, ldx, comps, ldcomp,
                                                                                     plane, ws);
    }
    return cudaGetLastError();
}

// Both operands of an FP32 GEMM (A: M x K, B: K x N) into planes of row
// pitch ldcomp laid out as the GEMM workspace holds them, in one launch; with
// C non-null also C <- 0.
cudaError_t launch_split_f32_gemm(const float *A, int64_t M, int64_t K, int64_t lda, const float *B, int64_t N,
                                  int64_t ldb, uint16_t *Ap, uint16_t *Bp, int64_t ldcomp, WsHeader *ws, float *C,
                                  int64_t ldc, cudaStream_t st)
{
    if (M == 0 || N == 0 || K == 0) return cudaSuccess;
    // Operands of at most 256 tiles of 64 x 64 each: one block per tile, A by
    // tiles too, and at most 96 blocks clearing C, so that the launch is one
    // wave (608 blocks: four 256-thread blocks per SM at the kernel's 64
    // registers) and its time one round trip to DRAM.  Larger operands: rows
    // of A on 608 blocks, 608 blocks of B tiles (measured faster there).
    const int64_t tiles_a = ((M + kTile - 1) / kTile) * ((K + kTile - 1) / kTile);
    const int64_t tiles_b = ((K + kTile - 1) / kTile) * ((N + kTile - 1) / kTile);
    const bool small = tiles_a <= 256 && tiles_b <= 256;
    int64_t ax = 0, nA = tiles_a, nB = tiles_b, nC = 0;
    if (small) {
        nC = C ? (M < 96 ? M : 96) : 0;
    } else {
        ax = (K + 8 * kThreads - 1) / (8 * kThreads);
        const int64_t want = (152 * 4 + ax - 1) / ax;
        nA = ax * (M < want ? M : want);
        nB = grid_for(tiles_b, 152 * 4);
        nC = C ? (M < 152 ? M : 152) : 0;
    }
    cudaError_t e;
    // a programmatic dependent of the clearing of the workspace header, which
    // only its flag publication waits for
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(nA + nB + nC));
    cfg.blockDim = dim3(kThreads);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, split_f32_gemm_kernel, A, M, K, lda, B, N, ldb, Ap, Bp, ldcomp, ws, ax, nA, nB, C,
                           ldc, nC);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace emu
