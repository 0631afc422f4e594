// Host-side launch functions of the kernels, shared by the C-ABI translation
// units (emu_api.cu, noalloc.cu, host_api.cu).  Each enqueues its kernels on
// `st` and returns the launch error; device-side failures set flag bits.
#pragma once

#include "common.cuh"

namespace emu {

// Eq. (fp32split): X [rows][ldx] FP32 -> 3 BF16 planes of [transpose ? cols : rows][ldcomp].
// plane: distance between planes in elements (0 = dense: (transpose ? cols : rows) * ldcomp).
cudaError_t launch_split_f32(const float *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose,
                             uint16_t *comps, int64_t ldcomp, WsHeader *ws, cudaStream_t st, int64_t plane = 0);

// Eq. (fp64split): X -> 6 BF16 planes and the level exponents v_out[6]; `slot`
// selects the header's per-operand state (0 = A, 1 = B).  nlev (3..6): only
// slices 0 .. nlev-1 are wanted (a product-sum with d = nlev uses no more);
// planes from nlev on are then left as they were and their levels read as
// zero levels, unless the speculative levels failed and the literal passes
// redid all six.
cudaError_t launch_split_f64(const double *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose,
                             uint16_t *comps, int64_t ldcomp, int32_t *v_out, WsHeader *ws, int slot,
                             cudaStream_t st, int nlev = 6);

// Both operands of an FP64 GEMM split as launch_split_f64 splits A (rows x
// cols = M x K, row-major planes, slot 0) and then B (K x N, K-major planes,
// slot 1), with the level-maximum passes of the two sharing one launch.
cudaError_t launch_split_f64_gemm(const double *A, int64_t M, int64_t K, int64_t lda, const double *B, int64_t N,
                                  int64_t ldb, uint16_t *Ap, uint16_t *Bp, int64_t ldcomp, int32_t *vA_out,
                                  int32_t *vB_out, WsHeader *ws, cudaStream_t st, int nlev);

// Number of diagonals d of an FP64-mode product count (Eq. (fp64productcounts):
// nprod = d (d + 1) / 2), i.e. the slices 0 .. d-1 a product-sum reads; 0 for
// any other count.
inline int f64_diagonals(int nprod)
{
    return nprod == 6 ? 3 : nprod == 10 ? 4 : nprod == 15 ? 5 : nprod == 21 ? 6 : 0;
}

// Eq. (fp64split) with one set of levels per plane row (an input row, or an
// input column when transposed): v_out[6][plane rows] (level-major);
// scratch: rc_scratch_bytes(plane rows) bytes, 8-byte aligned; slot: the
// header's per-operand state (0 = A, 1 = B).
// The whole-matrix FP64 split's verifier and literal fix passes (one
// cooperative launch after the speculative pass), and its form for an empty
// matrix.
cudaError_t launch_f64_fix(const double *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose, uint16_t *comps,
                           int64_t ldcomp, int64_t plane, WsHeader *ws, int slot, int32_t *v_out, cudaStream_t st,
                           int nlev);
cudaError_t launch_f64_fix_empty(WsHeader *ws, int slot, int32_t *v_out, cudaStream_t st);
cudaError_t launch_split_f64_rc(const double *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose,
                                uint16_t *comps, int64_t ldcomp, int32_t *v_out, void *scratch, WsHeader *ws,
                                int slot, cudaStream_t st);
inline size_t rc_scratch_bytes(int64_t plane_rows) { return (size_t)plane_rows * 28; }

// Product-sums from K-major planes; a_plane / b_plane: distance between the A /
// B planes in elements (0 = dense: M * ldcomp / N * ldcomp), so that a row
// panel of A or a column panel of B in a larger plane set can be multiplied
// on its own.
// c_zeroed: C is zero on entry, so when few output tiles would leave SMs idle
// the product-sum may split K in two and add both halves into C.
cudaError_t launch_prodsum_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                               int64_t ldcomp, float *C, int64_t ldc, uint32_t *flags, cudaStream_t st,
                               int64_t a_plane = 0, int64_t b_plane = 0, bool c_zeroed = false);
// Both operands of an FP32 GEMM (A: M x K row-major planes, B: K x N K-major
// planes, row pitch ldcomp, B's planes at Bp) split in one launch; with C
// non-null the launch also sets the M x N result C (ldc) to zero.
cudaError_t launch_split_f32_gemm(const float *A, int64_t M, int64_t K, int64_t lda, const float *B, int64_t N,
                                  int64_t ldb, uint16_t *Ap, uint16_t *Bp, int64_t ldcomp, WsHeader *ws, float *C,
                                  int64_t ldc, cudaStream_t st);
// Tile width (256, 128 or 64) the FP32 product-sums pick for an M x N result,
// and the number of K-parts (1 or 2) the product-sum takes when C is cleared
// first.
int f32_tile_columns(int64_t M, int64_t N);
int f32_prodsum_launches(int64_t M, int64_t N);
int f32_tile_rows(int64_t M, int64_t N);
int f32_split_parts(int64_t M, int64_t N, int64_t K);
// Eq. (fp32split) and the FP32 product-sum in one kernel: A (M x K, lda) and
// B (K x N, ldb) FP32 row-major are split inside the product-sum's producer;
// no planes are written.  flags receives the split's domain flags.
cudaError_t launch_gemm_f32_fused(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda, const float *B,
                                  int64_t ldb, float *C, int64_t ldc, uint32_t *flags, cudaStream_t st);
// acc: FP64 accumulator scratch of f64_acc_bytes(M, N) bytes (16-byte aligned).
// rowcol: vA / vB are levels per row of A ([6][M]) and per column of B ([6][N]).
// T (optional, M x N FP32 with leading dimension ldt): a merged tail, added to
// every element once after the last product.
cudaError_t launch_prodsum_f64(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                               int64_t ldcomp, const int32_t *vA, const int32_t *vB, int nprod, double *C,
                               int64_t ldc, double *acc, uint32_t *flags, cudaStream_t st, int64_t a_plane = 0,
                               bool rowcol = false, const float *T = nullptr, int64_t ldt = 0);
// Merged tail of the FP64 mode: T (M x N FP32, leading dimension ldt) = the
// sum over the products (i, j) with L <= i + j < d of A_i B_j, accumulated in
// one FP32 tensor-memory accumulator over all of K; 3 <= L < d <= 6.
cudaError_t launch_prodsum_tail(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                                int64_t ldcomp, int L, int d, float *T, int64_t ldt, uint32_t *flags,
                                cudaStream_t st);

// How the FP64 product-sum covers an M x N result: tiles of rows x cols
// (128 x 128, 128 x 256, or 256 x 256 on CTA pairs), `tiles` of them in the
// first launch and, when launches == 2, the remaining rest tiles as 128 x 128
// parts in a second launch of the 128 x 128 kernel.
struct F64Plan {
    int rows = 0, cols = 0, launches = 0;
    int64_t tiles = 0, rest = 0;
};
F64Plan f64_plan(int64_t M, int64_t N);
// Tile width (128 or 256) the FP64 product-sum picks for an M x N result.
int f64_tile_columns(int64_t M, int64_t N);
// The FP64 product-sum on 128 x 256 tiles, or with pair on 256 x 256 tiles
// computed by clusters of two CTAs (prodsum_f64w.cu); launch_prodsum_f64
// calls it for the first `tiles` tiles in raster order.  acc:
// f64_acc_bytes(M, N) bytes.
cudaError_t launch_prodsum_f64_wide(int64_t M, int64_t N, int64_t K, const uint16_t *Ap, const uint16_t *Bp,
                                    int64_t ldcomp, const int32_t *vA, const int32_t *vB, int nprod, double *C,
                                    int64_t ldc, double *acc, uint32_t *flags, cudaStream_t st, int64_t a_plane,
                                    bool rowcol, const float *T, int64_t ldt, int64_t tiles, bool pair);

// Bytes of the FP64 product-sum's accumulator, enough for either tile shape:
// one FP64 tile of 128 x 128 (narrow kernel) or 128 x 256 (wide kernel) per
// CTA tile.
inline size_t f64_acc_bytes(int64_t M, int64_t N)
{
    const size_t tm = (size_t)((M + 127) / 128);
    const size_t narrow = tm * (size_t)((N + 127) / 128) * 128u * 128u * sizeof(double);
    const size_t wide = tm * (size_t)((N + 255) / 256) * 128u * 256u * sizeof(double);
    return narrow > wide ? narrow : wide;
}

// General-GEMM epilogue: C <- fl(fl(alpha P) + fl(beta C)) (beta = 0: C <- fl(alpha P), C not read).
cudaError_t launch_axpby_f32(const float *P, int64_t ldp, float *C, int64_t ldc, int64_t M, int64_t N, float alpha,
                             float beta, cudaStream_t st);
cudaError_t launch_axpby_f64(const double *P, int64_t ldp, double *C, int64_t ldc, int64_t M, int64_t N,
                             double alpha, double beta, cudaStream_t st);

}  // namespace emu
