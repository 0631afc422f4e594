/*
 * emu.h -- C-ABI of the GB300 (sm_103a) BF16 component-product GEMM emulation
 * of arXiv 2609.04663, "BF16 Component-Product Emulation of FP32 and FP64 GEMM
 * on Intel AMX".
 *
 *   FP32 mode: C = A.B for FP32 A, B.  Each operand is split into 3 BF16
 *   slices (Eq. (fp32split)) and the 6 products with i + j <= 2 are kept
 *   (Eq. (fp32six), Algorithm 1), accumulated in FP32.
 *
 *   FP64 mode: C = A.B for FP64 A, B inside the BF16 exponent range
 *   (Eq. (bf16rangefp64)).  Each operand is split into 6 BF16 slices by the
 *   fixed simplified Ozaki projection (Eq. (fp64split)); nprod = 6, 10, 15 or
 *   21 products (i + j < d, d = 3..6, Eq. (fp64productcounts)) are kept.  Each
 *   product is formed in FP32 per K-chunk of 256 (exact partials, summed
 *   exactly) and widened and accumulated in FP64 (Eq. (fp64reconstruction),
 *   Algorithm 2).
 *
 * Common conventions
 *   - Every pointer argument named as a matrix, plane set, workspace or v_out
 *     is a DEVICE pointer owned by the caller.  The library never allocates,
 *     frees or keeps a reference to caller memory after the call returns.
 *   - Matrices are row-major with a leading dimension in elements (ld >= cols).
 *   - All work is enqueued on `stream` and is asynchronous to the host; the
 *     only host synchronisation is emu_read_flags.
 *   - Synchronous errors (bad arguments, launch failures) are returned as an
 *     emu_status before or while enqueuing.  Numerical-domain violations and
 *     watchdog timeouts are found on the device: they set EMU_FLAG_* bits in
 *     the flag word at the start of the workspace, which every call clears
 *     first; read them with emu_read_flags.  The paper has no fallback for
 *     such inputs (Sections 3.1, 3.2): results are then unspecified.
 *   - M = 0 or N = 0 is a no-op; K = 0 writes zeros to C.
 *   - Component planes ("comps"): BF16 bit patterns (uint16), plane r of
 *     a set at comps + r * rows_out * ldcomp, each plane row-major
 *     [rows_out][ldcomp].  For an A operand (transpose = 0) rows_out = rows of
 *     X; for a B operand (transpose = 1) the plane is stored transposed,
 *     [cols][rows] -- K-major, as the tensor-core GEMM reads both operands.
 *   - Product-sum entry points take planes as written by the split with
 *     ldcomp a multiple of 8 and 16-byte aligned plane bases (the tensor
 *     memory accelerator requires 16-byte strides); otherwise
 *     EMU_ERR_MISALIGNED.
 *   - Requires an sm_103 (GB300) device; the library holds sm_103a code only.
 */
#ifndef EMU_H
#define EMU_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; 0 is the legacy default stream. */
typedef struct CUstream_st *emu_stream_t;

typedef enum {
    EMU_OK = 0,
    EMU_ERR_INVALID_ARG = 1,          /* negative size, ld < cols, bad nprod, NULL pointer */
    EMU_ERR_MISALIGNED = 2,           /* plane base / ldcomp not 16-byte compatible */
    EMU_ERR_WORKSPACE_TOO_SMALL = 3,  /* ws_bytes below the *_workspace_bytes value */
    EMU_ERR_CUDA = 4,                 /* a CUDA call or kernel launch failed */
    EMU_ERR_UNSUPPORTED = 5           /* size beyond the library's limits */
} emu_status;

/* Asynchronous flag bits (emu_read_flags). */
#define EMU_FLAG_NONFINITE 0x1u  /* an input entry is NaN or infinite */
#define EMU_FLAG_RANGE     0x2u  /* an FP64 input entry is outside F64^B, Eq. (bf16rangefp64) */
#define EMU_FLAG_SLICE     0x4u  /* a slice entry is not a normal BF16 value: FP64 mode,
                                    Z != fl_BF16(Z), or Z nonzero with |Z| < 2^-126
                                    (Section 4.3); FP32 mode, a non-finite slice */
#define EMU_FLAG_TIMEOUT   0x8u  /* a bounded wait inside a kernel gave up (about 2 s);
                                    the kernel stopped early and C is incomplete */

/* v_out value of a level whose residual is all zero (Section 4.3). */
#define EMU_ZERO_LEVEL INT32_MIN

/* Bytes of workspace emu_split_f32 / emu_split_f64 need (flag word and the
 * per-level maxima of the FP64 split).  mode is 32 or 64. */
size_t emu_split_workspace_bytes(int mode);

/* The splits take `transpose` (the B operand's K-major planes) and a plane
 * row pitch `ldcomp` in place of a layout selector: planes in memory are
 * always planar rows, and the shared-memory swizzle the tensor cores need is
 * applied by the tensor memory accelerator when a tile is loaded. */

/* FP32 three-slice split, Eq. (fp32split) / Algorithm 1 (Split_FP32):
 *   A_r = fl_BF16(A^(r)), A^(r+1) = fl32(A^(r) - A_r), r = 0, 1, 2,
 * fl_BF16 = round to nearest, ties to even (Section 4.2).
 * X: rows x cols FP32, leading dimension ldx (elements, >= cols).
 * transpose = 0: comps holds 3 planes [rows][ldcomp] (ldcomp >= cols);
 * transpose = 1: comps holds 3 planes [cols][ldcomp] (ldcomp >= rows).
 * Padding columns of the planes are not written.  Bit-exact and
 * deterministic.  Flags: EMU_FLAG_NONFINITE, EMU_FLAG_SLICE. */
emu_status emu_split_f32(const float *X, int64_t rows, int64_t cols, int64_t ldx, int transpose,
                         uint16_t *comps, int64_t ldcomp, void *ws, size_t ws_bytes,
                         emu_stream_t stream);

/* FP64 six-slice split, Eq. (fp64split) / Algorithm 2 (Split_FP64):
 *   v^(r) = ceil(log2(max_ij |A^(r)_ij|)) over the whole matrix,
 *   Z = fl64(fl64(A^(r) + 2^(v+45)) - 2^(v+45)), A_r = fl_BF16(Z),
 *   A^(r+1) = fl64(A^(r) - A_r), r = 0..5; an all-zero residual makes its
 *   slice and all later slices zero with v = EMU_ZERO_LEVEL.
 * Layout as emu_split_f32 with 6 planes.  v_out: device int32[6] receiving
 * v^(0..5).  Bit-exact and deterministic for inputs in the domain.  Flags:
 * EMU_FLAG_NONFINITE, EMU_FLAG_RANGE, EMU_FLAG_SLICE (planes then unspecified). */
emu_status emu_split_f64(const double *X, int64_t rows, int64_t cols, int64_t ldx, int transpose,
                         uint16_t *comps, int64_t ldcomp, int32_t *v_out, void *ws,
                         size_t ws_bytes, emu_stream_t stream);

/* Eq. (fp64split) with one set of six levels per plane row instead of one per
 * matrix: the vector scaling of the standard Ozaki scheme (Eq.
 * (ozakiscaled), Section 4.3).  Plane rows are the rows of X (transpose = 0)
 * or its columns (transpose = 1, K-major planes for the B operand), so a
 * GEMM gets levels per row of A and per column of B.  Each vector is split
 * exactly as the whole-matrix split would split it alone, so rows and columns
 * of very different magnitudes keep their own precision; results are
 * bit-identical to the oracle's split_f64_rows.  comps: 6 planes
 * [6][plane rows][ldcomp]; v_out: device int32 [6][plane rows]
 * (level-major; EMU_ZERO_LEVEL once a vector's residual is zero); ws: at
 * least emu_split_f64_rowcol_workspace_bytes(plane rows).  Flags as
 * emu_split_f64. */
size_t emu_split_f64_rowcol_workspace_bytes(int64_t plane_rows);
emu_status emu_split_f64_rowcol(const double *X, int64_t rows, int64_t cols, int64_t ldx,
                                int transpose, uint16_t *comps, int64_t ldcomp, int32_t *v_out,
                                void *ws, size_t ws_bytes, emu_stream_t stream);

/* FP64-mode GEMM (Algorithm 2, same product-outer sum as emu_gemm_f64)
 * with levels per row of A and per column of B (emu_split_f64_rowcol).
 * Every chunk partial stays exact in the unit of its own output element, so
 * C equals the oracle's gemm_f64_rowcol bit for bit.  Row and column scaling
 * by powers of two commutes with it exactly, which the whole-matrix levels
 * of emu_gemm_f64 cannot offer.  ws: at least
 * emu_gemm_f64_rowcol_workspace_bytes (the GEMM workspace plus the levels).
 * Errors as emu_gemm_f64. */
size_t emu_gemm_f64_rowcol_workspace_bytes(int64_t M, int64_t N, int64_t K);
emu_status emu_gemm_f64_rowcol(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda,
                               const double *B, int64_t ldb, double *C, int64_t ldc, int nprod,
                               void *ws, size_t ws_bytes, emu_stream_t stream);

/* emu_split_f64 for a product-sum that reads slices 0 .. nslices-1 only
 * (nslices = d = 3, 4, 5, 6 for nprod = 6, 10, 15, 21): the fused pass forms
 * and writes only those planes, and only their levels are verified.  Planes
 * 0 .. nslices-1 and v_out[0 .. nslices-1] equal emu_split_f64's; planes and
 * levels from nslices on are unspecified (left as they were, or formed
 * literally when a speculative level below nslices failed).  The GEMM entry
 * points split this way.  Errors as emu_split_f64; EMU_ERR_INVALID_ARG also
 * for nslices outside 3 .. 6. */
emu_status emu_split_f64_slices(const double *X, int64_t rows, int64_t cols, int64_t ldx, int transpose,
                                uint16_t *comps, int64_t ldcomp, int nslices, int32_t *v_out, void *ws,
                                size_t ws_bytes, emu_stream_t stream);

/* Workspace bytes for emu_gemm_f32 (mode 32) / emu_gemm_f64 (mode 64):
 * the flag word plus the slice planes of A (M x K) and B (K x N), and in
 * mode 64 the product-sum's FP64 accumulator (8 bytes per element of C,
 * rounded up to 128 x 128 tiles, or to 128 x 256 tiles where that is
 * larger). */
size_t emu_gemm_workspace_bytes(int mode, int64_t M, int64_t N, int64_t K);

/* The split step of a GEMM C = A . B as one call: A (M x K, lda) into
 * row-major planes Acomps [s][M][ldcomp] and B (K x N, ldb) into K-major
 * planes Bcomps [s][N][ldcomp] (ldcomp >= K), exactly as emu_split_f32 /
 * emu_split_f64_slices split each operand (planes and levels identical), in
 * fewer launches, as the GEMM entry points run it (FP32: one launch for
 * both; FP64: the level-0 maxima of both in one launch).  FP64: nslices in 3..6 as for emu_split_f64_slices; vA, vB:
 * device int32[6] receiving the level exponents of A and of B.  ws: at least
 * emu_split_workspace_bytes(mode); one flag word covers both operands.
 * Errors as the single-operand splits. */
emu_status emu_split_f32_pair(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda,
                              const float *B, int64_t ldb, uint16_t *Acomps, uint16_t *Bcomps,
                              int64_t ldcomp, void *ws, size_t ws_bytes, emu_stream_t stream);
emu_status emu_split_f64_pair(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda,
                              const double *B, int64_t ldb, uint16_t *Acomps, uint16_t *Bcomps,
                              int64_t ldcomp, int nslices, int32_t *vA, int32_t *vB, void *ws,
                              size_t ws_bytes, emu_stream_t stream);

/* FP32-mode emulated GEMM, Algorithm 1: C (M x N, ldc) = A (M x K, lda) . B
 * (K x N, ldb), all FP32 row-major.  Splits A and B into the workspace, then
 * runs the tensor-core product-sum: the 6 products of Eq. (fp32six) are
 * accumulated in one FP32 accumulator over all of K (Section 6.3, FP32
 * reconstruction), so C matches the oracle within FP32 reordering error.
 * When the result has too few 128 x 128 tiles to occupy the GPU, K is split
 * in two: each half has its own FP32 accumulator and the two are added into
 * C (cleared first) in L2, one rounding, independent of which half finishes
 * first; FP32 reductions there flush subnormal sums to zero.  C then differs
 * from the one-accumulator result by FP32 rounding only. */
emu_status emu_gemm_f32(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda,
                        const float *B, int64_t ldb, float *C, int64_t ldc, void *ws,
                        size_t ws_bytes, emu_stream_t stream);

/* FP32-mode emulated GEMM, Algorithm 1, with the split of Eq. (fp32split)
 * done inside the product-sum's producer (the streamed-slice variant that
 * Section 6.2 sets aside for the AMX loop order): each CTA splits the FP32
 * tiles of A and B it is about to multiply, so no slice planes are written
 * to or read from memory.  Same arguments, slices, product order and
 * accumulator as emu_gemm_f32, and C is bit-identical to it.  ws: device
 * workspace of at least emu_split_workspace_bytes(32) bytes (the flag word),
 * 16-byte aligned.  Errors and flags as emu_gemm_f32. */
emu_status emu_gemm_f32_fused(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda,
                              const float *B, int64_t ldb, float *C, int64_t ldc, void *ws,
                              size_t ws_bytes, emu_stream_t stream);

/* FP64-mode emulated GEMM, Algorithm 2: C = A . B for FP64 inputs, nprod in
 * {6, 10, 15, 21}.  Products are taken in Algorithm 2's diagonal order; for
 * each, the FP32 component product fl32(A_i B_j) is formed on the tensor
 * cores per K-chunk of 256 (every chunk partial is exact, Section 5.2), the
 * partials are summed exactly, and the total is added once into the FP64
 * result: C <- fl64(C + fl32(A_i B_j)).  C equals the oracle's product-outer
 * order bit for bit.  The FP64 accumulator lives in the workspace; C serves
 * as scratch for low-order words of the exact sums while the kernel runs. */
emu_status emu_gemm_f64(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda,
                        const double *B, int64_t ldb, double *C, int64_t ldc, int nprod,
                        void *ws, size_t ws_bytes, emu_stream_t stream);

/* FP64 mode with merged tail diagonals (an extension of Algorithm 2, not in
 * the paper): the products with i + j < merge_from are taken as in
 * emu_gemm_f64 (diagonal order, each summed exactly over K and added once in
 * FP64); the remaining products of S_d (merge_from <= i + j < d, with d = 3, 4,
 * 5, 6 for nprod = 6, 10, 15, 21) are accumulated together in ONE FP32 sum T
 * over all of K on the tensor cores, and C = fl64(C_head + T) adds it last.
 * The FP32 rounding of T is bounded by (number of tail MMA steps) x 2^-22 x
 * sum over the tail of |A_i||B_j|; in practice, at 4096^3 with nprod = 21
 * and merge_from = 4, e_F is about twice emu_gemm_f64's (still about 100x
 * below nprod = 15).  In exchange one operand stage feeds every tail product.
 * merge_from in {3, 4, 5, 6} and <= d;
 * merge_from = d gives emu_gemm_f64's result bit for bit.  ws: at least
 * emu_gemm_f64_merged_workspace_bytes(M, N, K) bytes (the FP64 GEMM workspace
 * plus an M x N FP32 buffer for T), 16-byte aligned.  Errors and flags as
 * emu_gemm_f64; EMU_ERR_INVALID_ARG also for merge_from out of range. */
size_t emu_gemm_f64_merged_workspace_bytes(int64_t M, int64_t N, int64_t K);
emu_status emu_gemm_f64_merged(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda,
                               const double *B, int64_t ldb, double *C, int64_t ldc, int nprod,
                               int merge_from, void *ws, size_t ws_bytes, emu_stream_t stream);

/* General GEMM (the "more complete BLAS semantics" of Section 9's future
 * work): C (M x N, ldc) <- alpha * op(A) op(B) + beta * C, all row-major.
 * op(X) is X as stored (EMU_OP_N) or its transpose (EMU_OP_T): with opA = N,
 * A is M x K (lda >= K), with opA = T it is stored K x M (lda >= M); with
 * opB = N, B is K x N (ldb >= N), with opB = T it is stored N x K (ldb >= K).
 * The product P = op(A) op(B) is the emulated one of emu_gemm_f32 (Algorithm
 * 1) or emu_gemm_f64 (Algorithm 2, nprod products), from the same kernels:
 * the split writes op(A) and op(B) into the same K-major planes whichever
 * way they are stored.  Then, each operation rounded once in FP32 / FP64
 * (no fused multiply-add): alpha = 1 and beta = 0 gives C = P (written
 * directly, bit-identical to emu_gemm_*); beta = 0 gives C = fl(alpha * P)
 * without reading C; otherwise C = fl(fl(alpha * P) + fl(beta * C)).  K = 0
 * gives P = 0.  ws: device workspace of at least
 * emu_gemm_ex_workspace_bytes (the GEMM workspace plus an M x N product
 * buffer), 16-byte aligned.  Errors as emu_gemm_*; EMU_ERR_INVALID_ARG also
 * for an op other than EMU_OP_N / EMU_OP_T. */
#define EMU_OP_N 0
#define EMU_OP_T 1
size_t emu_gemm_ex_workspace_bytes(int mode, int64_t M, int64_t N, int64_t K);
emu_status emu_gemm_ex_f32(int opA, int opB, int64_t M, int64_t N, int64_t K, float alpha,
                           const float *A, int64_t lda, const float *B, int64_t ldb, float beta,
                           float *C, int64_t ldc, void *ws, size_t ws_bytes, emu_stream_t stream);
emu_status emu_gemm_ex_f64(int opA, int opB, int64_t M, int64_t N, int64_t K, double alpha,
                           const double *A, int64_t lda, const double *B, int64_t ldb, double beta,
                           double *C, int64_t ldc, int nprod, void *ws, size_t ws_bytes,
                           emu_stream_t stream);

/* Workspace bytes for emu_gemm_f32_host (mode 32) / emu_gemm_f64_host (mode
 * 64): the header, the planes of A and B, staging space for the copied
 * inputs (FP32: two row panels of A and two K-panels of B; FP64: A and B
 * whole) and two row panels of C.  0 for negative sizes or another mode. */
size_t emu_gemm_host_workspace_bytes(int mode, int64_t M, int64_t N, int64_t K);

/* The GEMMs of emu_gemm_f32 / emu_gemm_f64 (Algorithms 1 and 2, same kernels,
 * bit-identical results) on operands in HOST memory: A (M x K, lda), B (K x N,
 * ldb) and C (M x N, ldc) are host pointers, row-major; ws is a DEVICE
 * workspace of at least emu_gemm_host_workspace_bytes bytes, 256-byte
 * aligned.  The call enqueues the whole job and returns; C is complete when
 * `stream` reaches the point after the call (synchronise it before reading
 * C).  The host buffers must stay valid and unchanged until then.  Pinned
 * (page-locked) host memory gives full copy speed and an asynchronous call;
 * pageable memory works but the runtime then copies synchronously.
 * Internally the copies, the split and the product-sum are pipelined over
 * panels on streams that the library creates once per device (the current
 * device must be the stream's device): FP32 copies B in K-panels and A in
 * row panels, each split as soon as it lands, and multiplies row panels as
 * their A rows arrive; FP64 copies A and B whole (its split needs the
 * maximum over the whole operand, Eq. (fp64split)) and overlaps B's copy
 * with A's split.  Finished row panels of C are copied back while the next
 * is computed.  Concurrent calls on one device are serialised by the
 * library.  The flag word (emu_read_flags on ws) reports the split and
 * watchdog flags of the call.  Errors: as emu_gemm_f32 / emu_gemm_f64;
 * EMU_ERR_MISALIGNED for a workspace not 256-byte aligned. */
emu_status emu_gemm_f32_host(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda,
                             const float *B, int64_t ldb, float *C, int64_t ldc, void *ws,
                             size_t ws_bytes, emu_stream_t stream);
emu_status emu_gemm_f64_host(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda,
                             const double *B, int64_t ldb, double *C, int64_t ldc, int nprod,
                             void *ws, size_t ws_bytes, emu_stream_t stream);

/* Product-sum alone, from planes already split (A: [3][M][ldcomp],
 * B: [3][N][ldcomp], i.e. split with transpose = 1).  Eq. (fp32six),
 * Section 6.3.  ws: at least emu_split_workspace_bytes(32) (flag word). */
emu_status emu_prodsum_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Acomps,
                           const uint16_t *Bcomps, int64_t ldcomp, float *C, int64_t ldc,
                           void *ws, size_t ws_bytes, emu_stream_t stream);

/* Workspace bytes for emu_prodsum_f32 (mode 32: the flag word) and
 * emu_prodsum_f64 (mode 64: the flag word and the FP64 accumulator of the
 * product-outer sum, 8 bytes per element of C rounded up to 128 x 128
 * tiles, or to 128 x 256 tiles where that is larger).  0 for negative sizes
 * or another mode. */
size_t emu_prodsum_workspace_bytes(int mode, int64_t M, int64_t N);

/* Output tiles of the FP32-mode product-sum for an M x N result
 * (emu_prodsum_f32, and emu_gemm_f32 when it does not split K), unless
 * EMU_F32_TILE (128x256, 128x128 or 128x64) or EMU_F32_PAIR=0 forces a
 * shape: width 256, 128 or 64 columns; height 128 rows, or 256 rows where
 * 256-column tiles run on a pair of SMs (a cluster of two CTAs sharing each
 * MMA); and the number of kernel launches, 1, or 2 when the pair tiles leave
 * the last wave partly empty and its tiles run as 128 x 128 quarters in a
 * second launch.  The paper has no counterpart: every shape gives identical
 * results, and the calls only report which kernels run.  0 for sizes < 1. */
int emu_prodsum_f32_tile_columns(int64_t M, int64_t N);
int emu_prodsum_f32_tile_rows(int64_t M, int64_t N);
int emu_prodsum_f32_launches(int64_t M, int64_t N);

/* Output-tile shape that the FP64-mode product-sum picks for an M x N
 * result, unless EMU_F64_TILE (128x128, 128x256 or 256x256) forces one:
 * width 128 or 256 columns; height 128 rows, or 256 rows where a 256-column
 * tile runs on a pair of SMs (a cluster of two CTAs sharing each MMA); and
 * the number of kernel launches (2 when the last, partial wave of 256-column
 * tiles runs as 128 x 128 tiles in a second launch).  The paper has no
 * counterpart: every shape gives identical results, and the calls only
 * report which kernels run.  0 for sizes < 1. */
int emu_prodsum_f64_tile_columns(int64_t M, int64_t N);
int emu_prodsum_f64_tile_rows(int64_t M, int64_t N);
int emu_prodsum_f64_launches(int64_t M, int64_t N);

/* Product-sum alone for FP64 mode, Eq. (fp64reconstruction), summed as in
 * emu_gemm_f64: A planes [6][M][ldcomp], B planes [6][N][ldcomp]; nprod in
 * {6, 10, 15, 21}.  vA, vB: the device arrays of level exponents v^(0..5)
 * that emu_split_f64 wrote for A and for B (its v_out).  They give each
 * product's unit, 2^(vA_i + vB_j - 16), which lets the kernel add a chunk
 * partial with one FP32 addition while the running sum stays below 2^24
 * units (provably exact); both may be NULL, and then every addition is done
 * as an error-free TwoSum (same result, slower).  ws: at least
 * emu_prodsum_workspace_bytes(64, M, N) (flag word and FP64 accumulator). */
emu_status emu_prodsum_f64(int64_t M, int64_t N, int64_t K, const uint16_t *Acomps,
                           const uint16_t *Bcomps, int64_t ldcomp, const int32_t *vA,
                           const int32_t *vB, int nprod, double *C, int64_t ldc, void *ws,
                           size_t ws_bytes, emu_stream_t stream);

/* FP64-mode emulated GEMM that allocates nothing and takes no workspace.
 * The paper has no counterpart: this entry point exists for callers that
 * cannot allocate device memory -- plugins inside host programs that own the
 * whole device memory budget and forbid allocation calls after start-up, or
 * latency-critical paths that cannot accept the implicit synchronisation of
 * cudaMalloc.  It computes exactly what emu_gemm_f64 computes (same kernels,
 * same results), with its scratch (flag word, level maxima, BF16 planes,
 * FP64 accumulator) in a static device array of EMU_NOALLOC_SCRATCH_BYTES
 * that every GPU loading the library holds until the library is unloaded.
 * Limit: 512 + 12 * (M + N) * roundup(K, 8) bytes of planes (256-byte
 * rounding per operand) plus 8 * roundup(M, 128) * roundup(N, 256) bytes of
 * accumulator must fit the array, e.g. M = N = K = 1024; larger problems
 * return EMU_ERR_UNSUPPORTED before any work is enqueued.
 * flags_out: device pointer receiving the EMU_FLAG_* word of this call
 * (may be NULL).  Every call looks up the array's device address in the
 * current context (a lookup that allocates nothing, so it stays right after
 * cudaDeviceReset re-creates the context); the first call on a device may
 * load the library's device code, so make that first call before any stream
 * capture.  All calls on a device share the array: calls whose work may
 * overlap on the GPU (different streams or host threads without ordering)
 * race and must be serialised by the caller. */
#define EMU_NOALLOC_SCRATCH_BYTES (40u << 20)
emu_status emu_gemm_f64_noalloc(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda,
                                const double *B, int64_t ldb, double *C, int64_t ldc, int nprod,
                                uint32_t *flags_out, emu_stream_t stream);

/* Copies the flag word of the last call that used `ws` to *host_flags after
 * synchronising `stream`.  ws: device workspace; host_flags: host pointer. */
emu_status emu_read_flags(const void *ws, uint32_t *host_flags, emu_stream_t stream);

/* Watchdog self-test: launches one kernel that waits, with the same bounded
 * wait the GEMM kernels use, on a barrier that nothing completes; after
 * timeout_us microseconds it gives up, sets EMU_FLAG_TIMEOUT in the
 * workspace flag word and returns, leaving the context usable.
 * timeout_us in [1, 10^6]. */
emu_status emu_selftest_timeout(void *ws, size_t ws_bytes, uint32_t timeout_us,
                                emu_stream_t stream);

/* Static description of an emu_status value. */
const char *emu_status_string(emu_status status);

#ifdef __cplusplus
}
#endif
#endif /* EMU_H */
