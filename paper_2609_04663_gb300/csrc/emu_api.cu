// C-ABI of the emulation library (declared in include/emu.h): argument
// checks, workspace layout and the launch sequence of each entry point.
#include "launchers.cuh"

namespace emu {

// Watchdog self-test: one bounded wait on a barrier that nothing completes.
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

using namespace emu;

namespace {

constexpr int64_t kMaxDim = (int64_t)1 << 31;      // kernels index with 32-bit coordinates

int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

// K-major plane leading dimension used inside the GEMM workspace: TMA needs
// row strides that are multiples of 16 bytes.
int64_t gemm_ldk(int64_t K) { return round_up(K < 1 ? 1 : K, 8); }

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

emu_status cuda_status(cudaError_t e) { return e == cudaSuccess ? EMU_OK : EMU_ERR_CUDA; }

emu_status check_planes(const void *Ap, const void *Bp, int64_t ldcomp, int64_t K)
{
    if (!Ap || !Bp || ldcomp < K || ldcomp < 1) return EMU_ERR_INVALID_ARG;
    if ((ldcomp & 7) != 0 || !aligned16(Ap) || !aligned16(Bp)) return EMU_ERR_MISALIGNED;
    return EMU_OK;
}

emu_status check_gemm_dims(int64_t M, int64_t N, int64_t K, int64_t lda, int64_t ldb, int64_t ldc)
{
    if (M < 0 || N < 0 || K < 0) return EMU_ERR_INVALID_ARG;
    if (lda < (K > 0 ? K : 1) || ldb < (N > 0 ? N : 1) || ldc < (N > 0 ? N : 1)) return EMU_ERR_INVALID_ARG;
    if (M >= kMaxDim || N >= kMaxDim || K >= kMaxDim) return EMU_ERR_UNSUPPORTED;
    return EMU_OK;
}

// C = 0 for K = 0 (rows of N elements with pitch ldc).
template <typename T>
emu_status zero_c(T *C, int64_t M, int64_t N, int64_t ldc, cudaStream_t st)
{
    return cuda_status(cudaMemset2DAsync(C, (size_t)ldc * sizeof(T), 0, (size_t)N * sizeof(T), (size_t)M, st));
}

// GEMM workspace: header, A planes [s][M][ldk], B planes [s][N][ldk], and in
// FP64 mode the product-sum's FP64 accumulator.
size_t gemm_ws_bytes(int s, int64_t M, int64_t N, int64_t K)
{
    const int64_t ldk = gemm_ldk(K);
    return kWsHeaderBytes + (size_t)round_up((int64_t)s * M * ldk * 2, 256) +
           (size_t)round_up((int64_t)s * N * ldk * 2, 256) + (s == 6 ? f64_acc_bytes(M, N) : 0);
}

// The FP64 accumulator that follows the planes of a GEMM workspace.
double *gemm_acc(void *ws, int64_t M, int64_t N, int64_t K)
{
    const int64_t ldk = gemm_ldk(K);
    return reinterpret_cast<double *>(static_cast<char *>(ws) + kWsHeaderBytes + round_up(6 * M * ldk * 2, 256) +
                                      round_up(6 * N * ldk * 2, 256));
}

}  // namespace

extern "C" {

size_t emu_split_workspace_bytes(int mode)
{
    (void)mode;
    return kWsHeaderBytes;
}

emu_status emu_split_f32(const float *X, int64_t rows, int64_t cols, int64_t ldx, int transpose, uint16_t *comps,
                         int64_t ldcomp, void *ws, size_t ws_bytes, emu_stream_t stream)
{
    if (rows < 0 || cols < 0 || ldx < (cols > 0 ? cols : 1) || !ws) return EMU_ERR_INVALID_ARG;
    if (ldcomp < (transpose ? rows : cols) || ldcomp < 1) return EMU_ERR_INVALID_ARG;
    if (rows > 0 && cols > 0 && (!X || !comps)) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < kWsHeaderBytes) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e == cudaSuccess) e = launch_split_f32(X, rows, cols, ldx, transpose != 0, comps, ldcomp, h, st);
    return cuda_status(e);
}

emu_status emu_split_f64(const double *X, int64_t rows, int64_t cols, int64_t ldx, int transpose, uint16_t *comps,
                         int64_t ldcomp, int32_t *v_out, void *ws, size_t ws_bytes, emu_stream_t stream)
{
    if (rows < 0 || cols < 0 || ldx < (cols > 0 ? cols : 1) || !ws || !v_out) return EMU_ERR_INVALID_ARG;
    if (ldcomp < (transpose ? rows : cols) || ldcomp < 1) return EMU_ERR_INVALID_ARG;
    if (rows > 0 && cols > 0 && (!X || !comps)) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < kWsHeaderBytes) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e == cudaSuccess) e = launch_split_f64(X, rows, cols, ldx, transpose != 0, comps, ldcomp, v_out, h, 0, st);
    return cuda_status(e);
}

emu_status emu_split_f64_slices(const double *X, int64_t rows, int64_t cols, int64_t ldx, int transpose,
                                uint16_t *comps, int64_t ldcomp, int nslices, int32_t *v_out, void *ws,
                                size_t ws_bytes, emu_stream_t stream)
{
    if (nslices < 3 || nslices > 6) return EMU_ERR_INVALID_ARG;
    if (rows < 0 || cols < 0 || ldx < (cols > 0 ? cols : 1) || !ws || !v_out) return EMU_ERR_INVALID_ARG;
    if (ldcomp < (transpose ? rows : cols) || ldcomp < 1) return EMU_ERR_INVALID_ARG;
    if (rows > 0 && cols > 0 && (!X || !comps)) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < kWsHeaderBytes) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e == cudaSuccess)
        e = launch_split_f64(X, rows, cols, ldx, transpose != 0, comps, ldcomp, v_out, h, 0, st, nslices);
    return cuda_status(e);
}

emu_status emu_split_f32_pair(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda, const float *B,
                              int64_t ldb, uint16_t *Acomps, uint16_t *Bcomps, int64_t ldcomp, void *ws,
                              size_t ws_bytes, emu_stream_t stream)
{
    emu_status s = check_gemm_dims(M, N, K, lda, ldb, N > 0 ? N : 1);
    if (s != EMU_OK) return s;
    if (!ws || ldcomp < (K > 0 ? K : 1)) return EMU_ERR_INVALID_ARG;
    if (M > 0 && N > 0 && K > 0 && (!A || !B || !Acomps || !Bcomps)) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < kWsHeaderBytes) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e == cudaSuccess && M > 0 && N > 0 && K > 0)
        e = launch_split_f32_gemm(A, M, K, lda, B, N, ldb, Acomps, Bcomps, ldcomp, h, nullptr, 0, st);
    return cuda_status(e);
}

emu_status emu_split_f64_pair(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda, const double *B,
                              int64_t ldb, uint16_t *Acomps, uint16_t *Bcomps, int64_t ldcomp, int nslices,
                              int32_t *vA, int32_t *vB, void *ws, size_t ws_bytes, emu_stream_t stream)
{
    emu_status s = check_gemm_dims(M, N, K, lda, ldb, N > 0 ? N : 1);
    if (s != EMU_OK) return s;
    if (nslices < 3 || nslices > 6 || !ws || !vA || !vB || ldcomp < (K > 0 ? K : 1)) return EMU_ERR_INVALID_ARG;
    if (M > 0 && N > 0 && K > 0 && (!A || !B || !Acomps || !Bcomps)) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < kWsHeaderBytes) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e == cudaSuccess)
        e = launch_split_f64_gemm(A, M, K, lda, B, N, ldb, Acomps, Bcomps, ldcomp, vA, vB, h, st, nslices);
    return cuda_status(e);
}

size_t emu_gemm_workspace_bytes(int mode, int64_t M, int64_t N, int64_t K)
{
    if (M < 0 || N < 0 || K < 0) return 0;
    return gemm_ws_bytes(mode == 64 ? 6 : 3, M, N, K);
}

emu_status emu_gemm_f32(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda, const float *B, int64_t ldb,
                        float *C, int64_t ldc, void *ws, size_t ws_bytes, emu_stream_t stream)
{
    emu_status s = check_gemm_dims(M, N, K, lda, ldb, ldc);
    if (s != EMU_OK) return s;
    if (!ws || (M > 0 && N > 0 && (!C || (K > 0 && (!A || !B))))) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < gemm_ws_bytes(3, M, N, K)) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e != cudaSuccess) return EMU_ERR_CUDA;
    if (M == 0 || N == 0) return EMU_OK;
    if (K == 0) return zero_c(C, M, N, ldc, st);
    const int64_t ldk = gemm_ldk(K);
    uint16_t *Ap = reinterpret_cast<uint16_t *>(static_cast<char *>(ws) + kWsHeaderBytes);
    uint16_t *Bp = reinterpret_cast<uint16_t *>(reinterpret_cast<char *>(Ap) + round_up(3 * M * ldk * 2, 256));
    // both splits in one launch; when the product-sum will split K in two
    // (few output tiles), the same launch clears C for the halves to add into
    const bool split_k = f32_split_parts(M, N, K) > 1;
    e = launch_split_f32_gemm(A, M, K, lda, B, N, ldb, Ap, Bp, ldk, h, split_k ? C : nullptr, ldc, st);
    if (e == cudaSuccess) e = launch_prodsum_f32(M, N, K, Ap, Bp, ldk, C, ldc, &h->flags, st, 0, 0, split_k);
    return cuda_status(e);
}

emu_status emu_gemm_f32_fused(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda, const float *B,
                              int64_t ldb, float *C, int64_t ldc, void *ws, size_t ws_bytes, emu_stream_t stream)
{
    emu_status s = check_gemm_dims(M, N, K, lda, ldb, ldc);
    if (s != EMU_OK) return s;
    if (!ws || (M > 0 && N > 0 && (!C || (K > 0 && (!A || !B))))) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < kWsHeaderBytes) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e != cudaSuccess) return EMU_ERR_CUDA;
    if (M == 0 || N == 0) return EMU_OK;
    if (K == 0) return zero_c(C, M, N, ldc, st);
    return cuda_status(launch_gemm_f32_fused(M, N, K, A, lda, B, ldb, C, ldc, &h->flags, st));
}

size_t emu_gemm_f64_merged_workspace_bytes(int64_t M, int64_t N, int64_t K)
{
    if (M < 0 || N < 0 || K < 0) return 0;
    return gemm_ws_bytes(6, M, N, K) + (size_t)round_up(M * N * 4, 256);
}

emu_status emu_gemm_f64_merged(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda, const double *B,
                               int64_t ldb, double *C, int64_t ldc, int nprod, int merge_from, void *ws,
                               size_t ws_bytes, emu_stream_t stream)
{
    emu_status s = check_gemm_dims(M, N, K, lda, ldb, ldc);
    if (s != EMU_OK) return s;
    const int d = f64_diagonals(nprod);
    if (d == 0 || merge_from < 3 || merge_from > d) return EMU_ERR_INVALID_ARG;
    if (!ws || (M > 0 && N > 0 && (!C || (K > 0 && (!A || !B))))) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < emu_gemm_f64_merged_workspace_bytes(M, N, K)) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e != cudaSuccess) return EMU_ERR_CUDA;
    if (M == 0 || N == 0) return EMU_OK;
    if (K == 0) return zero_c(C, M, N, ldc, st);
    const int64_t ldk = gemm_ldk(K);
    uint16_t *Ap = reinterpret_cast<uint16_t *>(static_cast<char *>(ws) + kWsHeaderBytes);
    uint16_t *Bp = reinterpret_cast<uint16_t *>(reinterpret_cast<char *>(Ap) + round_up(6 * M * ldk * 2, 256));
    float *T = merge_from < d ? reinterpret_cast<float *>(static_cast<char *>(ws) + gemm_ws_bytes(6, M, N, K)) : nullptr;
    // the product-sum uses slices 0 .. d-1 only
    const int nlev = f64_diagonals(nprod);
    e = launch_split_f64_gemm(A, M, K, lda, B, N, ldb, Ap, Bp, ldk, h->vout[0], h->vout[1], h, st, nlev);
    if (e == cudaSuccess && T) e = launch_prodsum_tail(M, N, K, Ap, Bp, ldk, merge_from, d, T, N, &h->flags, st);
    if (e == cudaSuccess)
        e = launch_prodsum_f64(M, N, K, Ap, Bp, ldk, h->vout[0], h->vout[1], merge_from * (merge_from + 1) / 2, C,
                               ldc, gemm_acc(ws, M, N, K), &h->flags, st, 0, false, T, N);
    return cuda_status(e);
}

emu_status emu_gemm_f64(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda, const double *B,
                        int64_t ldb, double *C, int64_t ldc, int nprod, void *ws, size_t ws_bytes,
                        emu_stream_t stream)
{
    emu_status s = check_gemm_dims(M, N, K, lda, ldb, ldc);
    if (s != EMU_OK) return s;
    if (nprod != 6 && nprod != 10 && nprod != 15 && nprod != 21) return EMU_ERR_INVALID_ARG;
    if (!ws || (M > 0 && N > 0 && (!C || (K > 0 && (!A || !B))))) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < gemm_ws_bytes(6, M, N, K)) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e != cudaSuccess) return EMU_ERR_CUDA;
    if (M == 0 || N == 0) return EMU_OK;
    if (K == 0) return zero_c(C, M, N, ldc, st);
    const int64_t ldk = gemm_ldk(K);
    uint16_t *Ap = reinterpret_cast<uint16_t *>(static_cast<char *>(ws) + kWsHeaderBytes);
    uint16_t *Bp = reinterpret_cast<uint16_t *>(reinterpret_cast<char *>(Ap) + round_up(6 * M * ldk * 2, 256));
    // the product-sum uses slices 0 .. d-1 only
    const int nlev = f64_diagonals(nprod);
    e = launch_split_f64_gemm(A, M, K, lda, B, N, ldb, Ap, Bp, ldk, h->vout[0], h->vout[1], h, st, nlev);
    if (e == cudaSuccess)
        e = launch_prodsum_f64(M, N, K, Ap, Bp, ldk, h->vout[0], h->vout[1], nprod, C, ldc, gemm_acc(ws, M, N, K),
                               &h->flags, st);
    return cuda_status(e);
}

int emu_prodsum_f32_tile_columns(int64_t M, int64_t N)
{
    if (M < 1 || N < 1) return 0;
    return f32_tile_columns(M, N);
}

int emu_prodsum_f32_tile_rows(int64_t M, int64_t N)
{
    if (M < 1 || N < 1) return 0;
    return f32_tile_rows(M, N);
}

int emu_prodsum_f32_launches(int64_t M, int64_t N)
{
    if (M < 1 || N < 1) return 0;
    return f32_prodsum_launches(M, N);
}

int emu_prodsum_f64_tile_columns(int64_t M, int64_t N)
{
    if (M < 1 || N < 1) return 0;
    return f64_tile_columns(M, N);
}

int emu_prodsum_f64_tile_rows(int64_t M, int64_t N)
{
    if (M < 1 || N < 1) return 0;
    return f64_plan(M, N).rows;
}

int emu_prodsum_f64_launches(int64_t M, int64_t N)
{
    if (M < 1 || N < 1) return 0;
    return f64_plan(M, N).launches;
}

size_t emu_prodsum_workspace_bytes(int mode, int64_t M, int64_t N)
{
    if (M < 0 || N < 0 || (mode != 32 && mode != 64)) return 0;
    return kWsHeaderBytes + (mode == 64 ? f64_acc_bytes(M, N) : 0);
}

size_t emu_gemm_ex_workspace_bytes(int mode, int64_t M, int64_t N, int64_t K)
{
    if (M < 0 || N < 0 || K < 0 || (mode != 32 && mode != 64)) return 0;
    return gemm_ws_bytes(mode == 64 ? 6 : 3, M, N, K) + (size_t)round_up(M * N * (mode == 64 ? 8 : 4), 256);
}

}  // extern "C"

namespace {

// Shared body of the general GEMMs: validation, the splits of op(A) and
// op(B) into K-major planes (the split's transpose flag absorbs op), the
// product-sum into C (alpha = 1, beta = 0) or into the workspace product
// buffer followed by the epilogue.
template <typename T>
emu_status gemm_ex(int opA, int opB, int64_t M, int64_t N, int64_t K, T alpha, const T *A, int64_t lda, const T *B,
                   int64_t ldb, T beta, T *C, int64_t ldc, int nprod, void *ws, size_t ws_bytes, cudaStream_t st)
{
    constexpr bool f64 = sizeof(T) == 8;
    constexpr int S = f64 ? 6 : 3;
    if ((opA != EMU_OP_N && opA != EMU_OP_T) || (opB != EMU_OP_N && opB != EMU_OP_T)) return EMU_ERR_INVALID_ARG;
    if (M < 0 || N < 0 || K < 0 || !ws) return EMU_ERR_INVALID_ARG;
    const int64_t a_cols = opA == EMU_OP_N ? K : M, b_cols = opB == EMU_OP_N ? N : K;
    if (lda < (a_cols > 0 ? a_cols : 1) || ldb < (b_cols > 0 ? b_cols : 1) || ldc < (N > 0 ? N : 1))
        return EMU_ERR_INVALID_ARG;
    if (M >= kMaxDim || N >= kMaxDim || K >= kMaxDim) return EMU_ERR_UNSUPPORTED;
    if (f64 && nprod != 6 && nprod != 10 && nprod != 15 && nprod != 21) return EMU_ERR_INVALID_ARG;
    if (M > 0 && N > 0 && (!C || (K > 0 && (!A || !B)))) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < emu_gemm_ex_workspace_bytes(f64 ? 64 : 32, M, N, K)) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e != cudaSuccess) return EMU_ERR_CUDA;
    if (M == 0 || N == 0) return EMU_OK;
    const int64_t ldk = gemm_ldk(K);
    char *w = static_cast<char *>(ws);
    uint16_t *Ap = reinterpret_cast<uint16_t *>(w + kWsHeaderBytes);
    uint16_t *Bp = reinterpret_cast<uint16_t *>(reinterpret_cast<char *>(Ap) + round_up(S * M * ldk * 2, 256));
    T *P = reinterpret_cast<T *>(reinterpret_cast<char *>(Bp) + round_up(S * N * ldk * 2, 256) +
                                 (f64 ? f64_acc_bytes(M, N) : 0));
    const bool direct = (alpha == T(1) && beta == T(0));
    T *out = direct ? C : P;
    const int64_t ldo = direct ? ldc : N;
    if (K == 0) {
        e = cudaMemset2DAsync(out, (size_t)ldo * sizeof(T), 0, (size_t)N * sizeof(T), (size_t)M, st);
    } else {
        // op(A) -> planes [S][M][ldk]; op(B) -> planes [S][N][ldk]
        const bool ta = opA == EMU_OP_T, tb = opB == EMU_OP_N;
        const int64_t ar = ta ? K : M, ac = ta ? M : K, br = tb ? K : N, bc = tb ? N : K;
        if constexpr (f64) {
            const int nlev = f64_diagonals(nprod);   // slices the product-sum uses
            e = launch_split_f64(A, ar, ac, lda, ta, Ap, ldk, h->vout[0], h, 0, st, nlev);
            if (e == cudaSuccess) e = launch_split_f64(B, br, bc, ldb, tb, Bp, ldk, h->vout[1], h, 1, st, nlev);
            if (e == cudaSuccess)
                e = launch_prodsum_f64(M, N, K, Ap, Bp, ldk, h->vout[0], h->vout[1], nprod, out, ldo,
                                       gemm_acc(ws, M, N, K), &h->flags, st);
        } else {
            e = launch_split_f32(A, ar, ac, lda, ta, Ap, ldk, h, st);
            if (e == cudaSuccess) e = launch_split_f32(B, br, bc, ldb, tb, Bp, ldk, h, st);
            if (e == cudaSuccess) e = launch_prodsum_f32(M, N, K, Ap, Bp, ldk, out, ldo, &h->flags, st);
        }
    }
    if (e == cudaSuccess && !direct) {
        if constexpr (f64) e = launch_axpby_f64(P, N, C, ldc, M, N, alpha, beta, st);
        else e = launch_axpby_f32(P, N, C, ldc, M, N, alpha, beta, st);
    }
    return cuda_status(e);
}

}  // namespace

extern "C" {

emu_status emu_gemm_ex_f32(int opA, int opB, int64_t M, int64_t N, int64_t K, float alpha, const float *A, int64_t lda,
                           const float *B, int64_t ldb, float beta, float *C, int64_t ldc, void *ws, size_t ws_bytes,
                           emu_stream_t stream)
{
    return gemm_ex<float>(opA, opB, M, N, K, alpha, A, lda, B, ldb, beta, C, ldc, 0, ws, ws_bytes,
                          reinterpret_cast<cudaStream_t>(stream));
}

emu_status emu_gemm_ex_f64(int opA, int opB, int64_t M, int64_t N, int64_t K, double alpha, const double *A,
                           int64_t lda, const double *B, int64_t ldb, double beta, double *C, int64_t ldc, int nprod,
                           void *ws, size_t ws_bytes, emu_stream_t stream)
{
    return gemm_ex<double>(opA, opB, M, N, K, alpha, A, lda, B, ldb, beta, C, ldc, nprod, ws, ws_bytes,
                           reinterpret_cast<cudaStream_t>(stream));
}

size_t emu_split_f64_rowcol_workspace_bytes(int64_t plane_rows)
{
    if (plane_rows < 0) return 0;
    return kWsHeaderBytes + (size_t)round_up((int64_t)rc_scratch_bytes(plane_rows), 256);
}

emu_status emu_split_f64_rowcol(const double *X, int64_t rows, int64_t cols, int64_t ldx, int transpose,
                                uint16_t *comps, int64_t ldcomp, int32_t *v_out, void *ws, size_t ws_bytes,
                                emu_stream_t stream)
{
    if (rows < 0 || cols < 0 || ldx < (cols > 0 ? cols : 1) || !ws || !v_out) return EMU_ERR_INVALID_ARG;
    const int64_t prow = transpose ? cols : rows;
    if (ldcomp < (transpose ? rows : cols) || ldcomp < 1) return EMU_ERR_INVALID_ARG;
    if (rows > 0 && cols > 0 && (!X || !comps)) return EMU_ERR_INVALID_ARG;
    if (rows >= kMaxDim || cols >= kMaxDim) return EMU_ERR_UNSUPPORTED;
    if (ws_bytes < emu_split_f64_rowcol_workspace_bytes(prow)) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    void *scratch = static_cast<char *>(ws) + kWsHeaderBytes;
    if (e == cudaSuccess) e = launch_split_f64_rc(X, rows, cols, ldx, transpose != 0, comps, ldcomp, v_out, scratch, h, 0, st);
    return cuda_status(e);
}

size_t emu_gemm_f64_rowcol_workspace_bytes(int64_t M, int64_t N, int64_t K)
{
    if (M < 0 || N < 0 || K < 0) return 0;
    return gemm_ws_bytes(6, M, N, K) + (size_t)round_up(6 * (M + N) * 4, 256) +
           (size_t)round_up((int64_t)rc_scratch_bytes(M > N ? M : N), 256);
}

emu_status emu_gemm_f64_rowcol(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda, const double *B,
                               int64_t ldb, double *C, int64_t ldc, int nprod, void *ws, size_t ws_bytes,
                               emu_stream_t stream)
{
    emu_status s = check_gemm_dims(M, N, K, lda, ldb, ldc);
    if (s != EMU_OK) return s;
    if (nprod != 6 && nprod != 10 && nprod != 15 && nprod != 21) return EMU_ERR_INVALID_ARG;
    if (!ws || (M > 0 && N > 0 && (!C || (K > 0 && (!A || !B))))) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < emu_gemm_f64_rowcol_workspace_bytes(M, N, K)) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    if (e != cudaSuccess) return EMU_ERR_CUDA;
    if (M == 0 || N == 0) return EMU_OK;
    if (K == 0) return zero_c(C, M, N, ldc, st);
    const int64_t ldk = gemm_ldk(K);
    char *w = static_cast<char *>(ws);
    uint16_t *Ap = reinterpret_cast<uint16_t *>(w + kWsHeaderBytes);
    uint16_t *Bp = reinterpret_cast<uint16_t *>(reinterpret_cast<char *>(Ap) + round_up(6 * M * ldk * 2, 256));
    char *tail = w + gemm_ws_bytes(6, M, N, K);                    // after the planes and the accumulator
    int32_t *vA = reinterpret_cast<int32_t *>(tail);
    int32_t *vB = vA + 6 * M;
    void *scratch = tail + round_up(6 * (M + N) * 4, 256);
    // A by rows (plane rows = rows of A), B by columns (plane rows = columns of B);
    // the two splits run in order on the stream and share the scratch
    e = launch_split_f64_rc(A, M, K, lda, false, Ap, ldk, vA, scratch, h, 0, st);
    if (e == cudaSuccess) e = launch_split_f64_rc(B, K, N, ldb, true, Bp, ldk, vB, scratch, h, 1, st);
    if (e == cudaSuccess)
        e = launch_prodsum_f64(M, N, K, Ap, Bp, ldk, vA, vB, nprod, C, ldc, gemm_acc(ws, M, N, K), &h->flags, st, 0,
                               true);
    return cuda_status(e);
}

emu_status emu_prodsum_f32(int64_t M, int64_t N, int64_t K, const uint16_t *Acomps, const uint16_t *Bcomps,
                           int64_t ldcomp, float *C, int64_t ldc, void *ws, size_t ws_bytes, emu_stream_t stream)
{
    if (M < 0 || N < 0 || K < 0 || ldc < (N > 0 ? N : 1) || !ws) return EMU_ERR_INVALID_ARG;
    if (M >= kMaxDim || N >= kMaxDim || K >= kMaxDim) return EMU_ERR_UNSUPPORTED;
    if (ws_bytes < kWsHeaderBytes) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    if (cudaMemsetAsync(&h->flags, 0, sizeof(uint32_t), st) != cudaSuccess) return EMU_ERR_CUDA;
    if (M == 0 || N == 0) return EMU_OK;
    if (!C) return EMU_ERR_INVALID_ARG;
    if (K == 0) return zero_c(C, M, N, ldc, st);
    emu_status s = check_planes(Acomps, Bcomps, ldcomp, K);
    if (s != EMU_OK) return s;
    return cuda_status(launch_prodsum_f32(M, N, K, Acomps, Bcomps, ldcomp, C, ldc, &h->flags, st));
}

emu_status emu_prodsum_f64(int64_t M, int64_t N, int64_t K, const uint16_t *Acomps, const uint16_t *Bcomps,
                           int64_t ldcomp, const int32_t *vA, const int32_t *vB, int nprod, double *C,
                           int64_t ldc, void *ws, size_t ws_bytes, emu_stream_t stream)
{
    if (M < 0 || N < 0 || K < 0 || ldc < (N > 0 ? N : 1) || !ws) return EMU_ERR_INVALID_ARG;
    if (nprod != 6 && nprod != 10 && nprod != 15 && nprod != 21) return EMU_ERR_INVALID_ARG;
    if (M >= kMaxDim || N >= kMaxDim || K >= kMaxDim) return EMU_ERR_UNSUPPORTED;
    if (ws_bytes < emu_prodsum_workspace_bytes(64, M, N)) return EMU_ERR_WORKSPACE_TOO_SMALL;
    if (!aligned16(ws)) return EMU_ERR_MISALIGNED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    if (cudaMemsetAsync(&h->flags, 0, sizeof(uint32_t), st) != cudaSuccess) return EMU_ERR_CUDA;
    if (M == 0 || N == 0) return EMU_OK;
    if (!C) return EMU_ERR_INVALID_ARG;
    if (K == 0) return zero_c(C, M, N, ldc, st);
    emu_status s = check_planes(Acomps, Bcomps, ldcomp, K);
    if (s != EMU_OK) return s;
    if ((vA == nullptr) != (vB == nullptr)) return EMU_ERR_INVALID_ARG;
    double *acc = reinterpret_cast<double *>(static_cast<char *>(ws) + kWsHeaderBytes);
    return cuda_status(launch_prodsum_f64(M, N, K, Acomps, Bcomps, ldcomp, vA, vB, nprod, C, ldc, acc, &h->flags, st));
}

emu_status emu_read_flags(const void *ws, uint32_t *host_flags, emu_stream_t stream)
{
    if (!ws || !host_flags) return EMU_ERR_INVALID_ARG;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(host_flags, &static_cast<const WsHeader *>(ws)->flags, sizeof(uint32_t),
                                    cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    return cuda_status(e);
}

emu_status emu_selftest_timeout(void *ws, size_t ws_bytes, uint32_t timeout_us, emu_stream_t stream)
{
    if (!ws || timeout_us < 1 || timeout_us > 1000000) return EMU_ERR_INVALID_ARG;
    if (ws_bytes < kWsHeaderBytes) return EMU_ERR_WORKSPACE_TOO_SMALL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    cudaError_t e = cudaMemsetAsync(&h->flags, 0, sizeof(uint32_t), st);
    if (e == cudaSuccess) e = launch_timeout_selftest(&h->flags, timeout_us, st);
    return cuda_status(e);
}

const char *emu_status_string(emu_status status)
{
    switch (status) {
    case EMU_OK: return "ok";
    case EMU_ERR_INVALID_ARG: return "invalid argument";
    case EMU_ERR_MISALIGNED: return "misaligned pointer or leading dimension";
    case EMU_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case EMU_ERR_CUDA: return "CUDA error";
    case EMU_ERR_UNSUPPORTED: return "unsupported size";
    }
    return "unknown status";
}

}  // extern "C"
