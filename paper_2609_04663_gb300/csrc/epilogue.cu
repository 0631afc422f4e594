// Epilogue of the general GEMM entry points (emu_gemm_ex_f32 / _f64):
// C <- fl(fl(alpha * P) + fl(beta * C)), or C <- fl(alpha * P) when beta = 0
// (C is then not read), elementwise over M x N, with P the emulated product
// op(A) op(B).  Each operation rounds once in the output format (no fused
// multiply-add), which is the definition the oracle follows.  HBM-bound:
// 12 (FP32) / 24 (FP64) bytes per element with beta != 0.
#include "launchers.cuh"

namespace emu {

namespace {

template <typename T> struct Arith;
template <> struct Arith<float> {
    static __device__ __forceinline__ float mul(float a, float b) { return __fmul_rn(a, b); }
    static __device__ __forceinline__ float add(float a, float b) { return __fadd_rn(a, b); }
};
template <> struct Arith<double> {
    static __device__ __forceinline__ double mul(double a, double b) { return __dmul_rn(a, b); }
    static __device__ __forceinline__ double add(double a, double b) { return __dadd_rn(a, b); }
};

template <typename T, bool READ_C>
__global__ void __launch_bounds__(256)
axpby_kernel(const T *__restrict__ P, int64_t ldp, T *__restrict__ C, int64_t ldc, int64_t M, int64_t N, T alpha,
             T beta)
{
    const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= N) return;
    for (int64_t i = blockIdx.y; i < M; i += gridDim.y) {
        const T ap = Arith<T>::mul(alpha, P[i * ldp + j]);
        C[i * ldc + j] = READ_C ? Arith<T>::add(ap, Arith<T>::mul(beta, C[i * ldc + j])) : ap;
    }
}

template <typename T>
cudaError_t launch_axpby(const T *P, int64_t ldp, T *C, int64_t ldc, int64_t M, int64_t N, T alpha, T beta,
                         cudaStream_t st)
{
    if (M == 0 || N == 0) return cudaSuccess;
    const int64_t bx = (N + 255) / 256;
    const int64_t want = (152 * 16 + bx - 1) / bx;
    const int64_t by = M < want ? M : (want < 65535 ? want : 65535);
    const dim3 grid((unsigned)bx, (unsigned)by);
    if (beta == T(0))
        axpby_kernel<T, false><<<grid, 256, 0, st>>>(P, ldp, C, ldc, M, N, alpha, beta);
    else
        axpby_kernel<T, true><<<grid, 256, 0, st>>>(P, ldp, C, ldc, M, N, alpha, beta);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_axpby_f32(const float *P, int64_t ldp, float *C, int64_t ldc, int64_t M, int64_t N, float alpha,
                             float beta, cudaStream_t st)
{
    return launch_axpby<float>(P, ldp, C, ldc, M, N, alpha, beta, st);
}

cudaError_t launch_axpby_f64(const double *P, int64_t ldp, double *C, int64_t ldc, int64_t M, int64_t N,
                             double alpha, double beta, cudaStream_t st)
{
    return launch_axpby<double>(P, ldp, C, ldc, M, N, alpha, beta, st);
}

}  // namespace emu
