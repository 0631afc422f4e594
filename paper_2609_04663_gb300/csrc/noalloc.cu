// FP64-mode GEMM for callers that cannot allocate device memory.
//
// Some host programs own the whole device memory budget and forbid further
// allocation calls once they are running (plugins inside a larger
// application, processes that carve all of HBM into their own pool up front),
// and some latency-critical paths cannot accept the implicit device
// synchronisation a cudaMalloc may cause.  Such callers can still pass their
// inputs and outputs, but not a workspace.  emu_gemm_f64_noalloc runs the
// same split and product-sum kernels as emu_gemm_f64, with the same number of
// slices, and keeps their scratch (flag word, level maxima, BF16 planes, FP64
// accumulator) in the file-scope device array below.
//
// The array is EMU_NOALLOC_SCRATCH_BYTES (40 MiB) on every GPU that loads the
// library, for as long as the library stays loaded.  All calls on a device
// share it: each call clears the parts that must start at zero and overwrites
// the rest, and calls whose work overlaps on the GPU (other streams, other
// host threads) race on it.
#include "launchers.cuh"

using namespace emu;

static __device__ __align__(256) unsigned char g_noalloc_scratch[EMU_NOALLOC_SCRATCH_BYTES];

namespace {

// Device address of the scratch array in the current context.  The name of a
// __device__ variable is only a host-side handle, so every call asks the
// runtime for the real address with the caller's device current.  The lookup
// allocates nothing, and asking each time (rather than caching per device)
// stays right when the context is torn down and re-created (cudaDeviceReset),
// after which the module, and with it the array, may sit elsewhere.
cudaError_t scratch_address(unsigned char **out)
{
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    *out = static_cast<unsigned char *>(p);
    return cudaSuccess;
}

int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

}  // namespace

extern "C" emu_status emu_gemm_f64_noalloc(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda,
                                           const double *B, int64_t ldb, double *C, int64_t ldc, int nprod,
                                           uint32_t *flags_out, emu_stream_t stream)
{
    if (M < 0 || N < 0 || K < 0) return EMU_ERR_INVALID_ARG;
    if (lda < (K > 0 ? K : 1) || ldb < (N > 0 ? N : 1) || ldc < (N > 0 ? N : 1)) return EMU_ERR_INVALID_ARG;
    if (nprod != 6 && nprod != 10 && nprod != 15 && nprod != 21) return EMU_ERR_INVALID_ARG;
    if (M > 0 && N > 0 && (!C || (K > 0 && (!A || !B)))) return EMU_ERR_INVALID_ARG;
    // scratch: header, 6 A planes [M][ldk] and 6 B planes [N][ldk] of BF16, FP64 accumulator.
    // Every factor is below 2^31 once the first check has passed, so each term
    // is computed without overflow and compared with the array on its own.
    const int64_t cap = (int64_t)EMU_NOALLOC_SCRATCH_BYTES;
    if (M >= ((int64_t)1 << 31) || N >= ((int64_t)1 << 31) || K >= ((int64_t)1 << 31)) return EMU_ERR_UNSUPPORTED;
    const int64_t ldk = round_up(K < 1 ? 1 : K, 8);
    if (M > cap / (12 * ldk) || N > cap / (12 * ldk)) return EMU_ERR_UNSUPPORTED;
    const int64_t a_bytes = round_up(6 * M * ldk * 2, 256);
    const int64_t b_bytes = round_up(6 * N * ldk * 2, 256);
    if ((M + 127) / 128 > cap / 131072 || (N + 127) / 128 > cap / 131072) return EMU_ERR_UNSUPPORTED;
    const int64_t acc_bytes = (int64_t)f64_acc_bytes(M, N);
    if ((int64_t)kWsHeaderBytes + a_bytes + b_bytes + acc_bytes > cap) return EMU_ERR_UNSUPPORTED;
    const int nlev = f64_diagonals(nprod);      // the slices the product-sum reads, as emu_gemm_f64 splits

    unsigned char *scratch = nullptr;
    if (scratch_address(&scratch) != cudaSuccess) return EMU_ERR_CUDA;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = reinterpret_cast<WsHeader *>(scratch);
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);     // flags and maxima start at zero
    if (e == cudaSuccess && M > 0 && N > 0) {
        if (K == 0) {
            e = cudaMemset2DAsync(C, (size_t)ldc * sizeof(double), 0, (size_t)N * sizeof(double), (size_t)M, st);
        } else {
            uint16_t *Ap = reinterpret_cast<uint16_t *>(scratch + kWsHeaderBytes);
            uint16_t *Bp = reinterpret_cast<uint16_t *>(scratch + kWsHeaderBytes + a_bytes);
            e = launch_split_f64_gemm(A, M, K, lda, B, N, ldb, Ap, Bp, ldk, h->vout[0], h->vout[1], h, st, nlev);
            if (e == cudaSuccess)
                e = launch_prodsum_f64(M, N, K, Ap, Bp, ldk, h->vout[0], h->vout[1], nprod, C, ldc,
                                       reinterpret_cast<double *>(scratch + kWsHeaderBytes + a_bytes + b_bytes),
                                       &h->flags, st);
        }
    }
    if (e == cudaSuccess && flags_out)
        e = cudaMemcpyAsync(flags_out, &h->flags, sizeof(uint32_t), cudaMemcpyDeviceToDevice, st);
    return e == cudaSuccess ? EMU_OK : EMU_ERR_CUDA;
}
