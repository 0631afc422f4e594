// The verifier and literal fix passes of the whole-matrix FP64 split
// (Eq. (fp64split)), in one cooperative launch after the speculative pass.
#include "split_common.cuh"

namespace emu {

namespace {

// Everything after the fused pass, in one cooperative launch: every block
// checks the speculative levels from the pass's maxima (the same answer in
// each block).  When they held -- the usual case -- block 0 publishes them
// and the launch ends, no block waiting on another.  Otherwise the literal
// passes redo the levels from the first wrong one: the maxima of levels
// fix_from + 1 .. 5 one pass each, then the rewrite of the planes with the
// final levels, the grid synchronised between passes.
template <bool TRANSPOSE>
__global__ void __launch_bounds__(kThreads)
f64_fix_kernel(const double *__restrict__ X, int64_t rows, int64_t cols, int64_t ldx, uint16_t *__restrict__ comps,
               int64_t ldcomp, int64_t plane, WsHeader *ws, int slot, int32_t *v_out, int nlev)
{
    extern __shared__ __align__(16) uint16_t smdyn[];
    __shared__ unsigned long long red[kThreads / 32];
    int v[6];
    const int ff = f64_verify_levels(ws, slot, v, nlev);
    if (ff == 6) {
        if (blockIdx.x == 0 && threadIdx.x == 0) {
            for (int r = 0; r < 6; ++r) ws->v[slot][r] = v[r];
            ws->fix_from[slot] = 6;
            f64_finalize(ws, slot, v_out, nlev);
        }
        return;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        for (int r = 0; r < 6; ++r) ws->v[slot][r] = v[r];
        ws->fix_from[slot] = ff;
    }
    grid_sync(ws, slot);
    f64_max_pass<1>(X, rows, cols, ldx, ws, slot, blockIdx.x, gridDim.x, red);
    grid_sync(ws, slot);
    f64_max_pass<2>(X, rows, cols, ldx, ws, slot, blockIdx.x, gridDim.x, red);
    grid_sync(ws, slot);
    f64_max_pass<3>(X, rows, cols, ldx, ws, slot, blockIdx.x, gridDim.x, red);
    grid_sync(ws, slot);
    f64_max_pass<4>(X, rows, cols, ldx, ws, slot, blockIdx.x, gridDim.x, red);
    grid_sync(ws, slot);
    f64_max_pass<5>(X, rows, cols, ldx, ws, slot, blockIdx.x, gridDim.x, red);
    grid_sync(ws, slot);
    split_tile_pass<double, 2, TRANSPOSE>(X, rows, cols, ldx, comps, ldcomp, plane, ws, slot, nullptr, nullptr,
                                          blockIdx.x, gridDim.x, smdyn);
    grid_sync(ws, slot);
    if (blockIdx.x == 0 && threadIdx.x == 0) f64_finalize(ws, slot, v_out, nlev);
}

}  // namespace

// Cooperative launch of f64_fix_kernel: as many blocks as fit on the device
// at once (at most 152 x 8), found once per device.
template <bool TRANSPOSE>
static cudaError_t launch_f64_fix_t(const double *X, int64_t rows, int64_t cols, int64_t ldx, uint16_t *comps,
                           int64_t ldcomp, int64_t plane, WsHeader *ws, int slot, int32_t *v_out, cudaStream_t st,
                           int nlev)
{
    constexpr int kMaxDev = 64;
    static int grid_of[kMaxDev] = {};
    const size_t sm = smem_bytes(6);
    auto kern = f64_fix_kernel<TRANSPOSE>;
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
    void *args[] = {(void *)&X, (void *)&rows, (void *)&cols, (void *)&ldx, (void *)&comps, (void *)&ldcomp,
                    (void *)&plane, (void *)&ws, (void *)&slot, (void *)&v_out, (void *)&nlev};
    return cudaLaunchCooperativeKernel((const void *)kern, dim3((unsigned)grid), dim3(kThreads), args, sm, st);
}


cudaError_t launch_f64_fix(const double *X, int64_t rows, int64_t cols, int64_t ldx, bool transpose, uint16_t *comps,
                           int64_t ldcomp, int64_t plane, WsHeader *ws, int slot, int32_t *v_out, cudaStream_t st,
                           int nlev)
{
    return transpose ? launch_f64_fix_t<true>(X, rows, cols, ldx, comps, ldcomp, plane, ws, slot, v_out, st, nlev)
                     : launch_f64_fix_t<false>(X, rows, cols, ldx, comps, ldcomp, plane, ws, slot, v_out, st, nlev);
}

// an empty matrix: all levels zero, nothing to fix (one block, no grid barrier)
cudaError_t launch_f64_fix_empty(WsHeader *ws, int slot, int32_t *v_out, cudaStream_t st)
{
    f64_fix_kernel<false><<<1, kThreads, 0, st>>>(nullptr, 0, 0, 1, nullptr, 1, 0, ws, slot, v_out, 6);
    return cudaGetLastError();
}

}  // namespace emu
