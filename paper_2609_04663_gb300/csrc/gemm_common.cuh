// Shared pieces of the tensor-core product-sum kernels: output-tile
// rasterisation, the FP64 diagonal product order, the FP32 TMEM epilogue, the
// bounded drain of in-flight TMA copies, and the host-side tensor-map
// encoding of a BF16 plane set.
#pragma once

#include "common.cuh"

namespace emu {

constexpr int kBM = 128;
constexpr int kGroupM = 8;       // rasterisation: 8 tile rows walk the N tiles together

__device__ __forceinline__ void tile_coords(int tile, int tiles_m, int tiles_n, int &tm, int &tn)
{
    const int group_size = kGroupM * tiles_n;
    const int first_m = (tile / group_size) * kGroupM;
    const int gm = min(tiles_m - first_m, kGroupM);
    const int local = tile % group_size;
    tm = first_m + local % gm;
    tn = local / gm;
}

// FP64 diagonal order (Algorithm 2): diagonal l = 0..5, i ascending, j = l - i.
// The first 6 / 10 / 15 / 21 entries are the sets S_3 .. S_6.
namespace {
__constant__ int8_t kDiag[21][2] = {{0, 0}, {0, 1}, {1, 0}, {0, 2}, {1, 1}, {2, 0}, {0, 3},
                                    {1, 2}, {2, 1}, {3, 0}, {0, 4}, {1, 3}, {2, 2}, {3, 1},
                                    {4, 0}, {0, 5}, {1, 4}, {2, 3}, {3, 2}, {4, 1}, {5, 0}};
}  // namespace

// Epilogue of one warp: accumulator columns [c0, c1) of the warp's TMEM lane
// quarter (tile rows quarter * 32 ..) -> C.
__device__ __forceinline__ void store_tile(uint32_t tmem, int quarter, int c0, int c1, int m0, int n0, int M, int N,
                                           float *__restrict__ C, int64_t ldc)
{
    tc_fence_after();
    const int row = m0 + quarter * 32 + lane_id();
    float *crow = C + (int64_t)row * ldc;
    const bool vec = ((ldc & 3) == 0) && ((reinterpret_cast<uintptr_t>(C) & 15u) == 0);
#pragma unroll 1
    for (int c = c0; c < c1; c += 32) {
        uint32_t v[32];
        tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c, v);
        tmem_ld_wait();
        const int col = n0 + c;
        if (row < M) {
            if (vec && col + 32 <= N) {
#pragma unroll
                for (int j = 0; j < 32; j += 4)
                    *reinterpret_cast<float4 *>(crow + col + j) =
                        make_float4(__uint_as_float(v[j]), __uint_as_float(v[j + 1]),
                                    __uint_as_float(v[j + 2]), __uint_as_float(v[j + 3]));
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (col + j < N) crow[col + j] = __uint_as_float(v[j]);
            }
        }
    }
}

// Wait (bounded) for the TMA loads the producer issued that the MMA warp may
// not have consumed: used only when a wait already timed out, so that no
// copy into shared memory is left in flight when the CTA exits.
__device__ __forceinline__ void drain_inflight(uint32_t full0, int stages, long issued, uint32_t *flags)
{
    for (long L = issued - stages < 0 ? 0 : issued - stages; L < issued; ++L)
        (void)mbar_wait(full0 + 8u * (uint32_t)(L % stages), (uint32_t)((L / stages) & 1), flags, 100000000ull);
}

// ------------------------------------------------------------ host side
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                   CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                   CUtensorMapFloatOOBfill);

inline EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = []() -> EncodeTiledFn {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return nullptr;
        return reinterpret_cast<EncodeTiledFn>(p);
    }();
    return fn;
}

// Tensor map over a plane set [S][rows][ldcomp] of BF16: dims (K, rows, S),
// box (kb, box_rows, 1), swizzle matching a kb * 2-byte row.  Out-of-range
// boxes (ragged M, N, K) read zeros.  plane: distance between planes in
// elements (0 = rows * ldcomp).
inline bool make_plane_map(CUtensorMap *map, const uint16_t *planes, int64_t K, int64_t rows, int S, int64_t ldcomp,
                    int kb, int box_rows, int64_t plane = 0)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)rows, (cuuint64_t)S};
    cuuint64_t strides[2] = {(cuuint64_t)ldcomp * 2, (cuuint64_t)(plane ? plane : rows * ldcomp) * 2};
    cuuint32_t box[3] = {(cuuint32_t)kb, (cuuint32_t)box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    const CUtensorMapSwizzle swz = (kb == 64) ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<uint16_t *>(planes), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor map over an FP32 matrix C [M][ldc] for 32 x 32 boxes (128-byte rows,
// 128-byte swizzle), the unit of the product-sum's reduction epilogue.
// False when C cannot be described (base not 16-byte aligned, row pitch not
// a multiple of 16 bytes) or when N is not a multiple of 4: a bulk tensor
// reduction clips a box at the end of a row only to whole 16-byte pieces
// (on GB300 a box over columns 320-351 of a 333-column C also wrote columns
// 333-335), which would reach into the padding of C.
inline bool make_c_map_f32(CUtensorMap *map, float *C, int64_t M, int64_t N, int64_t ldc)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc || (reinterpret_cast<uintptr_t>(C) & 15u) != 0 || (ldc & 3) != 0 || (N & 3) != 0) return false;
    cuuint64_t dims[2] = {(cuuint64_t)N, (cuuint64_t)M};
    cuuint64_t strides[1] = {(cuuint64_t)ldc * 4};
    cuuint32_t box[2] = {32, 32};
    cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, C, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The same for an FP64 C [M][ldc], boxes of 32 rows x 16 columns (128-byte
// rows); N must be even for the same reason.
inline bool make_c_map_f64(CUtensorMap *map, double *C, int64_t M, int64_t N, int64_t ldc)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc || (reinterpret_cast<uintptr_t>(C) & 15u) != 0 || (ldc & 1) != 0 || (N & 1) != 0) return false;
    cuuint64_t dims[2] = {(cuuint64_t)N, (cuuint64_t)M};
    cuuint64_t strides[1] = {(cuuint64_t)ldc * 8};
    cuuint32_t box[2] = {16, 32};
    cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT64, 2, C, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace emu
