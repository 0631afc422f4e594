// GEMM from host buffers (emu_gemm_f32_host / emu_gemm_f64_host, declared in
// include/emu.h): the call a user with data in host memory makes.  The copies
// to the device, the split (Eqs. (fp32split), (fp64split)), the product-sum
// and the copy of C back to the host are pipelined over panels on internal
// streams, so that the host link and the GPU work at the same time:
//
//   FP32: the first row panel of A arrives, then B's first column panel, A's
//   second row panel and the rest of B in column panels; as each column panel
//   lands it is split and both leading row panels multiply it (one block of C
//   each, on the two compute streams), so the GPU works while B streams in.  The remaining row panels of A then arrive, are split
//   and multiplied with all of B.  Every finished row panel of C goes back
//   while the next one is computed; row panels alternate between the two
//   compute streams so that one panel's last wave of CTAs overlaps the next.
//
//   FP64: the split needs the maximum over the whole operand (Eq. (fp64split)),
//   so A and B arrive whole; B's copy overlaps A's split, and C goes back in
//   row panels as above.
//
// The arithmetic is that of emu_gemm_f32 / emu_gemm_f64 (same kernels, same
// per-tile order), so the results are bit-identical to them.
#include <mutex>

#include "launchers.cuh"

using namespace emu;

namespace {

constexpr int kMaxDevices = 64;
constexpr int kPanelsM = 8;                         // row panels of C (at most)
constexpr int kPanelsN = 4;                         // column panels of B in FP32 mode (at most)
constexpr int kEvents = 2 * kPanelsN + 4 * kPanelsM + 8;
constexpr int64_t kMaxDim = (int64_t)1 << 31;

int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }
int64_t ceil_div(int64_t x, int64_t a) { return (x + a - 1) / a; }

// Internal streams and events of one device, created on first use and kept
// for the life of the process; a call holds the mutex while it enqueues.
struct HostCtx {
    cudaStream_t cin = nullptr, cout = nullptr, comp[2] = {nullptr, nullptr};
    cudaEvent_t ev[kEvents] = {};
    bool ready = false;
};
std::mutex g_mutex;
HostCtx g_ctx[kMaxDevices];

cudaError_t device_ctx(HostCtx **out)
{
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    HostCtx &c = g_ctx[dev];
    if (!c.ready) {
        cudaStream_t *ss[4] = {&c.cin, &c.cout, &c.comp[0], &c.comp[1]};
        for (cudaStream_t *s : ss)
            if (!*s && (e = cudaStreamCreateWithFlags(s, cudaStreamNonBlocking)) != cudaSuccess) return e;
        for (cudaEvent_t &v : c.ev)
            if (!v && (e = cudaEventCreateWithFlags(&v, cudaEventDisableTiming)) != cudaSuccess) return e;
        c.ready = true;
    }
    *out = &c;
    return cudaSuccess;
}

// Panel geometry: row panels of Mp rows (a multiple of the 128-row CTA tile),
// column panels of Nb columns (a multiple of the FP32 kernel's 256-column tile).
struct Geometry {
    int64_t ldk, Mp, PM, Nb, PN;
    Geometry(int64_t M, int64_t N, int64_t K)
    {
        ldk = round_up(K < 1 ? 1 : K, 8);
        Mp = round_up(ceil_div(M, kPanelsM), 128);
        if (Mp < 128) Mp = 128;
        PM = ceil_div(M, Mp);
        Nb = round_up(ceil_div(N, kPanelsN), 256);
        if (Nb < 256) Nb = 256;
        PN = ceil_div(N, Nb);
    }
};

// Workspace layout (each part 256-byte aligned): header, A planes [s][M][ldk],
// B planes [s][N][ldk], A staging, B staging, C ring of two row panels, and in
// FP64 mode one product-sum accumulator per ring slot.  FP32 stages two row
// panels of A and two column panels of B; FP64 stages A and B whole.
struct Layout {
    size_t ap, bp, ast, bst, cring, acc, total;
    Layout(int mode, int64_t M, int64_t N, int64_t K)
    {
        const Geometry g(M, N, K);
        const int64_t s = mode == 64 ? 6 : 3, esz = mode == 64 ? 8 : 4;
        ap = kWsHeaderBytes;
        bp = ap + (size_t)round_up(s * M * g.ldk * 2, 256);
        ast = bp + (size_t)round_up(s * N * g.ldk * 2, 256);
        const int64_t a_stage = mode == 64 ? M * K : 2 * g.Mp * K;
        const int64_t b_stage = mode == 64 ? K * N : 2 * K * g.Nb;
        bst = ast + (size_t)round_up(a_stage * esz, 256);
        cring = bst + (size_t)round_up(b_stage * esz, 256);
        acc = cring + (size_t)round_up(2 * g.Mp * N * esz, 256);
        total = acc + (mode == 64 ? 2 * f64_acc_bytes(g.Mp, N) : 0);   // FP64 accumulators of the two ring slots
    }
};

emu_status check_args(int64_t M, int64_t N, int64_t K, const void *A, int64_t lda, const void *B, int64_t ldb,
                      const void *C, int64_t ldc, const void *ws, size_t ws_bytes, int mode)
{
    if (M < 0 || N < 0 || K < 0 || !ws) return EMU_ERR_INVALID_ARG;
    if (lda < (K > 0 ? K : 1) || ldb < (N > 0 ? N : 1) || ldc < (N > 0 ? N : 1)) return EMU_ERR_INVALID_ARG;
    if (M >= kMaxDim || N >= kMaxDim || K >= kMaxDim) return EMU_ERR_UNSUPPORTED;
    if (M > 0 && N > 0 && (!C || (K > 0 && (!A || !B)))) return EMU_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return EMU_ERR_MISALIGNED;
    if (ws_bytes < Layout(mode, M, N, K).total) return EMU_ERR_WORKSPACE_TOO_SMALL;
    return EMU_OK;
}

// Shared part of both modes: the row-panel loop.  `compute(i, m0, mp, Cpanel,
// stream)` enqueues the product-sum of row panel i into the ring slot; the
// finished panel is copied to C rows m0 .. m0 + mp on the copy-out stream.
template <typename T, typename Compute, typename Prepare>
cudaError_t row_panels(HostCtx &cx, int &ne, const Geometry &g, int64_t M, int64_t N, T *C, int64_t ldc,
                       T *cring, Prepare prepare, Compute compute)
{
    cudaEvent_t cdone[kPanelsM] = {};
    cudaError_t e = cudaSuccess;
    for (int64_t i = 0; i < g.PM && e == cudaSuccess; ++i) {
        const int64_t m0 = i * g.Mp, mp = (M - m0 < g.Mp) ? M - m0 : g.Mp;
        const int slot = (int)(i & 1);
        cudaStream_t cs = cx.comp[slot];
        T *cr = cring + (int64_t)slot * g.Mp * N;
        e = prepare(i, m0, mp, cs);
        if (e == cudaSuccess && i >= 2) e = cudaStreamWaitEvent(cs, cdone[i - 2], 0);   // ring slot copied out
        if (e == cudaSuccess) e = compute(i, m0, mp, cr, cs);
        cudaEvent_t ready = cx.ev[ne++];
        if (e == cudaSuccess) e = cudaEventRecord(ready, cs);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cx.cout, ready, 0);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(C + m0 * ldc, (size_t)ldc * sizeof(T), cr, (size_t)N * sizeof(T),
                                  (size_t)N * sizeof(T), (size_t)mp, cudaMemcpyDeviceToHost, cx.cout);
        cdone[i] = cx.ev[ne++];
        if (e == cudaSuccess) e = cudaEventRecord(cdone[i], cx.cout);
    }
    return e;
}

// Orders the internal streams after the work already on `st` and clears the
// workspace header (flag word, split state) on `st`.
cudaError_t begin(HostCtx &cx, int &ne, WsHeader *h, cudaStream_t st)
{
    cudaError_t e = cudaMemsetAsync(h, 0, sizeof(WsHeader), st);
    cudaEvent_t start = cx.ev[ne++];
    if (e == cudaSuccess) e = cudaEventRecord(start, st);
    cudaStream_t ss[4] = {cx.cin, cx.cout, cx.comp[0], cx.comp[1]};
    for (cudaStream_t s : ss)
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s, start, 0);
    return e;
}

// `st` waits for the last copy of C (which follows every other step).
cudaError_t finish(HostCtx &cx, int &ne, cudaStream_t st)
{
    cudaEvent_t end = cx.ev[ne++];
    cudaError_t e = cudaEventRecord(end, cx.cout);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(st, end, 0);
    return e;
}

}  // namespace

extern "C" {

size_t emu_gemm_host_workspace_bytes(int mode, int64_t M, int64_t N, int64_t K)
{
    if (M < 0 || N < 0 || K < 0 || (mode != 32 && mode != 64)) return 0;
    return Layout(mode, M, N, K).total;
}

emu_status emu_gemm_f32_host(int64_t M, int64_t N, int64_t K, const float *A, int64_t lda, const float *B,
                             int64_t ldb, float *C, int64_t ldc, void *ws, size_t ws_bytes, emu_stream_t stream)
{
    emu_status s = check_args(M, N, K, A, lda, B, ldb, C, ldc, ws, ws_bytes, 32);
    if (s != EMU_OK) return s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    if (M == 0 || N == 0) return cudaMemsetAsync(h, 0, sizeof(WsHeader), st) == cudaSuccess ? EMU_OK : EMU_ERR_CUDA;

    std::lock_guard<std::mutex> lock(g_mutex);
    HostCtx *cx = nullptr;
    if (device_ctx(&cx) != cudaSuccess) return EMU_ERR_CUDA;
    const Geometry g(M, N, K);
    const Layout L(32, M, N, K);
    unsigned char *w = static_cast<unsigned char *>(ws);
    uint16_t *Ap = reinterpret_cast<uint16_t *>(w + L.ap), *Bp = reinterpret_cast<uint16_t *>(w + L.bp);
    float *Ast = reinterpret_cast<float *>(w + L.ast), *Bst = reinterpret_cast<float *>(w + L.bst);
    float *cring = reinterpret_cast<float *>(w + L.cring);
    const int64_t a_plane = M * g.ldk, b_plane = N * g.ldk;
    int ne = 0;
    cudaError_t e = begin(*cx, ne, h, st);
    if (K == 0) {                                     // C = 0, panel by panel
        auto none = [](int64_t, int64_t, int64_t, cudaStream_t) -> cudaError_t { return cudaSuccess; };
        auto zero = [&](int64_t, int64_t, int64_t mp, float *cr, cudaStream_t cs) -> cudaError_t {
            return cudaMemsetAsync(cr, 0, (size_t)mp * N * 4, cs);
        };
        if (e == cudaSuccess) e = row_panels(*cx, ne, g, M, N, C, ldc, cring, none, zero);
        if (e == cudaSuccess) e = finish(*cx, ne, st);
        return e == cudaSuccess ? EMU_OK : EMU_ERR_CUDA;
    }

    // row panel i of A: copy into staging slot i & 1, split into plane rows
    // m0 .. m0 + mp on stream cs
    cudaEvent_t asplit[kPanelsM] = {};
    auto load_a = [&](int64_t i, cudaStream_t cs) -> cudaError_t {
        const int64_t m0 = i * g.Mp, mp = (M - m0 < g.Mp) ? M - m0 : g.Mp;
        float *as = Ast + (i & 1) * g.Mp * K;
        cudaError_t r = (i >= 2) ? cudaStreamWaitEvent(cx->cin, asplit[i - 2], 0) : cudaSuccess;
        if (r == cudaSuccess)
            r = cudaMemcpy2DAsync(as, (size_t)K * 4, A + m0 * lda, (size_t)lda * 4, (size_t)K * 4, (size_t)mp,
                                  cudaMemcpyHostToDevice, cx->cin);
        cudaEvent_t landed = cx->ev[ne++];
        if (r == cudaSuccess) r = cudaEventRecord(landed, cx->cin);
        if (r == cudaSuccess) r = cudaStreamWaitEvent(cs, landed, 0);
        if (r == cudaSuccess) r = launch_split_f32(as, mp, K, K, false, Ap + m0 * g.ldk, g.ldk, h, cs, a_plane);
        asplit[i] = cx->ev[ne++];
        if (r == cudaSuccess) r = cudaEventRecord(asplit[i], cs);
        return r;
    };
    // C row panel i goes back to the host once computed on stream cs
    cudaEvent_t cdone[kPanelsM] = {};
    auto store_c = [&](int64_t i, cudaStream_t cs) -> cudaError_t {
        const int64_t m0 = i * g.Mp, mp = (M - m0 < g.Mp) ? M - m0 : g.Mp;
        cudaEvent_t ready = cx->ev[ne++];
        cudaError_t r = cudaEventRecord(ready, cs);
        if (r == cudaSuccess) r = cudaStreamWaitEvent(cx->cout, ready, 0);
        if (r == cudaSuccess)
            r = cudaMemcpy2DAsync(C + m0 * ldc, (size_t)ldc * 4, cring + (i & 1) * g.Mp * N, (size_t)N * 4,
                                  (size_t)N * 4, (size_t)mp, cudaMemcpyDeviceToHost, cx->cout);
        cdone[i] = cx->ev[ne++];
        if (r == cudaSuccess) r = cudaEventRecord(cdone[i], cx->cout);
        return r;
    };

    // the leading row panels, then B column by column, each column panel
    // multiplied by the leading row panels as soon as it is split.  Copy
    // order: A row panel 0, B column panel 0, A row panel 1, then the rest of
    // B, so that the first product-sum waits for two copies, not three.
    const int64_t lead = g.PM < 2 ? g.PM : 2;
    if (e == cudaSuccess) e = load_a(0, cx->comp[0]);
    cudaEvent_t bsplit[kPanelsN] = {};
    for (int64_t j = 0; j < g.PN && e == cudaSuccess; ++j) {
        const int64_t n0 = j * g.Nb, nb = (N - n0 < g.Nb) ? N - n0 : g.Nb;
        float *bs = Bst + (j & 1) * K * g.Nb;
        if (j >= 2) e = cudaStreamWaitEvent(cx->cin, bsplit[j - 2], 0);       // staging slot consumed
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(bs, (size_t)nb * 4, B + n0, (size_t)ldb * 4, (size_t)nb * 4, (size_t)K,
                                  cudaMemcpyHostToDevice, cx->cin);
        cudaEvent_t landed = cx->ev[ne++];
        if (e == cudaSuccess) e = cudaEventRecord(landed, cx->cin);
        if (e == cudaSuccess && j == 0 && lead > 1) e = load_a(1, cx->comp[1]);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cx->comp[0], landed, 0);
        if (e == cudaSuccess) e = launch_split_f32(bs, K, nb, nb, true, Bp + n0 * g.ldk, g.ldk, h, cx->comp[0], b_plane);
        bsplit[j] = cx->ev[ne++];
        if (e == cudaSuccess) e = cudaEventRecord(bsplit[j], cx->comp[0]);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cx->comp[1], bsplit[j], 0);
        for (int64_t i = 0; i < lead && e == cudaSuccess; ++i) {
            const int64_t m0 = i * g.Mp, mp = (M - m0 < g.Mp) ? M - m0 : g.Mp;
            e = launch_prodsum_f32(mp, nb, K, Ap + m0 * g.ldk, Bp + n0 * g.ldk, g.ldk, cring + i * g.Mp * N + n0, N,
                                   &h->flags, cx->comp[i], a_plane, b_plane);
        }
    }
    for (int64_t i = 0; i < lead && e == cudaSuccess; ++i) e = store_c(i, cx->comp[i]);
    // the remaining row panels against all of B (both compute streams have
    // waited for every column panel's split)
    for (int64_t i = lead; i < g.PM && e == cudaSuccess; ++i) {
        const int64_t m0 = i * g.Mp, mp = (M - m0 < g.Mp) ? M - m0 : g.Mp;
        cudaStream_t cs = cx->comp[i & 1];
        e = load_a(i, cs);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, cdone[i - 2], 0);   // C ring slot copied out
        if (e == cudaSuccess)
            e = launch_prodsum_f32(mp, N, K, Ap + m0 * g.ldk, Bp, g.ldk, cring + (i & 1) * g.Mp * N, N, &h->flags, cs,
                                   a_plane);
        if (e == cudaSuccess) e = store_c(i, cs);
    }
    if (e == cudaSuccess) e = finish(*cx, ne, st);
    return e == cudaSuccess ? EMU_OK : EMU_ERR_CUDA;
}

emu_status emu_gemm_f64_host(int64_t M, int64_t N, int64_t K, const double *A, int64_t lda, const double *B,
                             int64_t ldb, double *C, int64_t ldc, int nprod, void *ws, size_t ws_bytes,
                             emu_stream_t stream)
{
    if (nprod != 6 && nprod != 10 && nprod != 15 && nprod != 21) return EMU_ERR_INVALID_ARG;
    const int nlev = f64_diagonals(nprod);   // slices the product-sum uses
    emu_status s = check_args(M, N, K, A, lda, B, ldb, C, ldc, ws, ws_bytes, 64);
    if (s != EMU_OK) return s;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    WsHeader *h = static_cast<WsHeader *>(ws);
    if (M == 0 || N == 0) return cudaMemsetAsync(h, 0, sizeof(WsHeader), st) == cudaSuccess ? EMU_OK : EMU_ERR_CUDA;

    std::lock_guard<std::mutex> lock(g_mutex);
    HostCtx *cx = nullptr;
    if (device_ctx(&cx) != cudaSuccess) return EMU_ERR_CUDA;
    const Geometry g(M, N, K);
    const Layout L(64, M, N, K);
    unsigned char *w = static_cast<unsigned char *>(ws);
    uint16_t *Ap = reinterpret_cast<uint16_t *>(w + L.ap), *Bp = reinterpret_cast<uint16_t *>(w + L.bp);
    double *Ast = reinterpret_cast<double *>(w + L.ast), *Bst = reinterpret_cast<double *>(w + L.bst);
    double *cring = reinterpret_cast<double *>(w + L.cring);
    const int64_t a_plane = M * g.ldk;
    int ne = 0;
    cudaError_t e = begin(*cx, ne, h, st);

    if (K > 0) {
        // A whole, split (comp[0]) while B is copied; then B's split
        cudaEvent_t a_in = cx->ev[ne++], b_in = cx->ev[ne++], split = cx->ev[ne++];
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(Ast, (size_t)K * 8, A, (size_t)lda * 8, (size_t)K * 8, (size_t)M,
                                  cudaMemcpyHostToDevice, cx->cin);
        if (e == cudaSuccess) e = cudaEventRecord(a_in, cx->cin);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(Bst, (size_t)N * 8, B, (size_t)ldb * 8, (size_t)N * 8, (size_t)K,
                                  cudaMemcpyHostToDevice, cx->cin);
        if (e == cudaSuccess) e = cudaEventRecord(b_in, cx->cin);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cx->comp[0], a_in, 0);
        if (e == cudaSuccess)
            e = launch_split_f64(Ast, M, K, K, false, Ap, g.ldk, h->vout[0], h, 0, cx->comp[0], nlev);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cx->comp[0], b_in, 0);
        if (e == cudaSuccess)
            e = launch_split_f64(Bst, K, N, N, true, Bp, g.ldk, h->vout[1], h, 1, cx->comp[0], nlev);
        if (e == cudaSuccess) e = cudaEventRecord(split, cx->comp[0]);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(cx->comp[1], split, 0);
    }
    auto prepare = [](int64_t, int64_t, int64_t, cudaStream_t) -> cudaError_t { return cudaSuccess; };
    auto compute = [&](int64_t i, int64_t m0, int64_t mp, double *cr, cudaStream_t cs) -> cudaError_t {
        if (K == 0) return cudaMemsetAsync(cr, 0, (size_t)mp * N * 8, cs);
        double *acc = reinterpret_cast<double *>(w + L.acc + (i & 1) * f64_acc_bytes(g.Mp, N));
        return launch_prodsum_f64(mp, N, K, Ap + m0 * g.ldk, Bp, g.ldk, h->vout[0], h->vout[1], nprod, cr, N, acc,
                                  &h->flags, cs, a_plane);
    };
    if (e == cudaSuccess) e = row_panels(*cx, ne, g, M, N, C, ldc, cring, prepare, compute);
    if (e == cudaSuccess) e = finish(*cx, ne, st);
    return e == cudaSuccess ? EMU_OK : EMU_ERR_CUDA;
}

}  // extern "C"
