// rikfad_noalloc.cu -- an allocation-free variant of the R-iKFAD step for one
// matrix.
//
// The handle API (rikfad_create / rikfad_step) allocates its reduction
// workspace with cudaMalloc when the handle is created.  Some callers cannot
// do that: a framework whose caching allocator already owns the GPU's memory
// (a second allocator competing for it fails or fragments the pool), or a
// latency-bound service that forbids cudaMalloc after start-up because the
// call can synchronise the device and stall every stream.  For them,
// rikfad_step_matrix_noalloc takes caller-owned inputs and outputs and keeps
// its partial sums in the file-scope device array below, which is part of the
// library image itself: every GPU that loads the library holds it until the
// process exits.
//
// All calls share that one array and it keeps the last call's contents.  A
// call needs nothing in it to start at zero: it writes every partial sum it
// later reads (the partial sums of R, the row sums, the column partials)
// before reading them, in three launches ordered on the caller's stream.  Two
// calls whose kernels overlap on the GPU (different streams, no ordering)
// race on the array and produce wrong results.
#include <cuda_runtime.h>

#include <cmath>
#include <mutex>
#include <string>

#include "rikfad.h"
#include "rikfad_kernels.cuh"

using namespace rikfad;

namespace {

constexpr int64_t kNaMaxRows = 65536;            // largest matrix: 65536 x 1024
constexpr int64_t kNaMaxCols = kPanelMax;        // one column panel
constexpr int kNaMaxBlocks = 304;                // step blocks: 2 per SM of a GB300
constexpr int kNaRowGroup = 1024;                // rows per partial sum of R
constexpr int64_t kNaRsumFloats = kNaMaxRows / kNaRowGroup;     // 64
constexpr int kNaColsPerItem = 32;               // columns per block of the column finalise
constexpr int64_t kNaScratchFloats = kNaRsumFloats + kNaMaxRows + (int64_t)kNaMaxBlocks * kNaMaxCols;

}  // namespace

// 1.51 MB of scratch: partial sums of R (64) | row sums (rows) | column
// partials (blocks x cols).
static __device__ __align__(256) float g_noalloc_scratch[kNaScratchFloats];

namespace rikfad {
int report_error(int code, const std::string &msg);
}

namespace {

struct NoAllocParams {
    int64_t rows;
    int64_t cols;
    int nblocks;
    int vec;
    float *x;
    const void *g;
    float *p;
    float *R;
    float *C;
    float h, ex_cur, ex_prev, damp_prev, decay, gain, eps;
};

// Partial sums of R over groups of kNaRowGroup rows, in a fixed order.
__global__ void __launch_bounds__(kThreads) rikfad_noalloc_rsum_kernel(const float *R, int64_t rows,
                                                                       float *rsum)
{
    __shared__ float wsum[kWarps];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t r0 = (int64_t)blockIdx.x * kNaRowGroup;
    float v = 0.f;
    for (int64_t i = r0 + tid; i < rows && i < r0 + kNaRowGroup; i += kThreads)
        v += R[i];
    v = warp_sum(v);
    if (lane == 0)
        wsum[warp] = v;
    __syncthreads();
    if (tid == 0) {
        float t = 0.f;
        for (int k = 0; k < kWarps; ++k)
            t += wsum[k];
        rsum[blockIdx.x] = t;
    }
}

// The streaming pass: every block takes a contiguous range of rows with the
// same per-row code as the multi-tensor kernel and writes its column partial
// sums; the row sums go to the scratch too.
template <typename GT, bool REUSE>
__global__ void __launch_bounds__(kThreads, RIKFAD_STEP_MIN_BLOCKS)
    rikfad_noalloc_step_kernel(NoAllocParams na, float *scratch)
{
    __shared__ __align__(16) float Cs[kPanelMax];
    __shared__ __align__(16) float red[kWarps * kPanelMax];
    __shared__ void *ptrs[3];
    const float *rsum = scratch;
    float *rowsum = scratch + kNaRsumFloats;
    float *colpart = scratch + kNaRsumFloats + kNaMaxRows;
    const int tid = threadIdx.x, lane = tid & 31;
    const int b = blockIdx.x;
    const int w = (int)na.cols;

    // 1^T R from the partial sums, in the same fixed order in every warp.
    const int nrs = (int)((na.rows + kNaRowGroup - 1) / kNaRowGroup);
    float v = 0.f;
    for (int k = lane; k < nrs; k += 32)
        v += rsum[k];
    const float inv = inv_denominator(warp_sum(v), na.eps);
    for (int c = tid; c < w; c += kThreads)
        Cs[c] = na.C[c];
    for (int i = tid; i < kWarps * kPanelMax; i += kThreads)
        red[i] = 0.f;
    if (tid == 0) {
        ptrs[0] = na.x;
        ptrs[1] = const_cast<void *>(na.g);
        ptrs[2] = na.p;
    }
    __syncthreads();

    StepParams a{};
    a.xptr = reinterpret_cast<float *const *>(&ptrs[0]);
    a.gptr = reinterpret_cast<const void *const *>(&ptrs[1]);
    a.pptr = reinterpret_cast<float *const *>(&ptrs[2]);
    a.fac = na.R;
    a.rowpart = rowsum;
    a.h = na.h;
    a.ex_cur = na.ex_cur;
    a.ex_prev = na.ex_prev;
    a.damp_prev = na.damp_prev;
    a.decay = na.decay;
    a.gain = na.gain;
    a.eps = na.eps;
    TensorDev td{};
    td.rows = na.rows;
    td.cols = na.cols;
    td.npanels = 1;
    td.vec = na.vec;
    PanelDev pd{};
    pd.width = w;
    pd.nch = (w + kChunk - 1) / kChunk;
    pd.slot_end = 1;
    PieceDev pc{};
    pc.kind = kMatrixRows;
    pc.begin = na.rows * b / na.nblocks;
    pc.end = na.rows * (b + 1) / na.nblocks;
    if (na.vec)
        matrix_piece_vec<GT, REUSE>(a, pc, td, pd, Cs, red, inv);
    else
        matrix_piece_scalar<GT, REUSE>(a, pc, td, pd, Cs, red, inv);
    __syncthreads();
    for (int c = tid; c < w; c += kThreads) {
        float t = 0.f;
#pragma unroll
        for (int k = 0; k < kWarps; ++k)
            t += red[k * kPanelMax + c];
        colpart[(int64_t)b * w + c] = t;
    }
}

// The factor filter: blocks [0, nrow) update kThreads rows of R each from the
// row sums; the others update kNaColsPerItem columns of C each, the 8 warps
// adding every 8th block's partial and then the warp sums in order.
__global__ void __launch_bounds__(kThreads) rikfad_noalloc_finalize_kernel(NoAllocParams na,
                                                                           const float *scratch, int nrow)
{
    __shared__ float csum[kWarps][32];
    const float *rowsum = scratch + kNaRsumFloats;
    const float *colpart = scratch + kNaRsumFloats + kNaMaxRows;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if ((int)blockIdx.x < nrow) {
        const int64_t i = (int64_t)blockIdx.x * kThreads + tid;
        if (i < na.rows)
            na.R[i] = fmaf(na.gain, rowsum[i], na.decay * na.R[i]);
        return;
    }
    const int64_t c = (int64_t)(blockIdx.x - nrow) * kNaColsPerItem + lane;
    float acc = 0.f;
    if (c < na.cols) {
#pragma unroll 4
        for (int k = warp; k < na.nblocks; k += kWarps)
            acc += colpart[(int64_t)k * na.cols + c];
    }
    csum[warp][lane] = acc;
    __syncthreads();
    if (warp == 0 && c < na.cols) {
        float t = 0.f;
#pragma unroll
        for (int k = 0; k < kWarps; ++k)
            t += csum[k][lane];
        na.C[c] = fmaf(na.gain, t, na.decay * na.C[c]);
    }
}

// Device address of the scratch array, looked up once per device.
std::mutex g_na_mutex;
float *g_na_addr[128] = {};

int scratch_address(float **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return report_error(RIKFAD_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    if (dev < 0 || dev >= 128)
        return report_error(RIKFAD_ERR_STATE, "device index out of range");
    std::lock_guard<std::mutex> lock(g_na_mutex);
    if (g_na_addr[dev] == nullptr) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr)
            return report_error(RIKFAD_ERR_CUDA,
                                std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
        g_na_addr[dev] = static_cast<float *>(p);
    }
    *out = g_na_addr[dev];
    return RIKFAD_OK;
}

int na_fail(int code, const char *msg) { return report_error(code, msg); }

}  // namespace

extern "C" RIKFAD_API int rikfad_step_matrix_noalloc(int64_t rows, int64_t cols, double step,
                                                     double pending_step, const rikfad_hparams *hp,
                                                     int grad_dtype, float *x, const void *grad,
                                                     float *p, float *R, float *C, void *stream)
{
    if (rows < 0 || rows > kNaMaxRows)
        return na_fail(RIKFAD_ERR_ARG, "rows must be in [0, 65536]");
    if (cols < 1 || cols > kNaMaxCols)
        return na_fail(RIKFAD_ERR_ARG, "cols must be in [1, 1024]");
    if (hp == nullptr)
        return na_fail(RIKFAD_ERR_ARG, "hp is NULL");
    if (!(std::isfinite(hp->alpha) && hp->alpha > 0) || !(hp->mu > 0) ||
        !(std::isfinite(hp->gamma) && hp->gamma >= 0) ||
        !(std::isfinite(hp->eps_stab) && hp->eps_stab >= 0))
        return na_fail(RIKFAD_ERR_ARG, "hyperparameters out of range");
    if (!(std::isfinite(step) && step > 0) || !(std::isfinite(pending_step) && pending_step >= 0))
        return na_fail(RIKFAD_ERR_ARG, "step must be > 0 and pending_step >= 0");
    if (grad_dtype != RIKFAD_GRAD_F32 && grad_dtype != RIKFAD_GRAD_BF16)
        return na_fail(RIKFAD_ERR_ARG, "grad_dtype must be RIKFAD_GRAD_F32 or RIKFAD_GRAD_BF16");
    if (C == nullptr || (rows > 0 && (x == nullptr || grad == nullptr || p == nullptr || R == nullptr)))
        return na_fail(RIKFAD_ERR_ARG, "NULL pointer");
    const int vec = cols % 8 == 0;
    const size_t gbytes = grad_dtype == RIKFAD_GRAD_BF16 ? 2 : 4;
    const uintptr_t need = vec ? 16 : 4;
    if (rows > 0 && ((uintptr_t)x % need || (uintptr_t)p % need ||
                     (uintptr_t)grad % (vec ? 16 : gbytes)))
        return na_fail(RIKFAD_ERR_ALIGN, "x, grad and p must be 16-byte aligned");
    if ((uintptr_t)C % 4 || (uintptr_t)R % 4)
        return na_fail(RIKFAD_ERR_ALIGN, "R and C must be 4-byte aligned");

    float *scratch = nullptr;
    int rc = scratch_address(&scratch);
    if (rc)
        return rc;
    cudaStream_t s = (cudaStream_t)stream;

    NoAllocParams na{};
    na.rows = rows;
    na.cols = cols;
    na.nblocks = (int)std::max<int64_t>(1, std::min<int64_t>(kNaMaxBlocks, rows));
    na.vec = vec;
    na.x = x;
    na.g = grad;
    na.p = p;
    na.R = R;
    na.C = C;
    na.h = (float)step;
    na.ex_cur = (float)(-0.5 * step * M_LOG2E);
    na.ex_prev = (float)(-0.5 * pending_step * M_LOG2E);
    na.damp_prev = (float)std::exp(-hp->gamma * pending_step);
    na.decay = (float)std::exp(-hp->alpha * step);
    na.gain = std::isinf(hp->mu) ? 0.f : (float)(-std::expm1(-hp->alpha * step) / (hp->mu * hp->alpha));
    na.eps = (float)hp->eps_stab;
    const bool reuse = step == pending_step;
    // Three launches on the caller's stream: partial sums of R, the
    // streaming pass, the factor filter.
    const int nrs = (int)((rows + kNaRowGroup - 1) / kNaRowGroup);
    if (nrs > 0)
        rikfad_noalloc_rsum_kernel<<<nrs, kThreads, 0, s>>>(R, rows, scratch);
    if (grad_dtype == RIKFAD_GRAD_BF16) {
        if (reuse)
            rikfad_noalloc_step_kernel<__nv_bfloat16, true><<<na.nblocks, kThreads, 0, s>>>(na, scratch);
        else
            rikfad_noalloc_step_kernel<__nv_bfloat16, false><<<na.nblocks, kThreads, 0, s>>>(na, scratch);
    } else {
        if (reuse)
            rikfad_noalloc_step_kernel<float, true><<<na.nblocks, kThreads, 0, s>>>(na, scratch);
        else
            rikfad_noalloc_step_kernel<float, false><<<na.nblocks, kThreads, 0, s>>>(na, scratch);
    }
    const int nrow = (int)((rows + kThreads - 1) / kThreads);
    const int ncol = (int)((cols + kNaColsPerItem - 1) / kNaColsPerItem);
    rikfad_noalloc_finalize_kernel<<<nrow + ncol, kThreads, 0, s>>>(na, scratch, nrow);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return na_fail(RIKFAD_ERR_CUDA, cudaGetErrorString(e));
    return RIKFAD_OK;
}
