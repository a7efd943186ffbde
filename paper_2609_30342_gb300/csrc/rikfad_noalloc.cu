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
// All calls share that one array and it keeps the last call's contents.  The
// block counter that must start at zero is cleared by every call before its
// launch; the partial sums are fully rewritten each call.  Two calls whose
// kernels overlap on the GPU (different streams, no ordering) race on the
// array and produce wrong results.
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
constexpr int kNaMaxBlocks = 128;
constexpr int64_t kNaCtlFloats = 64;             // word 0: finished-block counter
constexpr int64_t kNaScratchFloats = kNaCtlFloats + kNaMaxRows + (int64_t)kNaMaxBlocks * kNaMaxCols;

}  // namespace

// 4.45 MB of scratch: counter | row sums (rows) | column partials (blocks x cols).
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

// One launch does the whole step: every block streams its row range with the
// same per-row code as the multi-tensor kernel, writes its column partial
// sums, and the block that finishes last folds all partials into R and C.
template <typename GT, bool REUSE>
__global__ void __launch_bounds__(kThreads) rikfad_noalloc_step_kernel(NoAllocParams na, float *scratch)
{
    __shared__ __align__(16) float Cs[kPanelMax];
    __shared__ __align__(16) float red[kWarps * kPanelMax];
    __shared__ void *ptrs[3];
    __shared__ float wsum[kWarps];
    __shared__ int is_last;
    unsigned *counter = reinterpret_cast<unsigned *>(scratch);
    float *rowsum = scratch + kNaCtlFloats;
    float *colpart = scratch + kNaCtlFloats + kNaMaxRows;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.x;
    const int w = (int)na.cols;

    // 1^T R, summed in the same fixed order by every block.
    float v = 0.f;
    for (int64_t i = tid; i < na.rows; i += kThreads)
        v += na.R[i];
    v = warp_sum(v);
    if (lane == 0)
        wsum[warp] = v;
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
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < kWarps; ++k)
        s += wsum[k];
    const float inv = inv_denominator(s, na.eps);

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

    // The last block to get here applies the factor update.
    __threadfence();
    __syncthreads();
    if (tid == 0)
        is_last = atomicAdd(counter, 1u) == (unsigned)(na.nblocks - 1);
    __syncthreads();
    if (!is_last)
        return;
    __threadfence();
    for (int64_t i = tid; i < na.rows; i += kThreads)
        na.R[i] = fmaf(na.gain, __ldcg(rowsum + i), na.decay * na.R[i]);
    for (int c = tid; c < w; c += kThreads) {
        float t = 0.f;
        for (int k = 0; k < na.nblocks; ++k)
            t += __ldcg(colpart + (int64_t)k * w + c);
        na.C[c] = fmaf(na.gain, t, na.decay * na.C[c]);
    }
    if (tid == 0)
        *counter = 0u;
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
    cudaError_t e = cudaMemsetAsync(scratch, 0, sizeof(float) * kNaCtlFloats, s);
    if (e != cudaSuccess)
        return na_fail(RIKFAD_ERR_CUDA, cudaGetErrorString(e));

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
    e = cudaGetLastError();
    if (e != cudaSuccess)
        return na_fail(RIKFAD_ERR_CUDA, cudaGetErrorString(e));
    return RIKFAD_OK;
}
