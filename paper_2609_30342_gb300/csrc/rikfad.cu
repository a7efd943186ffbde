// rikfad.cu -- C ABI of the R-iKFAD optimiser on GB300 (sm_103a): handle,
// argument checking, device state, and the launches of the step kernels.
#include <cuda_runtime.h>

#include <atomic>
#include <climits>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "rikfad.h"
#include "rikfad_aux_kernels.cuh"
#include "rikfad_sweep.cuh"
#include "rikfad_diag_kernels.cuh"
#include "rikfad_planner.hpp"

using namespace rikfad;

namespace {

thread_local std::string g_last_error;

int fail(int code, const std::string &msg)
{
    g_last_error = msg;
    return code;
}

int cuda_fail(cudaError_t e, const char *what)
{
    g_last_error = std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
    return RIKFAD_ERR_CUDA;
}

#define RK_CUDA(call, what)                                   \
    do {                                                      \
        cudaError_t e_ = (call);                              \
        if (e_ != cudaSuccess)                                \
            return cuda_fail(e_, what);                       \
    } while (0)

// Every device and page-locked host allocation of the library goes through
// these wrappers.  They count the allocations currently held (a leak check
// for tests) and can be told to report the n-th allocation from now on as
// failed (rikfad_debug_fail_allocation), which exercises the clean-up paths
// without exhausting any memory.
std::atomic<int64_t> g_fail_at{0};
std::atomic<int64_t> g_alloc_calls{0};
std::atomic<int64_t> g_live_allocs{0};

bool injected_failure()
{
    const int64_t n = g_fail_at.load();
    return n > 0 && g_alloc_calls.fetch_add(1) + 1 == n;
}

cudaError_t rk_malloc(void **p, size_t nb)
{
    *p = nullptr;
    if (injected_failure())
        return cudaErrorMemoryAllocation;
    const cudaError_t e = cudaMalloc(p, nb);
    if (e == cudaSuccess)
        ++g_live_allocs;
    else
        *p = nullptr;
    return e;
}

cudaError_t rk_malloc_host(void **p, size_t nb, unsigned flags)
{
    *p = nullptr;
    if (injected_failure())
        return cudaErrorMemoryAllocation;
    const cudaError_t e = cudaHostAlloc(p, nb, flags);
    if (e == cudaSuccess)
        ++g_live_allocs;
    else
        *p = nullptr;
    return e;
}

void rk_free(void *p)
{
    if (p) {
        cudaFree(p);
        --g_live_allocs;
    }
}

void rk_free_host(void *p)
{
    if (p) {
        cudaFreeHost(p);
        --g_live_allocs;
    }
}

int alloc_fail(cudaError_t e, const char *what)
{
    if (e == cudaErrorMemoryAllocation)
        return fail(RIKFAD_ERR_OOM, std::string(what) + " failed: out of memory");
    return cuda_fail(e, what);
}

constexpr uint64_t kImageTag = 0x31444146694b5221ull;   // "!RKiFAD1"
constexpr size_t kImageHeader = 64;

struct ImageHeader {
    uint64_t tag;
    int64_t ntensors;
    double pending_step;
    int64_t fac_floats;
    double alpha, mu, gamma, eps_stab;
};
static_assert(sizeof(ImageHeader) <= kImageHeader, "header too large");

// A device table of per-tensor pointers, uploaded only when it changes.
struct PtrTable {
    int count = 0;                  // pointers in the table
    void **dev = nullptr;
    void **pinned = nullptr;        // staging for the host-to-device copy
    std::vector<void *> cached;
    bool valid = false;
    cudaEvent_t uploaded = nullptr;
};

}  // namespace

namespace rikfad {
// Lets the library's other translation units report through rikfad_last_error.
int report_error(int code, const std::string &msg)
{
    g_last_error = msg;
    return code;
}
}  // namespace rikfad

struct rikfad_handle_s {
    int device = 0;
    bool pageable_ok = false;       // the device reads pageable host memory (host page tables)
    int ntensors = 0;
    int grad_bytes = 4;
    rikfad_hparams hp{};
    Plan plan;
    int max_blocks = 1;
    double pending_step = 0.0;      // h_prev
    std::vector<rikfad_shape> shapes;

    // device memory
    TensorDev *d_tensors = nullptr;
    PanelDev *d_panels = nullptr;
    PieceDev *d_pieces = nullptr;
    int32_t *d_block_piece = nullptr;
    int64_t *d_slot_off = nullptr;
    FinItemDev *d_fin = nullptr;
    float *d_fac = nullptr;
    float *d_rowpart = nullptr;
    float *d_colpart = nullptr;
    float *d_spart = nullptr;
    float *d_den = nullptr;
    float *h_den = nullptr;         // pinned
    int32_t *d_guard = nullptr;     // lowest tensor with a non-finite result (INT32_MAX: none)
    int32_t *h_guard = nullptr;     // mapped page-locked host flag, set by the kernels
    int32_t *h_guard_dev = nullptr; // its device address
    int32_t *d_checks = nullptr;    // failed device checks: count, first code (checked builds)
    size_t workspace = 0;

    PtrTable step_ptrs;             // x | grad | p
    PtrTable canon_ptrs;            // src | dst

    // full iKFAD with shadow R-iKFAD factors (friction diagnostics)
    bool shadow = false;
    float *d_diag_u = nullptr, *d_diag_v = nullptr, *d_diag_w = nullptr, *d_diag_wpart = nullptr;
    double *d_diag_norms = nullptr, *d_diag_upart = nullptr, *d_diag_wsq = nullptr;
    DiagState *d_diag_state = nullptr;
    DiagState *h_diag_state = nullptr;   // pinned

    // in-order ("sweep") schedule, allocated only when selected
    bool sweep = false;
    int sweep_blocks = 0;
    UnitDev *d_units = nullptr;
    NodeDev *d_nodes = nullptr;
    PanelTreeDev *d_trees = nullptr;
    float *d_partials = nullptr;
    int32_t *d_counts = nullptr;    // node counters | tensor counters
    unsigned long long *d_fetch = nullptr;   // unit counter | exit counter

    bool profiling = false;
    std::vector<cudaEvent_t> prof_events;   // 3 per recorded step
    size_t prof_used = 0;
};

namespace {

int check_handle(rikfad_handle h)
{
    if (h == nullptr)
        return fail(RIKFAD_ERR_ARG, "handle is NULL");
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return cuda_fail(e, "cudaGetDevice");
    if (dev != h->device)
        return fail(RIKFAD_ERR_STATE, "current CUDA device " + std::to_string(dev) +
                                          " differs from the handle's device " +
                                          std::to_string(h->device));
    return RIKFAD_OK;
}

template <typename T>
int upload(T **dst, const std::vector<T> &src, size_t &bytes)
{
    *dst = nullptr;
    if (src.empty())
        return RIKFAD_OK;
    const size_t nb = src.size() * sizeof(T);
    cudaError_t e = rk_malloc((void **)dst, nb);
    if (e != cudaSuccess)
        return alloc_fail(e, "cudaMalloc of a plan table");
    bytes += nb;
    RK_CUDA(cudaMemcpy(*dst, src.data(), nb, cudaMemcpyHostToDevice), "cudaMemcpy plan table");
    return RIKFAD_OK;
}

int alloc_zero(float **dst, int64_t floats, size_t &bytes)
{
    *dst = nullptr;
    if (floats <= 0)
        return RIKFAD_OK;
    const size_t nb = (size_t)floats * sizeof(float);
    cudaError_t e = rk_malloc((void **)dst, nb);
    if (e != cudaSuccess)
        return alloc_fail(e, "cudaMalloc");
    bytes += nb;
    RK_CUDA(cudaMemset(*dst, 0, nb), "cudaMemset");
    return RIKFAD_OK;
}

int ptrtable_init(PtrTable &t, int count, size_t &bytes)
{
    t.count = count;
    t.cached.assign(count, nullptr);
    t.valid = false;
    if (count == 0)
        return RIKFAD_OK;
    cudaError_t e = rk_malloc((void **)&t.dev, sizeof(void *) * count);
    if (e != cudaSuccess)
        return alloc_fail(e, "cudaMalloc of the pointer table");
    bytes += sizeof(void *) * count;
    e = rk_malloc_host((void **)&t.pinned, sizeof(void *) * count, cudaHostAllocDefault);
    if (e != cudaSuccess)
        return alloc_fail(e, "cudaHostAlloc of the pointer staging");
    RK_CUDA(cudaEventCreateWithFlags(&t.uploaded, cudaEventDisableTiming), "cudaEventCreate");
    return RIKFAD_OK;
}

void ptrtable_free(PtrTable &t)
{
    rk_free(t.dev);
    rk_free_host(t.pinned);
    if (t.uploaded)
        cudaEventDestroy(t.uploaded);
    t = PtrTable();
}

// Every pointer the kernels will dereference must be memory this device can
// address: its own device memory, page-locked host memory, or pageable host
// memory when the device reads that through the host's page tables
// (pageable_ok).  Checked on the host for the entries that changed, so a
// wrong pointer is an argument error instead of a device fault.  `what`
// names the list entries: entry i is tensor i % ntensors of list i / ntensors.
int check_pointers(const PtrTable &t, const std::vector<void *> &want, int device, bool pageable_ok,
                   int ntensors, const char *const *lists)
{
    for (int i = 0; i < t.count; ++i) {
        if (want[i] == nullptr || (t.valid && want[i] == t.cached[i]))
            continue;
        cudaPointerAttributes a{};
        const cudaError_t e = cudaPointerGetAttributes(&a, want[i]);
        const std::string where = std::string(lists[i / ntensors]) + " pointer of tensor " +
                                  std::to_string(i % ntensors);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(RIKFAD_ERR_ARG, where + " is not an address CUDA recognises");
        }
        if (a.type == cudaMemoryTypeDevice && a.device != device)
            return fail(RIKFAD_ERR_ARG, where + " is memory of device " + std::to_string(a.device) +
                                            ", not of the handle's device " + std::to_string(device));
        if (a.type == cudaMemoryTypeUnregistered && !pageable_ok)
            return fail(RIKFAD_ERR_ARG, where + " is pageable host memory, which this device cannot "
                                                "read; use device or page-locked host memory");
    }
    return RIKFAD_OK;
}

// Make the device table equal `want`; enqueue the copy on `stream` if needed.
int ptrtable_set(PtrTable &t, const std::vector<void *> &want, cudaStream_t stream)
{
    if (t.count == 0 || (t.valid && want == t.cached))
        return RIKFAD_OK;
    // The staging buffer may still feed the previous copy.
    RK_CUDA(cudaEventSynchronize(t.uploaded), "cudaEventSynchronize (pointer staging)");
    std::memcpy(t.pinned, want.data(), sizeof(void *) * t.count);
    RK_CUDA(cudaMemcpyAsync(t.dev, t.pinned, sizeof(void *) * t.count, cudaMemcpyHostToDevice, stream),
            "cudaMemcpyAsync pointer table");
    RK_CUDA(cudaEventRecord(t.uploaded, stream), "cudaEventRecord");
    t.cached = want;
    t.valid = true;
    return RIKFAD_OK;
}

bool hparams_ok(const rikfad_hparams &hp, std::string &why)
{
    if (!(std::isfinite(hp.alpha) && hp.alpha > 0)) {
        why = "alpha must be finite and > 0";
        return false;
    }
    if (!(hp.mu > 0) || std::isnan(hp.mu)) {
        why = "mu must be > 0";
        return false;
    }
    if (!(std::isfinite(hp.gamma) && hp.gamma >= 0)) {
        why = "gamma must be finite and >= 0";
        return false;
    }
    if (!(std::isfinite(hp.eps_stab) && hp.eps_stab >= 0)) {
        why = "eps_stab must be finite and >= 0";
        return false;
    }
    return true;
}

void release(rikfad_handle h)
{
    for (void *p : {(void *)h->d_tensors, (void *)h->d_panels, (void *)h->d_pieces, (void *)h->d_block_piece,
                    (void *)h->d_slot_off, (void *)h->d_fin, (void *)h->d_fac, (void *)h->d_rowpart,
                    (void *)h->d_colpart, (void *)h->d_spart, (void *)h->d_den, (void *)h->d_guard,
                    (void *)h->d_checks, (void *)h->d_diag_u, (void *)h->d_diag_v, (void *)h->d_diag_w,
                    (void *)h->d_diag_wpart, (void *)h->d_diag_norms, (void *)h->d_diag_upart, (void *)h->d_diag_wsq,
                    (void *)h->d_diag_state, (void *)h->d_units, (void *)h->d_nodes,
                    (void *)h->d_trees, (void *)h->d_partials, (void *)h->d_counts, (void *)h->d_fetch})
        rk_free(p);
    rk_free_host(h->h_den);
    rk_free_host(h->h_guard);
    rk_free_host(h->h_diag_state);
    ptrtable_free(h->step_ptrs);
    ptrtable_free(h->canon_ptrs);
    for (cudaEvent_t ev : h->prof_events)
        cudaEventDestroy(ev);
    delete h;
}

// Alignment a tensor's pointers need: 16 bytes for the 8-wide paths,
// natural alignment otherwise.
bool aligned_for(const TensorDev &td, const void *ptr, size_t natural)
{
    const uintptr_t v = (uintptr_t)ptr;
    const bool wide = td.cols == 0 || td.vec;
    return (v % (wide ? 16 : natural)) == 0;
}

int64_t numel(const TensorDev &td) { return td.cols == 0 ? td.rows : td.rows * td.cols; }

// Launch with programmatic stream serialisation: the kernel may begin while
// its predecessor in the stream finishes; it waits (griddepcontrol.wait)
// before touching any data.
template <typename Kern, typename Arg>
cudaError_t launch_pdl(Kern kernel, int nblocks, int nthreads, cudaStream_t s, const Arg &arg)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)nblocks);
    cfg.blockDim = dim3((unsigned)nthreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, arg);
}

template <typename GT>
cudaError_t launch_step(const StepParams &p, bool reuse, bool shadow, int nblocks, cudaStream_t s)
{
    if (shadow)     // full-friction matrices: reuse never applies (no pending factor)
        return launch_pdl(rikfad_step_kernel<GT, false, true>, nblocks, kThreads, s, p);
    if (reuse)
        return launch_pdl(rikfad_step_kernel<GT, true>, nblocks, kThreads, s, p);
    return launch_pdl(rikfad_step_kernel<GT, false>, nblocks, kThreads, s, p);
}

template <typename GT>
void launch_sweep(const StepParams &p, const SweepParams &sp, bool reuse, int nblocks, cudaStream_t s)
{
    if (reuse)
        rikfad_sweep_kernel<GT, true><<<nblocks, kThreads, 0, s>>>(p, sp);
    else
        rikfad_sweep_kernel<GT, false><<<nblocks, kThreads, 0, s>>>(p, sp);
}

CheckBounds bounds(const rikfad_handle h)
{
    const Plan &p = h->plan;
    CheckBounds cb{};
    cb.ntensors = (int32_t)p.tensors.size();
    cb.npanels = (int32_t)p.panels.size();
    cb.npieces = (int32_t)p.pieces.size();
    cb.nblocks = p.nblocks;
    cb.nfin = (int32_t)p.fin_items.size();
    cb.nslots = (int32_t)p.slot_off.size();
    cb.fac_floats = p.fac_floats;
    cb.rowpart_floats = p.rowpart_floats;
    cb.colpart_floats = p.colpart_floats;
    cb.spart_floats = p.spart_floats;
    cb.errors = h->d_checks;
    return cb;
}

Guard guard(const rikfad_handle h) { return Guard{h->d_guard, h->h_guard_dev}; }

// Forget an earlier non-finite report (the device word and the host flag);
// stream-ordered for the device word.
int clear_guard(rikfad_handle h, cudaStream_t stream)
{
    static const int32_t none = INT32_MAX;
    RK_CUDA(cudaMemcpyAsync(h->d_guard, &none, sizeof none, cudaMemcpyHostToDevice, stream),
            "cudaMemcpyAsync guard");
    RK_CUDA(cudaStreamSynchronize(stream), "cudaStreamSynchronize");
    *(volatile int32_t *)h->h_guard = 0;
    return RIKFAD_OK;
}

// RIKFAD_ERR_NONFINITE naming the offending tensor, if the kernels reported
// one (call after the work has completed).
int nonfinite_status(rikfad_handle h, cudaStream_t stream)
{
    if (*(volatile int32_t *)h->h_guard == 0)
        return RIKFAD_OK;
    int32_t first = INT32_MAX;
    RK_CUDA(cudaMemcpyAsync(&first, h->d_guard, sizeof first, cudaMemcpyDeviceToHost, stream),
            "cudaMemcpyAsync guard");
    RK_CUDA(cudaStreamSynchronize(stream), "cudaStreamSynchronize");
    return fail(RIKFAD_ERR_NONFINITE,
                "a step produced a non-finite factor, friction or denominator (first tensor: " +
                    (first == INT32_MAX ? std::string("unknown") : std::to_string(first)) +
                    "); restore the state (rikfad_import_state, rikfad_set_factors) and call "
                    "rikfad_check_finite to clear the report");
}

int finalize(rikfad_handle h, float decay, float gain, int resum_only, cudaStream_t stream)
{
    if (h->plan.fin_items.empty())
        return RIKFAD_OK;
    FinParams f{};
    f.tensors = h->d_tensors;
    f.panels = h->d_panels;
    f.items = h->d_fin;
    f.slot_off = h->d_slot_off;
    f.fac = h->d_fac;
    f.rowpart = h->d_rowpart;
    f.colpart = h->d_colpart;
    f.spart = h->d_spart;
    f.decay = decay;
    f.gain = gain;
    f.resum_only = resum_only;
    f.guard = guard(h);
    f.chk = bounds(h);
    RK_CUDA(launch_pdl(rikfad_finalize_kernel, (int)h->plan.fin_items.size(), kFinThreads, stream, f),
            "launch rikfad_finalize_kernel");
    return RIKFAD_OK;
}

int canonical(rikfad_handle h, const float *const *src, float *const *dst, bool commit,
              cudaStream_t stream)
{
    const int T = h->ntensors;
    std::vector<void *> want(2 * (size_t)T);
    for (int t = 0; t < T; ++t) {
        const TensorDev &td = h->plan.tensors[t];
        const bool empty = numel(td) == 0;
        if (!empty && (src[t] == nullptr || dst[t] == nullptr))
            return fail(RIKFAD_ERR_ARG, "momentum pointer of tensor " + std::to_string(t) + " is NULL");
        if (!empty && (!aligned_for(td, src[t], 4) || !aligned_for(td, dst[t], 4)))
            return fail(RIKFAD_ERR_ALIGN, "momentum pointer of tensor " + std::to_string(t) +
                                              " is not aligned");
        if (!commit && !empty && src[t] == dst[t] && td.cols != 0)
            return fail(RIKFAD_ERR_ARG, "out must not alias p");
        want[t] = (void *)src[t];
        want[T + t] = (void *)dst[t];
    }
    if (h->plan.nblocks > 0) {
        static const char *const lists[2] = {"source momentum", "destination momentum"};
        int rc = check_pointers(h->canon_ptrs, want, h->device, h->pageable_ok, T, lists);
        if (rc)
            return rc;
        rc = ptrtable_set(h->canon_ptrs, want, stream);
        if (rc)
            return rc;
        CanonParams c{};
        c.tensors = h->d_tensors;
        c.panels = h->d_panels;
        c.pieces = h->d_pieces;
        c.block_piece = h->d_block_piece;
        c.src = (const float *const *)h->canon_ptrs.dev;
        c.dst = (float *const *)(h->canon_ptrs.dev + T);
        c.fac = h->d_fac;
        c.spart = h->d_spart;
        c.ex_prev = (float)(-0.5 * h->pending_step * M_LOG2E);
        c.damp_prev = (float)std::exp(-h->hp.gamma * h->pending_step);
        c.eps = (float)h->hp.eps_stab;
        c.chk = bounds(h);
        RK_CUDA(launch_pdl(rikfad_canonical_kernel, h->plan.nblocks, kThreads, stream, c),
                "launch rikfad_canonical_kernel");
    }
    if (commit)
        h->pending_step = 0.0;
    return RIKFAD_OK;
}

int create_impl(const rikfad_shape *shapes, int ntensors, const rikfad_hparams *hp, int grad_dtype,
                rikfad_handle *out, bool shadow = false);

}  // namespace

extern "C" {

RIKFAD_API const char *rikfad_last_error(void) { return g_last_error.c_str(); }

RIKFAD_API int rikfad_abi_version(void) { return 1; }

RIKFAD_API size_t rikfad_state_bytes_for(const rikfad_shape *shapes, int ntensors, int include_momentum)
{
    if (!check_shapes(shapes, ntensors).empty())
        return 0;
    size_t scalars = 0;
    for (int t = 0; t < ntensors; ++t) {
        const int64_t m = shapes[t].rows, n = shapes[t].cols;
        if (n == 0)
            scalars += (size_t)m + (include_momentum ? (size_t)m : 0);
        else
            scalars += (size_t)(m + n) + (include_momentum ? (size_t)(m * n) : 0);
    }
    return scalars * sizeof(float);
}

RIKFAD_API int64_t rikfad_plan_query(const rikfad_shape *shapes, int ntensors, int grad_dtype,
                                     int nctas, int64_t *out, int64_t cap)
{
    if (grad_dtype != RIKFAD_GRAD_F32 && grad_dtype != RIKFAD_GRAD_BF16)
        return fail(RIKFAD_ERR_ARG, "grad_dtype must be RIKFAD_GRAD_F32 or RIKFAD_GRAD_BF16");
    if (cap > 0 && out == nullptr)
        return fail(RIKFAD_ERR_ARG, "out is NULL");
    Plan plan;
    std::string err = build_plan(shapes, ntensors, grad_dtype == RIKFAD_GRAD_BF16 ? 2 : 4, nctas, plan);
    if (!err.empty())
        return fail(RIKFAD_ERR_ARG, err);
    int64_t row = 0;
    for (int b = 0; b < plan.nblocks; ++b) {
        for (int q = plan.block_piece[b]; q < plan.block_piece[b + 1]; ++q, ++row) {
            if (row >= cap)
                continue;
            const PieceDev &pc = plan.pieces[q];
            int64_t *r = out + row * 8;
            r[0] = b;
            r[1] = pc.tensor;
            r[2] = pc.kind;
            r[3] = pc.kind == kMatrixRows ? plan.panels[pc.panel].col0 : 0;
            r[4] = pc.kind == kMatrixRows ? plan.panels[pc.panel].width : 0;
            r[5] = pc.begin;
            r[6] = pc.end;
            r[7] = pc.slot;
        }
    }
    return row;
}

RIKFAD_API int rikfad_create(const rikfad_shape *shapes, int ntensors, const rikfad_hparams *hp,
                             int grad_dtype, rikfad_handle *out)
{
    return create_impl(shapes, ntensors, hp, grad_dtype, out);
}

RIKFAD_API int rikfad_create_ikfad_shadow(const rikfad_shape *shapes, int ntensors,
                                          const rikfad_hparams *hp, int grad_dtype, rikfad_handle *out)
{
    return create_impl(shapes, ntensors, hp, grad_dtype, out, true);
}

RIKFAD_API int rikfad_create_ikfad(const rikfad_shape *shapes, int ntensors, const rikfad_hparams *hp,
                                   int grad_dtype, rikfad_handle *out)
{
    if (out == nullptr)
        return fail(RIKFAD_ERR_ARG, "out is NULL");
    *out = nullptr;
    std::string why = check_shapes(shapes, ntensors);
    if (!why.empty())
        return fail(RIKFAD_ERR_ARG, why);
    // Full friction: every tensor follows the element-wise rule over its
    // rows x cols elements.
    std::vector<rikfad_shape> flat(ntensors);
    for (int t = 0; t < ntensors; ++t) {
        flat[t].rows = shapes[t].cols == 0 ? shapes[t].rows : shapes[t].rows * shapes[t].cols;
        flat[t].cols = 0;
    }
    return create_impl(flat.data(), ntensors, hp, grad_dtype, out);
}

}  // extern "C"

namespace {

int create_impl(const rikfad_shape *shapes, int ntensors, const rikfad_hparams *hp, int grad_dtype,
                rikfad_handle *out, bool shadow)
{
    if (out == nullptr)
        return fail(RIKFAD_ERR_ARG, "out is NULL");
    *out = nullptr;
    if (hp == nullptr)
        return fail(RIKFAD_ERR_ARG, "hp is NULL");
    std::string why;
    if (!hparams_ok(*hp, why))
        return fail(RIKFAD_ERR_ARG, why);
    if (grad_dtype != RIKFAD_GRAD_F32 && grad_dtype != RIKFAD_GRAD_BF16)
        return fail(RIKFAD_ERR_ARG, "grad_dtype must be RIKFAD_GRAD_F32 or RIKFAD_GRAD_BF16");
    why = check_shapes(shapes, ntensors);
    if (!why.empty())
        return fail(RIKFAD_ERR_ARG, why);

    int dev = 0, sms = 0, occ = 0;
    RK_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
    RK_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev), "cudaDeviceGetAttribute");
    int pageable = 0;
    RK_CUDA(cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, dev), "cudaDeviceGetAttribute");
    // Persistent grid: as many blocks as can be resident at once.
    int occ_min = 1 << 30;
    const void *kernels[6] = {(const void *)rikfad_step_kernel<float, true>,
                              (const void *)rikfad_step_kernel<float, false>,
                              (const void *)rikfad_step_kernel<__nv_bfloat16, true>,
                              (const void *)rikfad_step_kernel<__nv_bfloat16, false>,
                              (const void *)rikfad_step_kernel<float, false, true>,
                              (const void *)rikfad_step_kernel<__nv_bfloat16, false, true>};
    for (const void *k : kernels) {
        RK_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k, kThreads, 0),
                "cudaOccupancyMaxActiveBlocksPerMultiprocessor");
        occ_min = std::min(occ_min, occ);
    }
    if (occ_min < 1)
        return fail(RIKFAD_ERR_CUDA, "step kernel cannot be resident on this device");
    // Static schedule by default; RIKFAD_SCHEDULE=sweep selects the in-order
    // one-kernel schedule (slower on GB300, see rikfad_sweep.cuh), whose
    // units, trees and partials are built and allocated only then.
    const char *env = std::getenv("RIKFAD_SCHEDULE");
    const bool sweep = env && std::strcmp(env, "sweep") == 0 && !shadow;
    int occ_sweep = 1 << 30;
    if (sweep) {
        const void *sweep_kernels[4] = {(const void *)rikfad_sweep_kernel<float, true>,
                                        (const void *)rikfad_sweep_kernel<float, false>,
                                        (const void *)rikfad_sweep_kernel<__nv_bfloat16, true>,
                                        (const void *)rikfad_sweep_kernel<__nv_bfloat16, false>};
        for (const void *k : sweep_kernels) {
            RK_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k, kThreads, 0),
                    "cudaOccupancyMaxActiveBlocksPerMultiprocessor");
            occ_sweep = std::min(occ_sweep, occ);
        }
        if (occ_sweep < 1)
            return fail(RIKFAD_ERR_CUDA, "sweep kernel cannot be resident on this device");
    }

    rikfad_handle h = new rikfad_handle_s();
    h->device = dev;
    h->pageable_ok = pageable != 0;
    h->ntensors = ntensors;
    h->grad_bytes = grad_dtype == RIKFAD_GRAD_BF16 ? 2 : 4;
    h->hp = *hp;
    h->shapes.assign(shapes, shapes + ntensors);
    h->max_blocks = sms * occ_min;
    h->shadow = shadow;
    why = build_plan(shapes, ntensors, h->grad_bytes, h->max_blocks, h->plan, shadow);
    if (!why.empty()) {
        delete h;
        return fail(RIKFAD_ERR_ARG, why);
    }
    h->sweep = sweep;
    if (sweep) {
        build_sweep(shapes, ntensors, h->plan);
        h->sweep_blocks = sms * occ_sweep;
    }
    const Plan &p = h->plan;
    size_t ws = 0;
    int rc = RIKFAD_OK;
    if (!rc) rc = upload(&h->d_tensors, p.tensors, ws);
    if (!rc) rc = upload(&h->d_panels, p.panels, ws);
    if (!rc) rc = upload(&h->d_pieces, p.pieces, ws);
    if (!rc) rc = upload(&h->d_block_piece, p.block_piece, ws);
    if (!rc) rc = upload(&h->d_slot_off, p.slot_off, ws);
    if (!rc) rc = upload(&h->d_fin, p.fin_items, ws);
    size_t state = 0;
    if (!rc) rc = alloc_zero(&h->d_fac, p.fac_floats, state);
    if (!rc) rc = alloc_zero(&h->d_rowpart, p.rowpart_floats, ws);
    if (!rc) rc = alloc_zero(&h->d_colpart, p.colpart_floats, ws);
    if (!rc) rc = alloc_zero(&h->d_spart, p.spart_floats, ws);
    if (!rc) rc = alloc_zero(&h->d_den, std::max(ntensors, 1), ws);
    if (!rc) {
        cudaError_t e = rk_malloc_host((void **)&h->h_den, sizeof(float) * std::max(ntensors, 1),
                                       cudaHostAllocDefault);
        if (e != cudaSuccess)
            rc = alloc_fail(e, "cudaHostAlloc of the denominator read-back");
    }
    // Non-finite guard: a device word (lowest offending tensor) and a mapped
    // host flag the kernels set, so rikfad_step sees a report without waiting.
    if (!rc) rc = alloc_zero((float **)&h->d_guard, 1, ws);
    if (!rc) {
        cudaError_t e = rk_malloc_host((void **)&h->h_guard, sizeof(int32_t), cudaHostAllocMapped);
        if (e != cudaSuccess)
            rc = alloc_fail(e, "cudaHostAlloc of the non-finite flag");
        else if ((e = cudaHostGetDevicePointer((void **)&h->h_guard_dev, h->h_guard, 0)) != cudaSuccess)
            rc = cuda_fail(e, "cudaHostGetDevicePointer");
    }
    if (!rc) rc = alloc_zero((float **)&h->d_checks, 2, ws);
    if (!rc && sweep) {
        rc = upload(&h->d_units, p.units, ws);
        if (!rc) rc = upload(&h->d_nodes, p.nodes, ws);
        if (!rc) rc = upload(&h->d_trees, p.trees, ws);
        if (!rc) rc = alloc_zero(&h->d_partials, p.partial_floats, ws);
        if (!rc) rc = alloc_zero((float **)&h->d_counts, (int64_t)p.nodes.size() + ntensors + 1, ws);
        if (!rc) rc = alloc_zero((float **)&h->d_fetch, 4, ws);
    }
    if (!rc && shadow) {
        int64_t max_m = 1, max_n = 1, max_parts = 1;
        for (const TensorDev &td : p.tensors)
            if (td.cols > 0) {
                max_m = std::max(max_m, td.rows);
                max_n = std::max(max_n, td.cols);
                max_parts = std::max<int64_t>(max_parts, (td.rows + diag_rows_per_group(td.rows) - 1) /
                                                             diag_rows_per_group(td.rows));
            }
        rc = alloc_zero(&h->d_diag_u, max_m, ws);
        if (!rc) rc = alloc_zero(&h->d_diag_v, max_n, ws);
        if (!rc) rc = alloc_zero(&h->d_diag_w, max_n, ws);
        if (!rc) rc = alloc_zero(&h->d_diag_wpart, max_parts * max_n, ws);
        if (!rc) rc = alloc_zero((float **)&h->d_diag_norms, 4 * ((max_m + kWarps - 1) / kWarps), ws);
        if (!rc) rc = alloc_zero((float **)&h->d_diag_upart, 2 * ((max_m + kWarps - 1) / kWarps), ws);
        if (!rc) rc = alloc_zero((float **)&h->d_diag_wsq, 2 * ((max_n + 31) / 32), ws);
        if (!rc) rc = alloc_zero((float **)&h->d_diag_state, (int64_t)(sizeof(DiagState) / sizeof(float)), ws);
        if (!rc) {
            cudaError_t e = rk_malloc_host((void **)&h->h_diag_state, sizeof(DiagState), cudaHostAllocDefault);
            if (e != cudaSuccess)
                rc = alloc_fail(e, "cudaHostAlloc of the diagnostic state read-back");
        }
    }
    if (!rc) rc = ptrtable_init(h->step_ptrs, 3 * ntensors, ws);
    if (!rc) rc = ptrtable_init(h->canon_ptrs, 2 * ntensors, ws);
    if (!rc) rc = clear_guard(h, 0);
    if (!rc) {
        cudaError_t e = cudaDeviceSynchronize();
        if (e != cudaSuccess)
            rc = cuda_fail(e, "cudaDeviceSynchronize after create");
    }
    if (rc) {
        std::string msg = g_last_error;
        release(h);
        g_last_error = msg;
        return rc;
    }
    h->workspace = ws;
    *out = h;
    return RIKFAD_OK;
}

}  // namespace

extern "C" {

RIKFAD_API void rikfad_destroy(rikfad_handle h)
{
    if (h == nullptr)
        return;
    const int dev = h->device;
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != dev)
        cudaSetDevice(dev);
    cudaDeviceSynchronize();
    release(h);
    if (cur >= 0 && cur != dev)
        cudaSetDevice(cur);
}

RIKFAD_API int rikfad_step(rikfad_handle h, double step, float *const *x, const void *const *grad,
                           float *const *p, void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (!(std::isfinite(step) && step > 0))
        return fail(RIKFAD_ERR_ARG, "step must be finite and > 0");
    const int T = h->ntensors;
    if (T > 0 && (x == nullptr || grad == nullptr || p == nullptr))
        return fail(RIKFAD_ERR_ARG, "pointer array is NULL");
    // A non-finite result reported by an earlier step (seen without waiting):
    // nothing more is enqueued until the report is cleared.
    if (*(volatile int32_t *)h->h_guard != 0)
        return fail(RIKFAD_ERR_NONFINITE, "an earlier step produced a non-finite factor, friction or "
                                          "denominator; rikfad_check_finite names the tensor and clears "
                                          "the report");
    const double decay_d = std::exp(-h->hp.alpha * step);
    const double gain_d = std::isinf(h->hp.mu) ? 0.0 : -std::expm1(-h->hp.alpha * step) / (h->hp.mu * h->hp.alpha);
    if (!std::isfinite((float)gain_d))
        return fail(RIKFAD_ERR_ARG, "(1 - e^{-alpha h})/(mu alpha) overflows float32");
    std::vector<void *> want(3 * (size_t)T);
    for (int t = 0; t < T; ++t) {
        const TensorDev &td = h->plan.tensors[t];
        if (numel(td) == 0) {
            want[t] = want[T + t] = want[2 * T + t] = nullptr;
            continue;
        }
        if (x[t] == nullptr || grad[t] == nullptr || p[t] == nullptr)
            return fail(RIKFAD_ERR_ARG, "pointer of tensor " + std::to_string(t) + " is NULL");
        if (!aligned_for(td, x[t], 4) || !aligned_for(td, p[t], 4) ||
            !aligned_for(td, grad[t], (size_t)h->grad_bytes))
            return fail(RIKFAD_ERR_ALIGN, "pointer of tensor " + std::to_string(t) +
                                              " is not 16-byte aligned");
        want[t] = x[t];
        want[T + t] = (void *)grad[t];
        want[2 * T + t] = p[t];
    }
    cudaStream_t s = (cudaStream_t)stream;
    RK_CUDA(cudaPeekAtLastError(), "earlier CUDA error");
    if (h->plan.nblocks > 0) {
        static const char *const lists[3] = {"x", "grad", "p"};
        rc = check_pointers(h->step_ptrs, want, h->device, h->pageable_ok, T, lists);
        if (rc)
            return rc;
        rc = ptrtable_set(h->step_ptrs, want, s);
        if (rc)
            return rc;
    }
    cudaEvent_t *ev = nullptr;
    if (h->profiling) {
        if (h->prof_used + 3 > h->prof_events.size()) {
            for (int i = 0; i < 3; ++i) {
                cudaEvent_t e;
                RK_CUDA(cudaEventCreate(&e), "cudaEventCreate");
                h->prof_events.push_back(e);
            }
        }
        ev = &h->prof_events[h->prof_used];
        h->prof_used += 3;
        RK_CUDA(cudaEventRecord(ev[0], s), "cudaEventRecord");
    }
    // Static schedule: the step kernel (if any element) then the finalise
    // kernel.  Sweep schedule: one kernel does both (it also runs when only
    // matrices without rows are present: their C still decays).
    const bool run_kernel = h->sweep ? !h->plan.units.empty() : h->plan.nblocks > 0;
    if (run_kernel) {
        StepParams a{};
        a.tensors = h->d_tensors;
        a.panels = h->d_panels;
        a.pieces = h->d_pieces;
        a.block_piece = h->d_block_piece;
        a.xptr = (float *const *)h->step_ptrs.dev;
        a.gptr = (const void *const *)(h->step_ptrs.dev + T);
        a.pptr = (float *const *)(h->step_ptrs.dev + 2 * T);
        a.fac = h->d_fac;
        a.rowpart = h->d_rowpart;
        a.colpart = h->d_colpart;
        a.spart = h->d_spart;
        a.h = (float)step;
        a.ex_cur = (float)(-0.5 * step * M_LOG2E);
        a.ex_prev = (float)(-0.5 * h->pending_step * M_LOG2E);
        a.damp_prev = (float)std::exp(-h->hp.gamma * h->pending_step);
        a.damp_cur = (float)std::exp(-h->hp.gamma * step);
        a.decay = (float)decay_d;
        a.gain = (float)gain_d;
        a.eps = (float)h->hp.eps_stab;
        a.guard = guard(h);
        a.chk = bounds(h);
        const bool reuse = (step == h->pending_step);
        if (h->sweep) {
            SweepParams sp{};
            sp.units = h->d_units;
            sp.nodes = h->d_nodes;
            sp.trees = h->d_trees;
            sp.nunits = (int64_t)h->plan.units.size();
            sp.partials = h->d_partials;
            sp.spart = h->d_spart;
            sp.node_count = h->d_counts;
            sp.tensor_count = h->d_counts + h->plan.nodes.size();
            sp.fetch = h->d_fetch;
            sp.exits = reinterpret_cast<unsigned int *>(h->d_fetch + 1);
            if (h->grad_bytes == 2)
                launch_sweep<__nv_bfloat16>(a, sp, reuse, h->sweep_blocks, s);
            else
                launch_sweep<float>(a, sp, reuse, h->sweep_blocks, s);
            RK_CUDA(cudaGetLastError(), "launch rikfad_sweep_kernel");
        } else {
            if (h->grad_bytes == 2)
                RK_CUDA(launch_step<__nv_bfloat16>(a, reuse, h->shadow, h->plan.nblocks, s),
                        "launch rikfad_step_kernel");
            else
                RK_CUDA(launch_step<float>(a, reuse, h->shadow, h->plan.nblocks, s), "launch rikfad_step_kernel");
        }
    }
    if (ev)
        RK_CUDA(cudaEventRecord(ev[1], s), "cudaEventRecord");
    if (!h->sweep) {
        rc = finalize(h, (float)decay_d, (float)gain_d, 0, s);
        if (rc)
            return rc;
    }
    if (ev)
        RK_CUDA(cudaEventRecord(ev[2], s), "cudaEventRecord");
    h->pending_step = step;
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_materialize(rikfad_handle h, float *const *p, void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (h->ntensors > 0 && p == nullptr)
        return fail(RIKFAD_ERR_ARG, "p is NULL");
    return canonical(h, (const float *const *)p, p, true, (cudaStream_t)stream);
}

RIKFAD_API int rikfad_canonical_momentum(rikfad_handle h, const float *const *p, float *const *out,
                                         void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (h->ntensors > 0 && (p == nullptr || out == nullptr))
        return fail(RIKFAD_ERR_ARG, "p or out is NULL");
    return canonical(h, p, out, false, (cudaStream_t)stream);
}

RIKFAD_API size_t rikfad_state_bytes(rikfad_handle h, int include_momentum)
{
    if (h == nullptr)
        return 0;
    size_t b = rikfad_state_bytes_for(h->shapes.data(), h->ntensors, include_momentum);
    if (h->shadow)      // plus the element-wise friction of every matrix
        for (const rikfad_shape &sh : h->shapes)
            if (sh.cols > 0)
                b += sizeof(float) * (size_t)(sh.rows * sh.cols);
    return b;
}

RIKFAD_API size_t rikfad_workspace_bytes(rikfad_handle h) { return h ? h->workspace : 0; }

RIKFAD_API double rikfad_pending_step(rikfad_handle h) { return h ? h->pending_step : 0.0; }

RIKFAD_API int rikfad_get_factors(rikfad_handle h, int t, float *R_host, float *C_host)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (t < 0 || t >= h->ntensors)
        return fail(RIKFAD_ERR_ARG, "tensor index out of range");
    const TensorDev &td = h->plan.tensors[t];
    RK_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
    if (R_host && td.rows > 0)
        RK_CUDA(cudaMemcpy(R_host, h->d_fac + td.fac_off, sizeof(float) * td.rows, cudaMemcpyDeviceToHost),
                "cudaMemcpy factors");
    if (C_host && td.cols > 0)
        RK_CUDA(cudaMemcpy(C_host, h->d_fac + td.fac_off + td.rows, sizeof(float) * td.cols,
                           cudaMemcpyDeviceToHost),
                "cudaMemcpy factors");
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_set_factors(rikfad_handle h, int t, const float *R_host, const float *C_host)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (t < 0 || t >= h->ntensors)
        return fail(RIKFAD_ERR_ARG, "tensor index out of range");
    const TensorDev &td = h->plan.tensors[t];
    const int64_t nr = td.rows, nc = td.cols;
    for (int64_t i = 0; R_host && i < nr; ++i)
        if (!(std::isfinite(R_host[i]) && R_host[i] >= 0))
            return fail(RIKFAD_ERR_ARG, "factor values must be finite and >= 0");
    for (int64_t j = 0; C_host && j < nc; ++j)
        if (!(std::isfinite(C_host[j]) && C_host[j] >= 0))
            return fail(RIKFAD_ERR_ARG, "factor values must be finite and >= 0");
    RK_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
    rc = clear_guard(h, 0);
    if (rc)
        return rc;
    if (R_host && nr > 0)
        RK_CUDA(cudaMemcpy(h->d_fac + td.fac_off, R_host, sizeof(float) * nr, cudaMemcpyHostToDevice),
                "cudaMemcpy factors");
    if (C_host && nc > 0)
        RK_CUDA(cudaMemcpy(h->d_fac + td.fac_off + nr, C_host, sizeof(float) * nc, cudaMemcpyHostToDevice),
                "cudaMemcpy factors");
    rc = finalize(h, 1.f, 0.f, 1, 0);
    if (rc)
        return rc;
    RK_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_read_denominators(rikfad_handle h, float *host_out, void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (host_out == nullptr)
        return fail(RIKFAD_ERR_ARG, "host_out is NULL");
    const int T = h->ntensors;
    if (T == 0)
        return RIKFAD_OK;
    cudaStream_t s = (cudaStream_t)stream;
    DenParams d{h->d_tensors, h->d_spart, h->d_den, T, bounds(h)};
    const int warps = 8;
    rikfad_denominators_kernel<<<(T + warps - 1) / warps, 32 * warps, 0, s>>>(d);
    RK_CUDA(cudaGetLastError(), "launch rikfad_denominators_kernel");
    RK_CUDA(cudaMemcpyAsync(h->h_den, h->d_den, sizeof(float) * T, cudaMemcpyDeviceToHost, s),
            "cudaMemcpyAsync denominators");
    RK_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
    std::memcpy(host_out, h->h_den, sizeof(float) * T);
    return nonfinite_status(h, s);
}

RIKFAD_API int rikfad_enqueue_denominators(rikfad_handle h, float *host_out, void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (host_out == nullptr)
        return fail(RIKFAD_ERR_ARG, "host_out is NULL");
    const int T = h->ntensors;
    if (T == 0)
        return RIKFAD_OK;
    cudaStream_t s = (cudaStream_t)stream;
    RK_CUDA(cudaPeekAtLastError(), "earlier CUDA error");
    // Page-locked memory mapped into the device's address space takes the
    // kernel's stores directly, so no copy sits between this step's finalise
    // and the next step's kernels (PDL launches chain through); other host
    // memory gets a copy from the device buffer.
    float *direct = nullptr;
    if (cudaHostGetDevicePointer((void **)&direct, host_out, 0) != cudaSuccess) {
        cudaGetLastError();     // not mapped: clear the query's error
        direct = nullptr;
    }
    DenParams d{h->d_tensors, h->d_spart, direct ? direct : h->d_den, T, bounds(h)};
    const int warps = 8;
    RK_CUDA(launch_pdl(rikfad_denominators_kernel, (T + warps - 1) / warps, 32 * warps, s, d),
            "launch rikfad_denominators_kernel");
    if (!direct)
        RK_CUDA(cudaMemcpyAsync(host_out, h->d_den, sizeof(float) * T, cudaMemcpyDeviceToHost, s),
                "cudaMemcpyAsync denominators");
    return RIKFAD_OK;
}

RIKFAD_API size_t rikfad_state_image_bytes(rikfad_handle h)
{
    return h ? kImageHeader + sizeof(float) * (size_t)h->plan.fac_floats : 0;
}

RIKFAD_API int rikfad_export_state(rikfad_handle h, void *dev_dst, void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (dev_dst == nullptr)
        return fail(RIKFAD_ERR_ARG, "dev_dst is NULL");
    if ((uintptr_t)dev_dst % 16)
        return fail(RIKFAD_ERR_ALIGN, "dev_dst must be 16-byte aligned");
    cudaStream_t s = (cudaStream_t)stream;
    ImageHeader hd{};
    hd.tag = kImageTag;
    hd.ntensors = h->ntensors;
    hd.pending_step = h->pending_step;
    hd.fac_floats = h->plan.fac_floats;
    hd.alpha = h->hp.alpha;
    hd.mu = h->hp.mu;
    hd.gamma = h->hp.gamma;
    hd.eps_stab = h->hp.eps_stab;
    // The header is small; a synchronous copy keeps the host struct's lifetime simple.
    RK_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
    RK_CUDA(cudaMemcpy(dev_dst, &hd, sizeof hd, cudaMemcpyHostToDevice), "cudaMemcpy image header");
    if (h->plan.fac_floats > 0)
        RK_CUDA(cudaMemcpyAsync((char *)dev_dst + kImageHeader, h->d_fac, sizeof(float) * h->plan.fac_floats,
                                cudaMemcpyDeviceToDevice, s),
                "cudaMemcpyAsync image");
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_import_state(rikfad_handle h, const void *dev_src, void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (dev_src == nullptr)
        return fail(RIKFAD_ERR_ARG, "dev_src is NULL");
    if ((uintptr_t)dev_src % 16)
        return fail(RIKFAD_ERR_ALIGN, "dev_src must be 16-byte aligned");
    cudaStream_t s = (cudaStream_t)stream;
    ImageHeader hd{};
    RK_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
    RK_CUDA(cudaMemcpy(&hd, dev_src, sizeof hd, cudaMemcpyDeviceToHost), "cudaMemcpy image header");
    if (hd.tag != kImageTag)
        return fail(RIKFAD_ERR_ARG, "not an R-iKFAD state image");
    if (hd.ntensors != h->ntensors || hd.fac_floats != h->plan.fac_floats)
        return fail(RIKFAD_ERR_ARG, "state image was exported for other shapes");
    if (hd.alpha != h->hp.alpha || hd.mu != h->hp.mu || hd.gamma != h->hp.gamma ||
        hd.eps_stab != h->hp.eps_stab)
        return fail(RIKFAD_ERR_ARG, "state image was exported with other hyperparameters");
    rc = clear_guard(h, s);
    if (rc)
        return rc;
    if (h->plan.fac_floats > 0)
        RK_CUDA(cudaMemcpyAsync(h->d_fac, (const char *)dev_src + kImageHeader,
                                sizeof(float) * h->plan.fac_floats, cudaMemcpyDeviceToDevice, s),
                "cudaMemcpyAsync image");
    rc = finalize(h, 1.f, 0.f, 1, s);
    if (rc)
        return rc;
    h->pending_step = hd.pending_step;
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_profile_enable(rikfad_handle h, int enable)
{
    if (h == nullptr)
        return fail(RIKFAD_ERR_ARG, "handle is NULL");
    h->profiling = enable != 0;
    h->prof_used = 0;
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_profile_read(rikfad_handle h, double *step_kernel_ms, double *finalize_kernel_ms,
                                   int64_t *steps)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    double a = 0, b = 0;
    for (size_t i = 0; i + 3 <= h->prof_used; i += 3) {
        float t1 = 0, t2 = 0;
        RK_CUDA(cudaEventSynchronize(h->prof_events[i + 2]), "cudaEventSynchronize");
        RK_CUDA(cudaEventElapsedTime(&t1, h->prof_events[i], h->prof_events[i + 1]), "cudaEventElapsedTime");
        RK_CUDA(cudaEventElapsedTime(&t2, h->prof_events[i + 1], h->prof_events[i + 2]),
                "cudaEventElapsedTime");
        a += t1;
        b += t2;
    }
    if (step_kernel_ms)
        *step_kernel_ms = a;
    if (finalize_kernel_ms)
        *finalize_kernel_ms = b;
    if (steps)
        *steps = (int64_t)(h->prof_used / 3);
    h->prof_used = 0;
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_launches_per_step(rikfad_handle h)
{
    if (h == nullptr)
        return 0;
    if (h->sweep)
        return h->plan.units.empty() ? 0 : 1;
    return (h->plan.nblocks > 0 ? 1 : 0) + (h->plan.fin_items.empty() ? 0 : 1);
}

RIKFAD_API int rikfad_get_friction(rikfad_handle h, int t, float *xi_host)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (t < 0 || t >= h->ntensors)
        return fail(RIKFAD_ERR_ARG, "tensor index out of range");
    const TensorDev &td = h->plan.tensors[t];
    int64_t off, count;
    if (td.cols == 0) {
        off = td.fac_off;
        count = td.rows;
    } else if (td.full) {
        off = td.xi_off;
        count = td.rows * td.cols;
    } else {
        return fail(RIKFAD_ERR_ARG, "tensor " + std::to_string(t) + " has rank-1 friction (use rikfad_get_factors)");
    }
    if (count > 0 && xi_host == nullptr)
        return fail(RIKFAD_ERR_ARG, "xi_host is NULL");
    RK_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
    if (count > 0)
        RK_CUDA(cudaMemcpy(xi_host, h->d_fac + off, sizeof(float) * count, cudaMemcpyDeviceToHost),
                "cudaMemcpy friction");
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_friction_diagnostics(rikfad_handle h, int t, int max_iters, double tol, double *out,
                                           void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    if (!h->shadow)
        return fail(RIKFAD_ERR_STATE, "friction diagnostics need a handle from rikfad_create_ikfad_shadow");
    if (t < 0 || t >= h->ntensors || h->plan.tensors[t].cols == 0)
        return fail(RIKFAD_ERR_ARG, "tensor index is not a matrix");
    if (out == nullptr || max_iters < 1 || !(tol >= 0))
        return fail(RIKFAD_ERR_ARG, "out is NULL, max_iters < 1 or tol < 0");
    const TensorDev &td = h->plan.tensors[t];
    const int64_t m = td.rows, n = td.cols;
    for (int k = 0; k < 6; ++k)
        out[k] = 0.0;
    if (m == 0)
        return RIKFAD_OK;
    cudaStream_t s = (cudaStream_t)stream;
    const float *xi = h->d_fac + td.xi_off;
    const float *R = h->d_fac + td.fac_off;
    const float *C = h->d_fac + td.fac_off + m;
    // 1^T R exactly as the step kernels form it, then inv, the start vector
    // (C normalised) and a cleared iteration state, all on the device.
    DenParams d{h->d_tensors, h->d_spart, h->d_den, h->ntensors, bounds(h)};
    rikfad_denominators_kernel<<<(h->ntensors + kWarps - 1) / kWarps, kThreads, 0, s>>>(d);
    rikfad_diag_setup_kernel<<<1, kDiagFinThreads, 0, s>>>(h->d_den + t, (float)h->hp.eps_stab, C, n,
                                                           h->d_diag_v, h->d_diag_state);
    // ||xi||^2 and ||xi - xi~||^2
    const int nb_rows = (int)((m + kWarps - 1) / kWarps);
    rikfad_diag_norms_kernel<<<nb_rows, kThreads, 0, s>>>(xi, m, n, R, C, h->d_diag_state, h->d_diag_norms);
    RK_CUDA(cudaGetLastError(), "launch diagnostic set-up kernels");
    // sigma_1 by power iteration on xi^T xi, starting from C (the shadow
    // column factor, close to the top right singular vector).  A batch of
    // kBatch iterations (four kernels each) and the read-back of the state
    // record are captured once into a CUDA graph, which is replayed until
    // the iteration is done; after convergence the remaining kernels of a
    // batch return at once.  One graph launch replaces 32 kernel launches.
    const int nb_t = (int)((m + diag_rows_per_group(m) - 1) / diag_rows_per_group(m));
    const dim3 grid_t((unsigned)nb_t, (unsigned)((n + kThreads - 1) / kThreads));
    const int nb_c = (int)((n + 31) / 32);
    constexpr int kBatch = 8;
    DiagState &st = *h->h_diag_state;
    cudaStream_t cs = nullptr;
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    auto cleanup = [&]() {
        if (exec)
            cudaGraphExecDestroy(exec);
        if (graph)
            cudaGraphDestroy(graph);
        if (cs)
            cudaStreamDestroy(cs);
    };
    cudaError_t e = cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking);
    if (e == cudaSuccess)
        e = cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal);
    if (e == cudaSuccess) {
        for (int b = 0; b < kBatch; ++b) {
            rikfad_diag_matvec_kernel<<<nb_rows, kThreads, 0, cs>>>(xi, m, n, h->d_diag_v, h->d_diag_u,
                                                                    h->d_diag_upart, h->d_diag_state);
            rikfad_diag_matvec_t_kernel<<<grid_t, kThreads, 0, cs>>>(xi, m, n, h->d_diag_u, h->d_diag_wpart,
                                                                     h->d_diag_state);
            rikfad_diag_colsum_kernel<<<nb_c, kDiagFinThreads, 0, cs>>>(h->d_diag_wpart, nb_t, n, h->d_diag_w,
                                                                 h->d_diag_wsq, h->d_diag_state);
            rikfad_diag_iterate_kernel<<<1, kDiagFinThreads, 0, cs>>>(h->d_diag_w, n, h->d_diag_wsq, nb_c,
                                                                     h->d_diag_upart, nb_rows, h->d_diag_v,
                                                                     h->d_diag_state, tol, max_iters);
        }
        cudaMemcpyAsync(h->h_diag_state, h->d_diag_state, sizeof(DiagState), cudaMemcpyDeviceToHost, cs);
        e = cudaStreamEndCapture(cs, &graph);
    }
    if (e == cudaSuccess)
        e = cudaGraphInstantiate(&exec, graph, 0);
    if (e != cudaSuccess) {
        cleanup();
        return cuda_fail(e, "capture of the power iteration");
    }
    for (int enqueued = 0; enqueued < max_iters; enqueued += kBatch) {
        e = cudaGraphLaunch(exec, s);
        if (e == cudaSuccess)
            e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) {
            cleanup();
            return cuda_fail(e, "power iteration");
        }
        if (st.done)
            break;
    }
    cleanup();
    std::vector<double> parts(2 * (size_t)nb_rows);
    RK_CUDA(cudaMemcpyAsync(parts.data(), h->d_diag_norms, sizeof(double) * parts.size(), cudaMemcpyDeviceToHost, s),
            "cudaMemcpyAsync");
    RK_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
    double f2 = 0.0, e2 = 0.0;
    for (int b = 0; b < nb_rows; ++b) {
        f2 += parts[2 * b];
        e2 += parts[2 * b + 1];
    }
    const double sigma2 = st.sigma2;
    const int it = st.it;
    const double sigma1 = std::sqrt(sigma2);
    if (f2 > 0.0) {
        out[0] = std::sqrt(e2 / f2);                                    // ||xi - xi~|| / ||xi||
        out[1] = std::sqrt(std::max(0.0, 1.0 - sigma2 / f2));            // Eckart-Young floor
        out[2] = sigma2 > 0.0 ? f2 / sigma2 : 0.0;                       // stable rank
    }
    out[3] = sigma1;
    out[4] = std::sqrt(f2);
    out[5] = (double)std::min(it, max_iters);
    return RIKFAD_OK;
}

RIKFAD_API int rikfad_check_finite(rikfad_handle h, void *stream)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
    cudaStream_t s = (cudaStream_t)stream;
    RK_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
    rc = nonfinite_status(h, s);
    if (rc == RIKFAD_ERR_NONFINITE) {
        const std::string msg = g_last_error;
        const int rc2 = clear_guard(h, s);
        if (rc2)
            return rc2;
        g_last_error = msg;
    }
    return rc;
}

RIKFAD_API int rikfad_debug_check_failures(rikfad_handle h, int64_t *count, int *first_code)
{
    int rc = check_handle(h);
    if (rc)
        return rc;
#ifdef RIKFAD_CHECKED
    int32_t w[2] = {0, 0};
    RK_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
    RK_CUDA(cudaMemcpy(w, h->d_checks, sizeof w, cudaMemcpyDeviceToHost), "cudaMemcpy check counters");
    if (count)
        *count = w[0];
    if (first_code)
        *first_code = w[1];
#else
    if (count)
        *count = -1;
    if (first_code)
        *first_code = 0;
#endif
    return RIKFAD_OK;
}

RIKFAD_API void rikfad_debug_fail_allocation(int64_t n)
{
    g_fail_at.store(0);
    g_alloc_calls.store(0);
    g_fail_at.store(n > 0 ? n : 0);
}

RIKFAD_API int64_t rikfad_debug_live_allocations(void) { return g_live_allocs.load(); }


}  // extern "C"
