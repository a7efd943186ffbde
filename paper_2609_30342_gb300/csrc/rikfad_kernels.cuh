// rikfad_kernels.cuh -- sm_103a kernels of the R-iKFAD optimiser step.
//
// The method (BACD splitting, Appendix A of the paper):
//   B  P^(B) = P_n - h G
//   A  X_{n+1} = X_n + h P^(B)
//   C  P^(1) = P^(B) exp(-(h/2) xi~_n),  xi~ = R C^T / (1^T R + eps)   (Eq. xi_def)
//      R_{n+1} = e^{-alpha h} R_n + k [P^(1)]^2 1_n,  k = (1 - e^{-alpha h})/(mu alpha)
//      C_{n+1} = e^{-alpha h} C_n + k ([P^(1)]^2)^T 1_m
//      P^(2) = P^(1) exp(-(h/2) xi~_{n+1})
//   D  P_{n+1} = P^(2) e^{-gamma h}
//
// Scheduling.  R_{n+1}, C_{n+1} are reductions over the whole matrix, so
// P^(2) cannot be formed in the same pass that produces P^(1).  The step
// kernel therefore stores P^(1) and the NEXT step applies the pending factor
// exp(-(h_prev/2) xi~_{n+1}) e^{-gamma h_prev} on the fly, with the factors
// that the finalise kernel of this step wrote.  Every element is read once
// and written once per step (grad, X, P read; X, P written).  When the step
// size does not change, the pending factor and this step's first half-damp
// are the same exponential and one exp2 serves both.
//
// Reductions are deterministic: a warp owns a row segment (row sums by a
// fixed shuffle tree), each lane owns fixed columns (column sums accumulate
// row by row in lane-private shared memory, then across warps in warp order,
// then across the blocks of a panel in slot order in the finalise kernel).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "rikfad_checks.cuh"
#include "rikfad_plan.hpp"

namespace rikfad {

// Non-finite guard.  A kernel that produces a non-finite factor, friction or
// denominator records the tensor: the lowest such index in device memory
// (atomicMin; INT32_MAX when there is none) and a flag in page-locked host
// memory that the host reads without waiting for the device.
struct Guard {
    int32_t *first;
    volatile int32_t *host;
};

__device__ __forceinline__ void report_nonfinite(const Guard &g, int tensor)
{
    atomicMin(g.first, tensor);
    *g.host = 1;
}

struct StepParams {
    const TensorDev *tensors;
    const PanelDev *panels;
    const PieceDev *pieces;
    const int32_t *block_piece;
    float *const *xptr;        // ntensors device pointers
    const void *const *gptr;
    float *const *pptr;
    float *fac;                // R, C of matrices; friction of vectors
    float *rowpart;
    float *colpart;
    const float *spart;        // partial sums of R (denominators)
    float h;                   // step size
    float ex_cur;              // -(h/2) log2(e): exp(-(h/2) xi) = exp2(ex_cur xi)
    float ex_prev;             // -(h_prev/2) log2(e)
    float damp_prev;           // e^{-gamma h_prev}
    float damp_cur;            // e^{-gamma h} (vectors finish D inside the step)
    float decay;               // e^{-alpha h}
    float gain;                // (1 - e^{-alpha h})/(mu alpha)
    float eps;                 // eps_stab
    Guard guard;
    CheckBounds chk;           // read by checked builds only
};

// ---------------------------------------------------------------- helpers

// Programmatic dependent launch: the kernels of a step are launched so that
// they may start before their predecessor in the stream has finished; they
// run this wait before touching any data the predecessor may write, and let
// their own successor start launching early.
__device__ __forceinline__ void wait_for_predecessor()
{
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

__device__ __forceinline__ void allow_successor_launch()
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ float warp_sum(float v)
{
    // Butterfly: float addition is commutative, so every lane ends with the
    // bitwise-same total.
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// 1^T R of a matrix from the finalise kernel's partial sums, in a fixed order
// (identical in every warp that computes it).
__device__ __forceinline__ float row_total(const float *spart, const TensorDev &td)
{
    const int lane = threadIdx.x & 31;
    float v = 0.f;
    for (int c = lane; c < td.spart_cnt; c += 32)
        v += spart[td.spart_off + c];
    return warp_sum(v);
}

// 1 / (1^T R + eps), with the friction set to zero when the denominator is
// zero (eps = 0 and R = 0; Theorem 3's convention).
__device__ __forceinline__ float inv_denominator(float s, float eps)
{
    const float den = s + eps;
    return den == 0.f ? 0.f : 1.f / den;
}

template <typename GT> struct Grad8;

template <> struct Grad8<float> {
    float v[8];
    __device__ __forceinline__ void load(const float *g)
    {
        const float4 a = __ldcs(reinterpret_cast<const float4 *>(g));
        const float4 b = __ldcs(reinterpret_cast<const float4 *>(g) + 1);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
    __device__ __forceinline__ float get(int e) const { return v[e]; }
};

template <> struct Grad8<__nv_bfloat16> {
    uint32_t w[4];
    __device__ __forceinline__ void load(const __nv_bfloat16 *g)
    {
        const uint4 a = __ldcs(reinterpret_cast<const uint4 *>(g));
        w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w;
    }
    // bf16 -> f32 is exact: the bf16 bits are the high half of the f32.
    __device__ __forceinline__ float get(int e) const
    {
        const uint32_t word = w[e >> 1];
        return __uint_as_float((e & 1) ? (word & 0xffff0000u) : (word << 16));
    }
};

__device__ __forceinline__ float grad_at(const float *g, int64_t i) { return __ldcs(g + i); }
__device__ __forceinline__ float grad_at(const __nv_bfloat16 *g, int64_t i)
{
    return __bfloat162float(g[i]);
}

__device__ __forceinline__ void load8(const float *p, float (&v)[8])
{
    const float4 a = __ldcs(reinterpret_cast<const float4 *>(p));
    const float4 b = __ldcs(reinterpret_cast<const float4 *>(p) + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

__device__ __forceinline__ void store8(float *p, const float (&v)[8])
{
    __stcs(reinterpret_cast<float4 *>(p), make_float4(v[0], v[1], v[2], v[3]));
    __stcs(reinterpret_cast<float4 *>(p) + 1, make_float4(v[4], v[5], v[6], v[7]));
}

// ------------------------------------------- one element, matrix rule
//
// p_hat is the stored P^(1) of the previous step.  Returns P^(1) of this step
// and updates x.  e_cur = exp(-(h/2) xi~_ij), e_prev = exp(-(h_prev/2) xi~_ij),
// both with the current factors (= R_{n}, C_{n} of this step).
__device__ __forceinline__ float matrix_element(float &x, float p_hat, float g, float e_cur,
                                                float e_prev, const StepParams &a)
{
    const float p_n = (p_hat * e_prev) * a.damp_prev;   // pending C half-damp, then D
    const float p_b = fmaf(-a.h, g, p_n);                 // B
    x = fmaf(a.h, p_b, x);                                // A
    return p_b * e_cur;                                   // C, first half-damp
}

// ------------------------------------------------- matrix piece, 8-wide

// 256-column chunks whose loads are issued together (registers: ~20 per chunk).
#ifndef RIKFAD_CHUNK_GROUP
#define RIKFAD_CHUNK_GROUP 1
#endif

// ACCUM: add each row's squares into the warp's column buffer (several rows
// per warp); otherwise store them (one row per warp, buffer not cleared).
// RPW rows per warp (1, 2 or 4; panels of at most kPanelMax / RPW columns):
// each of the warp's RPW lane groups takes its own row, 256 / RPW columns per
// chunk, so a panel whose width is not a multiple of 256 still loads 256
// columns per warp and round trip; group h accumulates its columns at
// red[warp][h * kPanelMax / RPW + c].
template <typename GT, bool REUSE, bool ACCUM = true, int RPW = 1>
__device__ __forceinline__ void matrix_piece_vec(const StepParams &a, const PieceDev &pc,
                                                 const TensorDev &td, const PanelDev &pd,
                                                 const float *Cs, float *red, float inv)
{
    constexpr int kRowLanes = 32 / RPW;                 // lanes per row
    constexpr int kRowChunk = kRowLanes * 8;            // columns per chunk of one row
    constexpr int kRowsPerWarp = RPW;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rl = lane & (kRowLanes - 1), half = lane / kRowLanes;   // lane group = row
    const int64_t n = td.cols;
    const int w = pd.width;
    const int nch = RPW > 1 ? (w + kRowChunk - 1) / kRowChunk : pd.nch;
    float *X = a.xptr[pc.tensor];
    const GT *G = static_cast<const GT *>(a.gptr[pc.tensor]);
    float *P = a.pptr[pc.tensor];
    const float *R = a.fac + td.fac_off;
    float *rowpart = a.rowpart + td.rowpart_off + (int64_t)(pc.panel - td.panel0) * td.rows;
    float *myred = red + warp * kPanelMax + half * (kPanelMax / RPW);

    for (int64_t r0 = pc.begin + kRowsPerWarp * warp; r0 < pc.end; r0 += kRowsPerWarp * kWarps) {
        const int64_t row = r0 + half;
        const bool live = RPW == 1 || row < pc.end;     // ragged piece: trailing lane groups idle
        const float rhat = live ? R[row] * inv : 0.f;
        const float a_cur = a.ex_cur * rhat;
        const float a_prev = REUSE ? a_cur : a.ex_prev * rhat;
        const int64_t base = row * n + pd.col0;

        // RIKFAD_CHUNK_GROUP chunks at a time: every load of the group is
        // issued before any arithmetic on it.
        float racc = 0.f;
#pragma unroll 1
        for (int g0 = 0; g0 < nch; g0 += RIKFAD_CHUNK_GROUP) {
            float xv[RIKFAD_CHUNK_GROUP][8], pv[RIKFAD_CHUNK_GROUP][8];
            Grad8<GT> gv[RIKFAD_CHUNK_GROUP];
#pragma unroll
            for (int k = 0; k < RIKFAD_CHUNK_GROUP; ++k) {
                const int c = (g0 + k) * kRowChunk + rl * 8;
                if (live && c < w) {
                    gv[k].load(G + base + c);
                    load8(X + base + c, xv[k]);
                    load8(P + base + c, pv[k]);
                }
            }
#pragma unroll
            for (int k = 0; k < RIKFAD_CHUNK_GROUP; ++k) {
                const int c = (g0 + k) * kRowChunk + rl * 8;
                if (live && c < w) {
                    const float4 c0 = *reinterpret_cast<const float4 *>(Cs + c);
                    const float4 c1 = *reinterpret_cast<const float4 *>(Cs + c + 4);
                    const float cv[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
                    float q[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float e_cur = exp2f(a_cur * cv[e]);
                        const float e_prev = REUSE ? e_cur : exp2f(a_prev * cv[e]);
                        const float p1 = matrix_element(xv[k][e], pv[k][e], gv[k].get(e), e_cur,
                                                        e_prev, a);
                        pv[k][e] = p1;
                        q[e] = p1 * p1;
                        racc += q[e];
                    }
                    store8(X + base + c, xv[k]);
                    store8(P + base + c, pv[k]);
                    float4 *r4 = reinterpret_cast<float4 *>(myred + c);
                    if (ACCUM) {
                        float4 r0 = r4[0], r1 = r4[1];
                        r0.x += q[0]; r0.y += q[1]; r0.z += q[2]; r0.w += q[3];
                        r1.x += q[4]; r1.y += q[5]; r1.z += q[6]; r1.w += q[7];
                        r4[0] = r0;
                        r4[1] = r1;
                    } else {
                        r4[0] = make_float4(q[0], q[1], q[2], q[3]);
                        r4[1] = make_float4(q[4], q[5], q[6], q[7]);
                    }
                }
            }
        }
        if (RPW > 1) {
#pragma unroll
            for (int o = kRowLanes / 2; o > 0; o >>= 1)
                racc += __shfl_xor_sync(0xffffffffu, racc, o);
        } else {
            racc = warp_sum(racc);
        }
        if (live && rl == 0)
            rowpart[row] = racc;
    }
}

// ----------------------------------------------- matrix piece, scalar
// For matrices whose rows are not 8-aligned (cols % 8 != 0).

template <typename GT, bool REUSE, bool ACCUM = true>
__device__ __forceinline__ void matrix_piece_scalar(const StepParams &a, const PieceDev &pc,
                                                    const TensorDev &td, const PanelDev &pd,
                                                    const float *Cs, float *red, float inv)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t n = td.cols;
    const int w = pd.width;
    float *X = a.xptr[pc.tensor];
    const GT *G = static_cast<const GT *>(a.gptr[pc.tensor]);
    float *P = a.pptr[pc.tensor];
    const float *R = a.fac + td.fac_off;
    float *rowpart = a.rowpart + td.rowpart_off + (int64_t)(pc.panel - td.panel0) * td.rows;
    float *myred = red + warp * kPanelMax;

    for (int64_t row = pc.begin + warp; row < pc.end; row += kWarps) {
        const float rhat = R[row] * inv;
        const float a_cur = a.ex_cur * rhat;
        const float a_prev = REUSE ? a_cur : a.ex_prev * rhat;
        const int64_t base = row * n + pd.col0;
        float racc = 0.f;
        for (int c = lane; c < w; c += 32) {
            const float e_cur = exp2f(a_cur * Cs[c]);
            const float e_prev = REUSE ? e_cur : exp2f(a_prev * Cs[c]);
            float x = X[base + c];
            const float p1 = matrix_element(x, P[base + c], grad_at(G, base + c), e_cur, e_prev, a);
            X[base + c] = x;
            P[base + c] = p1;
            const float q = p1 * p1;
            racc += q;
            if (ACCUM)
                myred[c] += q;
            else
                myred[c] = q;
        }
        racc = warp_sum(racc);
        if (lane == 0)
            rowpart[row] = racc;
    }
}

// ------------------------------------------ element-wise rule (vectors)
//
// Element-wise iKFAD (Section 2, "Memory Complexity"): the friction xi of the
// element is local, so the whole step -- including the second half-damp and
// D -- completes here and P holds P_{n+1}.
__device__ __forceinline__ void vector_element(float &x, float &p, float &xi, float g,
                                               const StepParams &a)
{
    const float p_b = fmaf(-a.h, g, p);                       // B
    x = fmaf(a.h, p_b, x);                                    // A
    const float p1 = p_b * exp2f(a.ex_cur * xi);              // C, first half-damp
    xi = fmaf(a.gain, p1 * p1, a.decay * xi);                 // C, friction filter
    p = (p1 * exp2f(a.ex_cur * xi)) * a.damp_cur;             // C, second half-damp; D
}

template <typename GT>
__device__ __forceinline__ void vector_piece(const StepParams &a, const PieceDev &pc,
                                             const TensorDev &td)
{
    float *X = a.xptr[pc.tensor];
    const GT *G = static_cast<const GT *>(a.gptr[pc.tensor]);
    float *P = a.pptr[pc.tensor];
    float *XI = a.fac + td.fac_off;
    const int64_t b0 = pc.begin;                // multiple of 8 (planner)
    const int64_t nvec = (pc.end - b0) / 8;
    bool bad = false;
    for (int64_t v = threadIdx.x; v < nvec; v += kThreads) {
        const int64_t e0 = b0 + v * 8;
        Grad8<GT> g;
        g.load(G + e0);
        float x[8], p[8], xi[8];
        load8(X + e0, x);
        load8(P + e0, p);
        load8(XI + e0, xi);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            vector_element(x[e], p[e], xi[e], g.get(e), a);
            bad |= !isfinite(xi[e]);
        }
        store8(X + e0, x);
        store8(P + e0, p);
        store8(XI + e0, xi);
    }
    for (int64_t e = b0 + nvec * 8 + threadIdx.x; e < pc.end; e += kThreads) {
        float x = X[e], p = P[e], xi = XI[e];
        vector_element(x, p, xi, grad_at(G, e), a);
        bad |= !isfinite(xi);
        X[e] = x;
        P[e] = p;
        XI[e] = xi;
    }
    // The friction is d xi + k [P^(1)]^2: non-finite exactly when the
    // half-damped momentum (or the friction before) is.
    if (bad)
        report_nonfinite(a.guard, pc.tensor);
}

// ------------------------------ matrix with element-wise friction (full iKFAD)
//
// Full iKFAD on a matrix (Eqs. ikfad_1 to ikfad_3, the same expression as
// vector_element) with the squares of the half-damped momentum P^(1) also
// summed per row and per column, so the matrix's R, C follow R-iKFAD's factor
// filter as shadow factors of the same trajectory (the comparison of the
// paper's Section 4.4).  P holds P_{n+1}.
__device__ __forceinline__ float full_element(float &x, float &p, float &xi, float g,
                                              const StepParams &a)
{
    const float p_b = fmaf(-a.h, g, p);                       // B
    x = fmaf(a.h, p_b, x);                                    // A
    const float p1 = p_b * exp2f(a.ex_cur * xi);              // C, first half-damp
    xi = fmaf(a.gain, p1 * p1, a.decay * xi);                 // C, friction filter
    p = (p1 * exp2f(a.ex_cur * xi)) * a.damp_cur;             // C, second half-damp; D
    return p1 * p1;
}

template <typename GT>
__device__ __forceinline__ void matrix_piece_full(const StepParams &a, const PieceDev &pc,
                                                  const TensorDev &td, const PanelDev &pd,
                                                  float *red)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t n = td.cols;
    const int w = pd.width;
    float *X = a.xptr[pc.tensor];
    const GT *G = static_cast<const GT *>(a.gptr[pc.tensor]);
    float *P = a.pptr[pc.tensor];
    float *XI = a.fac + td.xi_off;
    float *rowpart = a.rowpart + td.rowpart_off + (int64_t)(pc.panel - td.panel0) * td.rows;
    float *myred = red + warp * kPanelMax;
    for (int64_t row = pc.begin + warp; row < pc.end; row += kWarps) {
        const int64_t base = row * n + pd.col0;
        float racc = 0.f;
        if (td.vec) {
#pragma unroll 1
            for (int ch = 0; ch < pd.nch; ++ch) {
                const int c = ch * kChunk + lane * 8;
                if (c < w) {
                    Grad8<GT> gv;
                    gv.load(G + base + c);
                    float x[8], p[8], xi[8];
                    load8(X + base + c, x);
                    load8(P + base + c, p);
                    load8(XI + base + c, xi);
                    float q[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        q[e] = full_element(x[e], p[e], xi[e], gv.get(e), a);
                        racc += q[e];
                    }
                    store8(X + base + c, x);
                    store8(P + base + c, p);
                    store8(XI + base + c, xi);
                    float4 *r4 = reinterpret_cast<float4 *>(myred + c);
                    float4 r0 = r4[0], r1 = r4[1];
                    r0.x += q[0]; r0.y += q[1]; r0.z += q[2]; r0.w += q[3];
                    r1.x += q[4]; r1.y += q[5]; r1.z += q[6]; r1.w += q[7];
                    r4[0] = r0;
                    r4[1] = r1;
                }
            }
        } else {
            for (int c = lane; c < w; c += 32) {
                float x = X[base + c], p = P[base + c], xi = XI[base + c];
                const float q = full_element(x, p, xi, grad_at(G, base + c), a);
                X[base + c] = x;
                P[base + c] = p;
                XI[base + c] = xi;
                racc += q;
                myred[c] += q;
            }
        }
        racc = warp_sum(racc);
        if (lane == 0)
            rowpart[row] = racc;
    }
}

// ------------------------------------------------------ the step kernel

// Blocks per SM the register budget is sized for (2: 128 registers/thread).
#ifndef RIKFAD_STEP_MIN_BLOCKS
#define RIKFAD_STEP_MIN_BLOCKS 2
#endif

// SHADOW: the instantiation for handles whose matrices keep element-wise
// friction with shadow factors (the R-iKFAD instantiation carries no code for
// it).
// out[c] = the piece's column sums: warp wi's lane group h holds its share at
// red[wi * kPanelMax + h * kPanelMax / RPW + c]; added warp by warp, groups in
// order.
template <int RPW>
__device__ __forceinline__ void column_partials(const float *red, float *out, int w)
{
    for (int c = threadIdx.x; c < w; c += kThreads) {
        float s = 0.f;
#pragma unroll
        for (int wi = 0; wi < kWarps; ++wi)
#pragma unroll
            for (int h = 0; h < RPW; ++h)
                s += red[wi * kPanelMax + h * (kPanelMax / RPW) + c];
        out[c] = s;
    }
}

// Rows per warp for an 8-wide panel (matrix_piece_vec RPW): a panel that is
// not a whole number of 256-column chunks takes 4 rows per warp up to 64
// columns and 2 up to kPanelMax / 2 columns; every other panel takes 1.
__device__ __forceinline__ int rows_per_warp(int w)
{
    if (w % kChunk == 0 || w > kPanelMax / 2)
        return 1;
    return w <= kChunk / 4 ? 4 : 2;
}

template <typename GT, bool REUSE, bool SHADOW = false>
__global__ void __launch_bounds__(kThreads, RIKFAD_STEP_MIN_BLOCKS) rikfad_step_kernel(StepParams a)
{
    __shared__ __align__(16) float Cs[kPanelMax];
    __shared__ __align__(16) float red[kWarps * kPanelMax];
    const int b = blockIdx.x;
    if (!RK_DEV_CHECK(a.chk, b < a.chk.nblocks, kChkBlock))
        return;
    const int q0 = a.block_piece[b], q1 = a.block_piece[b + 1];
    wait_for_predecessor();
    allow_successor_launch();
    if (!block_ok(a.chk, b, q0, q1))
        return;
    for (int q = q0; q < q1; ++q) {
        const PieceDev pc = a.pieces[q];
        if (!piece_tensor_ok(a.chk, pc))
            continue;
        const TensorDev td = a.tensors[pc.tensor];
        if (pc.kind == kElements) {
            if (vector_piece_ok(a.chk, pc, td, a.xptr[pc.tensor], a.gptr[pc.tensor], a.pptr[pc.tensor],
                                true))
                vector_piece<GT>(a, pc, td);
            continue;
        }
        if (!piece_panel_ok(a.chk, pc, td))
            continue;
        const PanelDev pd = a.panels[pc.panel];
        // Block-uniform: every thread evaluates the same checks on the same
        // entries, so a skipped piece is skipped by the whole block.
        if (!matrix_piece_ok(a.chk, pc, td, pd, a.xptr[pc.tensor], a.gptr[pc.tensor], a.pptr[pc.tensor],
                             true))
            continue;
        const int w = pd.width;
        // Stage this panel's C, clear the column accumulators.
        const float *C = a.fac + td.fac_off + td.rows + pd.col0;
        for (int c = threadIdx.x; c < w; c += kThreads)
            Cs[c] = C[c];
        for (int i = threadIdx.x; i < kWarps * kPanelMax; i += kThreads)
            red[i] = 0.f;
        const float inv = inv_denominator(row_total(a.spart, td), a.eps);
        __syncthreads();
        if (SHADOW && td.full) {
            matrix_piece_full<GT>(a, pc, td, pd, red);
        } else if (td.vec && rows_per_warp(w) == 4) {
            matrix_piece_vec<GT, REUSE, true, 4>(a, pc, td, pd, Cs, red, inv);
        } else if (td.vec && rows_per_warp(w) == 2) {
            matrix_piece_vec<GT, REUSE, true, 2>(a, pc, td, pd, Cs, red, inv);
        } else if (td.vec) {
            matrix_piece_vec<GT, REUSE>(a, pc, td, pd, Cs, red, inv);
        } else {
            matrix_piece_scalar<GT, REUSE>(a, pc, td, pd, Cs, red, inv);
        }
        __syncthreads();
        // Column partial sums of this piece, warps (and their lane groups) added in order.
        float *out = a.colpart + pc.colpart_off;
        const int rpw = td.vec && !(SHADOW && td.full) ? rows_per_warp(w) : 1;
        if (rpw == 1)
            column_partials<1>(red, out, w);
        else if (rpw == 2)
            column_partials<2>(red, out, w);
        else
            column_partials<4>(red, out, w);
        __syncthreads();
    }
}

}  // namespace rikfad
