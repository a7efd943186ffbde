// rikfad_diag_kernels.cuh -- kernels of the friction diagnostic: how far the
// rank-1 friction xi~ = R C^T / (1^T R + eps) built from shadow factors is
// from the full element-wise friction xi of the same trajectory, against the
// best rank-1 approximation (Eckart-Young: relative error
// sqrt(1 - sigma_1^2 / ||xi||_F^2)), and the stable rank ||xi||_F^2 /
// sigma_1^2 (the comparison of the paper's Section 4.4).  sigma_1 comes from
// power iteration on xi^T xi: two matrix-vector passes over xi per iteration
// (HBM-bound GEMVs; there is no dense contraction to put on tensor cores).
// The iteration runs on the device: the transposed product writes one
// partial per row group and column, a column kernel adds them, a one-block
// kernel normalises the iterate, forms the Rayleigh quotient and tests
// convergence, and every kernel of the loop returns at once after
// convergence, so the host enqueues iterations in batches and reads one small
// state record per batch.  Every reduction runs in a fixed order.  Float64
// is slow on this GPU: per element the kernels compute in float32, and
// float64 only adds partial sums (per row, per column block, per block).
#pragma once
#include "rikfad_kernels.cuh"

namespace rikfad {

constexpr int kDiagFinThreads = 1024;    // threads of the one-block kernels
constexpr int kDiagBatch = 8;            // loads a thread issues before consuming them
constexpr int kDiagMaxRowGroups = 512;   // row groups of the transposed product (partials per column)

// Rows per block of the transposed product: at least 32, with at most
// kDiagMaxRowGroups row groups (partials per column for the column kernel).
inline __host__ __device__ int64_t diag_rows_per_group(int64_t m)
{
    const int64_t r = (m + kDiagMaxRowGroups - 1) / kDiagMaxRowGroups;
    return r < 32 ? 32 : r;
}

// State of one power iteration, in device memory (read back by the host).
struct DiagState {
    double sigma2;     // Rayleigh quotient ||xi v||^2 of the current unit iterate
    double w2;         // ||xi^T xi v||^2
    int32_t it;        // iterations done
    int32_t done;      // converged, or max_iters reached, or xi^T xi v = 0
    float inv;         // 1 / (1^T R + eps_stab) of the shadow factors (0 if zero)
    int32_t pad_;
};

__device__ __forceinline__ double warp_sum_f64(double v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Block-wide sum of one double per thread, threads in a fixed tree order;
// the result is returned to every thread.  Float64 arithmetic is slow on
// this GPU, so only warp 0 combines the warp sums and the total is passed on
// through shared memory (scratch holds NT / 32 + 1 doubles).
template <int NT>
__device__ __forceinline__ double block_sum_f64(double v, double *scratch)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum_f64(v);
    __syncthreads();
    if (lane == 0)
        scratch[warp] = v;
    __syncthreads();
    if (warp == 0) {
        double t = lane < NT / 32 ? scratch[lane] : 0.0;
        t = warp_sum_f64(t);
        if (lane == 0)
            scratch[NT / 32] = t;
    }
    __syncthreads();
    return scratch[NT / 32];
}

// Start of a diagnostic: inv from 1^T R (den, as the step kernels form it),
// the unit start vector v = C / ||C|| (1/sqrt(n) per entry if C = 0), and a
// cleared state.  One block.
__global__ void __launch_bounds__(kDiagFinThreads) rikfad_diag_setup_kernel(const float *den, float eps,
                                                                           const float *C, int64_t n,
                                                                           float *v, DiagState *st)
{
    __shared__ double scratch[kDiagFinThreads / 32 + 1];
    __shared__ double s_scale;
    double a = 0.0;
    for (int64_t j = threadIdx.x; j < n; j += kDiagFinThreads)
        a += (double)C[j] * (double)C[j];
    const double c2 = block_sum_f64<kDiagFinThreads>(a, scratch);
    // One float64 square root and division for the block (float64 is slow on
    // this GPU), then a multiply per entry.
    if (threadIdx.x == 0)
        s_scale = c2 > 0.0 ? 1.0 / sqrt(c2) : 0.0;
    __syncthreads();
    const double sc = s_scale;
    const float uniform = (float)(1.0 / sqrt((double)n));
    for (int64_t j = threadIdx.x; j < n; j += kDiagFinThreads)
        v[j] = sc > 0.0 ? (float)((double)C[j] * sc) : uniform;
    if (threadIdx.x == 0) {
        const float d = *den + eps;
        st->inv = d == 0.f ? 0.f : 1.f / d;
        st->sigma2 = 0.0;
        st->w2 = 0.0;
        st->it = 0;
        st->done = 0;
    }
}

// Per block of 8 rows (one per warp): sum of xi^2 and of (xi - xi~)^2,
// written to part[2 * block] and part[2 * block + 1].  A row is added in
// float32 (xi - xi~ is the difference of two floats, exact where they are
// within a factor two of each other): each lane its elements, then the 32
// lanes by a butterfly; the rows and the blocks are added in float64.
__global__ void __launch_bounds__(kThreads) rikfad_diag_norms_kernel(const float *xi, int64_t m, int64_t n,
                                                                     const float *R, const float *C,
                                                                     const DiagState *st, double *part)
{
    __shared__ double s1[kWarps], s2[kWarps];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t row = (int64_t)blockIdx.x * kWarps + warp;
    const float inv = st->inv;
    float f1 = 0.f, f2 = 0.f;
    if (row < m) {
        const float rhat = R[row] * inv;
        // kDiagBatch loads in flight per lane, then the sums in element order
        for (int64_t j0 = lane; j0 < n; j0 += 32 * kDiagBatch) {
            float xv[kDiagBatch], cv[kDiagBatch];
#pragma unroll
            for (int k = 0; k < kDiagBatch; ++k) {
                const int64_t j = j0 + 32 * k;
                xv[k] = j < n ? xi[row * n + j] : 0.f;
                cv[k] = j < n ? C[j] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < kDiagBatch; ++k) {
                const float d = xv[k] - rhat * cv[k];
                f1 = fmaf(xv[k], xv[k], f1);
                f2 = fmaf(d, d, f2);
            }
        }
    }
    const double a1 = (double)warp_sum(f1);
    const double a2 = (double)warp_sum(f2);
    if (lane == 0) {
        s1[warp] = a1;
        s2[warp] = a2;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double t1 = 0.0, t2 = 0.0;
        for (int k = 0; k < kWarps; ++k) {
            t1 += s1[k];
            t2 += s2[k];
        }
        part[2 * blockIdx.x] = t1;
        part[2 * blockIdx.x + 1] = t2;
    }
}

// u = xi v, one warp per row, and per block of 8 rows the sum of u_i^2 in
// float64 (upart[block]).  Returns at once once the iteration is done.
__global__ void __launch_bounds__(kThreads) rikfad_diag_matvec_kernel(const float *xi, int64_t m, int64_t n,
                                                                      const float *v, float *u, double *upart,
                                                                      const DiagState *st)
{
    __shared__ double su[kWarps];
    if (st->done)
        return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t row = (int64_t)blockIdx.x * kWarps + warp;
    float acc = 0.f;
    if (row < m) {
        for (int64_t j0 = lane; j0 < n; j0 += 32 * kDiagBatch) {
            float a[kDiagBatch], b[kDiagBatch];
#pragma unroll
            for (int k = 0; k < kDiagBatch; ++k) {
                const int64_t j = j0 + 32 * k;
                a[k] = j < n ? xi[row * n + j] : 0.f;
                b[k] = j < n ? v[j] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < kDiagBatch; ++k)
                acc = fmaf(a[k], b[k], acc);
        }
        acc = warp_sum(acc);
        if (lane == 0)
            u[row] = acc;
    }
    if (lane == 0)
        su[warp] = row < m ? (double)acc * (double)acc : 0.0;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int k = 0; k < kWarps; ++k)
            t += su[k];
        upart[blockIdx.x] = t;
    }
}

// wpart[g][j] = sum over the rows of row group g (blockIdx.x) of xi_ij u_i,
// for the kThreads columns of tile blockIdx.y (one thread per column, rows
// in order).  Returns at once once the iteration is done.
__global__ void __launch_bounds__(kThreads) rikfad_diag_matvec_t_kernel(const float *xi, int64_t m, int64_t n,
                                                                        const float *u, float *wpart,
                                                                        const DiagState *st)
{
    if (st->done)
        return;
    const int64_t rpg = diag_rows_per_group(m);
    const int64_t r0 = (int64_t)blockIdx.x * rpg;
    const int64_t r1 = r0 + rpg < m ? r0 + rpg : m;
    const int64_t j = (int64_t)blockIdx.y * kThreads + threadIdx.x;
    if (j >= n)
        return;
    float acc = 0.f;
    for (int64_t i0 = r0; i0 < r1; i0 += kDiagBatch) {
        float a[kDiagBatch], b[kDiagBatch];
#pragma unroll
        for (int k = 0; k < kDiagBatch; ++k) {
            const int64_t i = i0 + k;
            a[k] = i < r1 ? xi[i * n + j] : 0.f;
            b[k] = i < r1 ? u[i] : 0.f;
        }
#pragma unroll
        for (int k = 0; k < kDiagBatch; ++k)
            acc = fmaf(a[k], b[k], acc);
    }
    wpart[(int64_t)blockIdx.x * n + j] = acc;
}

// w_j = sum over the row groups of wpart[g][j] for the 32 columns of block
// blockIdx.x (kDiagFinThreads threads): warp k adds groups k, k + 32,
// k + 64, ... in order, then warp 0 adds the 32 warp sums in warp order.  w
// goes to w, and the block's sum of w_j^2 (float64) to wsq[blockIdx.x].
// Returns at once once the iteration is done.
__global__ void __launch_bounds__(kDiagFinThreads) rikfad_diag_colsum_kernel(const float *wpart, int nb,
                                                                             int64_t n, float *w, double *wsq,
                                                                             const DiagState *st)
{
    constexpr int kColWarps = kDiagFinThreads / 32;
    __shared__ float part[kColWarps][32];
    if (st->done)
        return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t j = (int64_t)blockIdx.x * 32 + lane;
    float acc = 0.f;
    if (j < n) {
        for (int g0 = warp; g0 < nb; g0 += kColWarps * kDiagBatch) {
            float t[kDiagBatch];
#pragma unroll
            for (int k = 0; k < kDiagBatch; ++k) {
                const int g = g0 + k * kColWarps;
                t[k] = g < nb ? wpart[(int64_t)g * n + j] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < kDiagBatch; ++k)
                acc += t[k];
        }
    }
    part[warp][lane] = acc;
    __syncthreads();
    if (warp == 0) {
        float sum = 0.f;
#pragma unroll 8
        for (int k = 0; k < kColWarps; ++k)
            sum += part[k][lane];
        if (j < n)
            w[j] = sum;
        const double q = warp_sum_f64(j < n ? (double)sum * (double)sum : 0.0);
        if (lane == 0)
            wsq[blockIdx.x] = q;
    }
}

// End of one power iteration, one block: ||w||^2 from the column blocks'
// partials, sigma^2 = ||u||^2 (the Rayleigh quotient of xi^T xi at the unit
// v) from the row blocks' partials, the next iterate v = w / ||w||, and the
// convergence test |sigma^2 - previous| <= tol sigma^2 (from the second
// iteration on); done after max_iters iterations or when w = 0.
__global__ void __launch_bounds__(kDiagFinThreads) rikfad_diag_iterate_kernel(
    const float *w, int64_t n, const double *wsq, int nbw, const double *upart, int nbu, float *v,
    DiagState *st, double tol, int max_iters)
{
    __shared__ double scratch[kDiagFinThreads / 32 + 1];
    __shared__ double s_scale;
    if (st->done)
        return;
    double a = 0.0;
    for (int b = threadIdx.x; b < nbw; b += kDiagFinThreads)
        a += wsq[b];
    const double w2 = block_sum_f64<kDiagFinThreads>(a, scratch);
    double c = 0.0;
    for (int b = threadIdx.x; b < nbu; b += kDiagFinThreads)
        c += upart[b];
    const double u2 = block_sum_f64<kDiagFinThreads>(c, scratch);
    if (threadIdx.x == 0)
        s_scale = w2 > 0.0 ? 1.0 / sqrt(w2) : 0.0;
    __syncthreads();
    if (w2 > 0.0) {
        // The product in float64, rounded once (scaled in float32 the quotient
        // seldom settled to a 1e-10 convergence test).
        const double sc = s_scale;
        for (int64_t j = threadIdx.x; j < n; j += kDiagFinThreads)
            v[j] = (float)((double)w[j] * sc);
    }
    if (threadIdx.x == 0) {
        const double prev = st->sigma2;
        const int it = st->it + 1;
        st->it = it;
        st->sigma2 = u2;
        st->w2 = w2;
        if (w2 == 0.0 || it >= max_iters || (it > 1 && fabs(u2 - prev) <= tol * u2))
            st->done = 1;
    }
}

}  // namespace rikfad
