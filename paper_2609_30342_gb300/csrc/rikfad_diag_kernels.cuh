// rikfad_diag_kernels.cuh -- kernels of the friction diagnostic: how far the
// rank-1 friction xi~ = R C^T / (1^T R + eps) built from shadow factors is
// from the full element-wise friction xi of the same trajectory, against the
// best rank-1 approximation (Eckart-Young: relative error
// sqrt(1 - sigma_1^2 / ||xi||_F^2)), and the stable rank ||xi||_F^2 /
// sigma_1^2 (the comparison of the paper's Section 4.4).  sigma_1 comes from
// power iteration on xi^T xi: two matrix-vector passes over xi per iteration
// (HBM-bound GEMVs; there is no dense contraction to put on tensor cores).
// Every reduction runs in a fixed order.
#pragma once
#include "rikfad_kernels.cuh"

namespace rikfad {

constexpr int kDiagRowsPerBlock = 256;   // rows per block of the transposed product

__device__ __forceinline__ double warp_sum_f64(double v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Per block of 8 rows (one per warp): sum of xi^2 and of (xi - xi~)^2 in
// float64, written to part[2 * block] and part[2 * block + 1].
__global__ void __launch_bounds__(kThreads) rikfad_diag_norms_kernel(const float *xi, int64_t m, int64_t n,
                                                                     const float *R, const float *C,
                                                                     float inv, double *part)
{
    __shared__ double s1[kWarps], s2[kWarps];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t row = (int64_t)blockIdx.x * kWarps + warp;
    double a1 = 0.0, a2 = 0.0;
    if (row < m) {
        const float rhat = R[row] * inv;
        for (int64_t j = lane; j < n; j += 32) {
            const float v = xi[row * n + j];
            const double d = (double)v - (double)(rhat * C[j]);
            a1 += (double)v * (double)v;
            a2 += d * d;
        }
    }
    a1 = warp_sum_f64(a1);
    a2 = warp_sum_f64(a2);
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

// u = xi v, one warp per row.
__global__ void __launch_bounds__(kThreads) rikfad_diag_matvec_kernel(const float *xi, int64_t m, int64_t n,
                                                                      const float *v, float *u)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t row = (int64_t)blockIdx.x * kWarps + warp;
    if (row >= m)
        return;
    float acc = 0.f;
    for (int64_t j = lane; j < n; j += 32)
        acc = fmaf(xi[row * n + j], v[j], acc);
    acc = warp_sum(acc);
    if (lane == 0)
        u[row] = acc;
}

// wpart[b][j] = sum over the rows of block b of xi_ij u_i (one thread per
// column, rows in order).
__global__ void __launch_bounds__(kThreads) rikfad_diag_matvec_t_kernel(const float *xi, int64_t m, int64_t n,
                                                                        const float *u, float *wpart)
{
    const int64_t r0 = (int64_t)blockIdx.x * kDiagRowsPerBlock;
    const int64_t r1 = r0 + kDiagRowsPerBlock < m ? r0 + kDiagRowsPerBlock : m;
    for (int64_t j = threadIdx.x; j < n; j += kThreads) {
        float acc = 0.f;
        for (int64_t i = r0; i < r1; ++i)
            acc = fmaf(xi[i * n + j], u[i], acc);
        wpart[(int64_t)blockIdx.x * n + j] = acc;
    }
}

// w[j] = sum over blocks of wpart[b][j], blocks in order.
__global__ void __launch_bounds__(kThreads) rikfad_diag_colsum_kernel(const float *wpart, int nb, int64_t n,
                                                                      float *w)
{
    const int64_t j = (int64_t)blockIdx.x * kThreads + threadIdx.x;
    if (j >= n)
        return;
    float acc = 0.f;
    for (int b = 0; b < nb; ++b)
        acc += wpart[(int64_t)b * n + j];
    w[j] = acc;
}

}  // namespace rikfad
