// rikfad_quadratic.cu -- batched BACD integration of R-iKFAD on many small
// dense quadratics f(X) = 1/2 vec(X)^T A vec(X) (the test problem of the
// paper's numerical validation of the gamma = 0 rates, Section 3.2 and Table
// tab:g0_slopes: A = B B^T / d + 0.8 I, d = m n, integrated to t = 1e7).
//
// Every system is tiny (m n <= 32) and its steps are strictly sequential, so
// the kernel maps one system to one aligned group of L lanes and packs
// 32 / L systems into a warp (L = MB NB clamped to [4, 32], where MB and NB
// are m and n rounded up to powers of two; both are template parameters).
// Lane a of a group owns element a = i n + j (row-major vec(X), as the
// oracle): its X_a, its momentum and row a of A in registers, plus its own
// copies of R_i, C_j and 1^T R.  The gradient A vec(X) reads X from shared
// memory with 128-bit broadcast loads and accumulates with paired float32
// FMAs (two round-to-nearest FMAs per instruction).  [P^(1)]^2 is written
// twice: row-major with row stride RS and column-major with column stride CS
// (NB and MB, plus 4 when that is a multiple of 8, so that consecutive rows
// or columns start in different 16-byte bank groups; padding stays zero).
// A row sum and a column sum are then a few 128-bit loads each, added in a
// fixed order with paired adds, so the lanes of one row (column) hold
// bit-identical R_i (C_j).  The total comes from an xor butterfly of
// shuffles, which also leaves identical bits in every lane.  One warp barrier
// per step (everything is exchanged together, double buffered); no global
// memory inside the step loop but the recorded energies.

// One step k follows the BACD sub-steps of the splitting table (Appendix A):
//   B  P^(B)_k = P_k - h A vec(X_k)
//   A  X_{k+1} = X_k + h P^(B)_k
//   C  P^(1)   = P^(B)_k exp(-h/2 xi~_k);  R, C <- e^{-alpha h}(R, C) + k (row, column sums of [P^(1)]^2)
//      P^(2)   = P^(1) exp(-h/2 xi~_{k+1})
//   D  P_{k+1} = P^(2) e^{-gamma h}
// 1^T R is filtered alongside, from the total of [P^(1)]^2 (equal to the sum
// of the filtered R_i up to rounding).
//
// Precision.  With gamma = 0 the friction decays like 1/t, and by t ~ 1e5
// one step's damping h/2 xi~ is ~1e-7: below half a float32 ulp of P, so a
// stored P (1 - 1e-7) rounds back to P and the damping is lost (the decay
// slopes bend from -1 to -0.7).  The kernel therefore never stores a damped
// momentum between steps: it carries P^(B)_{k-1} and the pending
// e1 = expm1(-h/2 xi~_{k-1}), and forms the next kick as
//   P^(B)_k = P^(B)_{k-1} + [P^(B)_{k-1} em - h g],
//   em = expm1(-h/2 xi~_{k-1} - h/2 xi~_k - gamma h)
//      = (1 + e1)(1 + e2)(1 + expm1(-gamma h)) - 1,  e2 = expm1(-h/2 xi~_k),
// in which the damping is part of a bracket about 50 times smaller than P,
// represented to its own float32 precision; the one rounding of the sum is
// unbiased.  e2 also gives this step's first half-damp, so one expm1 per
// step serves both.  P_k itself (for the energy and the output) is
// P^(B)_{k-1} + P^(B)_{k-1} em.  A launch starts from the stored P_k with
// nothing pending, so runs split at a launch boundary are bit-identical.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <string>

#include "rikfad.h"

namespace rikfad {
int report_error(int code, const std::string &msg);
}

namespace {

constexpr int kQThreads = 128;                // 4 warps per block
constexpr int kQWarps = kQThreads / 32;
// Blocks per SM the registers are sized for (5: up to 102 registers).  A cap of
// 64 registers (8 blocks) measured slower in latency and in throughput.
#ifndef RIKFAD_QUAD_MIN_BLOCKS
#define RIKFAD_QUAD_MIN_BLOCKS 5
#endif
constexpr int kQMinBlocks = RIKFAD_QUAD_MIN_BLOCKS;
constexpr int64_t kQMaxDim = 32;
constexpr int kQBufFloats = 128;             // per warp and parity, for each padded copy

struct QuadParams {
    int64_t batch;
    int m, n, d;
    const float *A;
    float *X, *P, *R, *C;
    const int64_t *record;
    int64_t nrecord;
    float *energy;
    int64_t k0, k1;                           // this launch runs steps k0 .. k1 - 1 and stops at k1
    float h, half_h, eg, decay, gain, eps;    // half_h = -h/2, eg = expm1(-gamma h)
};

// Two float32 lanes in one 64-bit register, and the paired add and FMA on
// them (PTX add/fma.rn.f32x2: two independent round-to-nearest operations).
__device__ __forceinline__ uint64_t pack2(float lo, float hi)
{
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

__device__ __forceinline__ void unpack2(uint64_t v, float &lo, float &hi)
{
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}

__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b)
{
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c)
{
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}

// First index r with record[r] >= k (record ascending).
__device__ __forceinline__ int64_t first_record_at_or_after(const int64_t *record, int64_t nrecord, int64_t k)
{
    int64_t lo = 0, hi = nrecord;
    while (lo < hi) {
        const int64_t mid = lo + (hi - lo) / 2;
        if (record[mid] < k)
            lo = mid + 1;
        else
            hi = mid;
    }
    return lo;
}

// Step index of record[r] relative to the launch start, or -1 when there is
// none within this launch.
__device__ __forceinline__ int record_in_launch(const QuadParams &q, int64_t r, int steps)
{
    if (r >= q.nrecord)
        return -1;
    const int64_t rel = q.record[r] - q.k0;
    return rel <= steps ? (int)rel : -1;
}

// exp(z) - 1.  For |z| <= 1/16 the exponential series without its constant
// term, z (1 + z/2 (1 + z/3 (1 + z/4 (1 + z/5)))) written in Horner form with
// the coefficients 1/k!: the first omitted term, z^6/720, is below 1.3e-9 of
// the result.  Larger |z| use the library's expm1f.
__device__ __forceinline__ float expm1_small(float z)
{
    if (fabsf(z) <= 0.0625f)
        return z * fmaf(z, fmaf(z, fmaf(z, fmaf(z, 1.f / 120.f, 1.f / 24.f), 1.f / 6.f), 0.5f), 1.f);
    return expm1f(z);
}

template <int MB, int NB>
struct QShape {
    static constexpr int L = MB * NB >= 32 ? 32 : (MB * NB < 4 ? 4 : MB * NB);   // lanes per system
    // Row stride of the row-major copy and column stride of the column-major
    // copy: an extent that is a multiple of 8 floats gets 4 more, so that
    // consecutive rows (columns) start in different 16-byte bank groups.
    static constexpr int RS = NB % 8 == 0 ? NB + 4 : NB;
    static constexpr int CS = MB % 8 == 0 ? MB + 4 : MB;
    static constexpr int BLK = ((MB * RS > NB * CS ? MB * RS : NB * CS) + 3) / 4 * 4;   // floats per system
    static_assert((32 / L) * BLK <= kQBufFloats, "padded blocks must fit the warp's buffer");
};

// Sum of K consecutive floats at p (16-byte aligned when K >= 4), in a fixed
// order: for K >= 4 the even- and odd-placed elements are summed as the two
// halves of paired adds (PTX add.rn.f32x2), then the two halves are added.
template <int K>
__device__ __forceinline__ float sum_run(const float *p)
{
    if constexpr (K >= 4) {
        const ulonglong2 *v = reinterpret_cast<const ulonglong2 *>(p);
        ulonglong2 w = v[0];
        uint64_t acc = add2(w.x, w.y);
#pragma unroll
        for (int q = 1; q < K / 4; ++q) {
            w = v[q];
            acc = add2(acc, w.x);
            acc = add2(acc, w.y);
        }
        float lo, hi;
        unpack2(acc, lo, hi);
        return lo + hi;
    } else {
        float s0 = 0.f;
#pragma unroll
        for (int q = 0; q < K; ++q)
            s0 += p[q];
        return s0;
    }
}

template <int MB, int NB>
__global__ void __launch_bounds__(kQThreads, kQMinBlocks) rikfad_quadratic_kernel(QuadParams q)
{
    constexpr int L = QShape<MB, NB>::L;
    constexpr int RS = QShape<MB, NB>::RS;
    constexpr int CS = QShape<MB, NB>::CS;
    constexpr int BLK = QShape<MB, NB>::BLK;
    __shared__ __align__(16) float xs[kQWarps][2][32];
    __shared__ __align__(16) float sr[kQWarps][2][kQBufFloats];  // row-major, row stride RS
    __shared__ __align__(16) float sc[kQWarps][2][kQBufFloats];  // column-major, column stride CS
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int a = lane & (L - 1);             // element within the system
    const int base = lane - a;                // first lane of the system's group
    const int pbase = (lane / L) * BLK;       // the system's padded blocks
    const int64_t sys = ((int64_t)blockIdx.x * kQWarps + warp) * (32 / L) + lane / L;
    const bool live = sys < q.batch;
    const int m = q.m, n = q.n, d = q.d;
    const bool elem = live && a < d;
    const int i = elem ? a / n : 0;
    const int j = elem ? a - i * n : 0;

    // Row a of A as packed pairs (A_a,2c, A_a,2c+1) for the paired FMAs below.
    uint64_t arow2[L / 2];
#pragma unroll
    for (int c = 0; c < L / 2; ++c) {
        const float lo = (elem && 2 * c < d) ? q.A[(sys * d + a) * d + 2 * c] : 0.f;
        const float hi = (elem && 2 * c + 1 < d) ? q.A[(sys * d + a) * d + 2 * c + 1] : 0.f;
        arow2[c] = pack2(lo, hi);
    }
    float x = elem ? q.X[sys * d + a] : 0.f;
    float pb = elem ? q.P[sys * d + a] : 0.f;   // P_k0 at the launch's first step, then P^(B)
    float Ri = 0.f, Cj = 0.f, S = 0.f;
    if (live) {
        Ri = q.R[sys * m + i];
        Cj = q.C[sys * n + j];
        for (int t = 0; t < m; ++t)
            S += q.R[sys * m + t];
    }
    float e1 = 0.f;                           // pending expm1(-h/2 xi~_{k-1})
    int cur = 0;
#pragma unroll
    for (int u = 0; u < 2; ++u) {
        xs[warp][u][lane] = 0.f;
#pragma unroll
        for (int v = 0; v < kQBufFloats; v += 32) {
            sr[warp][u][lane + v] = 0.f;
            sc[warp][u][lane + v] = 0.f;
        }
    }
    __syncwarp();
    xs[warp][0][lane] = x;
    __syncwarp();

    const int steps = (int)(q.k1 - q.k0);
    int64_t ri = q.nrecord > 0 ? first_record_at_or_after(q.record, q.nrecord, q.k0) : 0;
    int next = record_in_launch(q, ri, steps);
    for (int s = 0;; ++s) {
        // Friction of the current factors and the damping owed since P^(B)
        // (none at the launch's first step, which starts from P_k itself).
        const float den = S + q.eps;
        const float inv = den > 0.f ? __fdividef(1.f, den) : 0.f;
        const float z2 = ((Ri * inv) * Cj) * q.half_h;
        const float e2 = expm1_small(z2);
        // expm1 of the owed exponent -h/2 (xi~_{k-1} + xi~_k) - gamma h from
        // the two half-damps' expm1 values: (1 + e1)(1 + e2)(1 + eg) - 1,
        // every term of one sign (no cancellation).
        float em = fmaf(e1, e2, e1 + e2);
        em = fmaf(q.eg, 1.f + em, em);
        if (s == 0)
            em = 0.f;
        // g = A vec(X): four partial sums over the columns 4c, 4c+1, 4c+2,
        // 4c+3, carried as two pairs and advanced by paired FMAs (each half
        // a round-to-nearest FMA, so the same arithmetic as four fmaf).
        const ulonglong2 *xv = reinterpret_cast<const ulonglong2 *>(&xs[warp][cur][base]);
        uint64_t g01 = 0ull, g23 = 0ull;
#pragma unroll
        for (int b4 = 0; b4 < L / 4; ++b4) {
            const ulonglong2 v = xv[b4];
            g01 = fma2(arow2[2 * b4], v.x, g01);
            g23 = fma2(arow2[2 * b4 + 1], v.y, g23);
        }
        float g0, g1, g2, g3;
        unpack2(g01, g0, g1);
        unpack2(g23, g2, g3);
        const float g = (g0 + g1) + (g2 + g3);
        while (s == next) {                   // energy of the state after k0 + s steps
            const float pk = fmaf(pb, em, pb);
            float e = 0.5f * x * g + 0.5f * pk * pk;
#pragma unroll
            for (int o = L / 2; o > 0; o >>= 1)
                e += __shfl_xor_sync(0xffffffffu, e, o);
            if (live && a == 0)
                q.energy[ri * q.batch + sys] = e;
            ++ri;
            next = record_in_launch(q, ri, steps);
        }
        if (s == steps) {
            if (elem) {
                q.X[sys * d + a] = x;
                q.P[sys * d + a] = fmaf(pb, em, pb);
                if (j == 0)
                    q.R[sys * m + i] = Ri;
                if (i == 0)
                    q.C[sys * n + j] = Cj;
            }
            return;
        }
        pb = pb + fmaf(-q.h, g, pb * em);     // B (with the owed damping)
        x = fmaf(q.h, pb, x);                 // A
        const float p1 = fmaf(pb, e2, pb);    // C, first half
        const float p1sq = p1 * p1;
        e1 = e2;
        xs[warp][cur ^ 1][lane] = x;
        if (elem) {
            sr[warp][cur][pbase + i * RS + j] = p1sq;
            sc[warp][cur][pbase + j * CS + i] = p1sq;
        }
        // Total of [P^(1)]^2 over the system: an xor butterfly within the
        // group.  Partners add the same two numbers, so every lane ends with
        // the same bits.
        float tot = elem ? p1sq : 0.f;
#pragma unroll
        for (int o = L / 2; o > 0; o >>= 1)
            tot += __shfl_xor_sync(0xffffffffu, tot, o);
        __syncwarp();
        // Factor filter: row sum and column sum, in a fixed order.
        const float rs = sum_run<NB>(&sr[warp][cur][pbase + i * RS]);
        const float cs = sum_run<MB>(&sc[warp][cur][pbase + j * CS]);
        Ri = fmaf(q.gain, rs, q.decay * Ri);
        Cj = fmaf(q.gain, cs, q.decay * Cj);
        S = fmaf(q.gain, tot, q.decay * S);
        cur ^= 1;
    }
}

int q_fail(int code, const char *msg) { return rikfad::report_error(code, msg); }

template <int MB, int NB>
cudaError_t launch_all(QuadParams q, int64_t nsteps, int64_t per_launch, cudaStream_t s)
{
    constexpr int L = QShape<MB, NB>::L;
    const int64_t groups = (q.batch + (32 / L) - 1) / (32 / L);   // warps
    const int64_t blocks = (groups + kQWarps - 1) / kQWarps;
    for (int64_t k0 = 0;; k0 += per_launch) {
        q.k0 = k0;
        q.k1 = k0 + per_launch < nsteps ? k0 + per_launch : nsteps;
        rikfad_quadratic_kernel<MB, NB><<<(unsigned)blocks, kQThreads, 0, s>>>(q);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess || q.k1 == nsteps)
            return e;
    }
}

template <int MB>
cudaError_t dispatch_nb(int nb, QuadParams q, int64_t nsteps, int64_t per_launch, cudaStream_t s)
{
    switch (nb) {
    case 1: return launch_all<MB, 1>(q, nsteps, per_launch, s);
    case 2: return launch_all<MB, 2>(q, nsteps, per_launch, s);
    case 4:
        if constexpr (MB <= 16)
            return launch_all<MB, 4>(q, nsteps, per_launch, s);
        break;
    case 8:
        if constexpr (MB <= 8)
            return launch_all<MB, 8>(q, nsteps, per_launch, s);
        break;
    case 16:
        if constexpr (MB <= 4)
            return launch_all<MB, 16>(q, nsteps, per_launch, s);
        break;
    case 32:
        if constexpr (MB <= 2)
            return launch_all<MB, 32>(q, nsteps, per_launch, s);
        break;
    default: break;
    }
    return cudaErrorInvalidValue;
}

int pow2_ceil(int v)
{
    int p = 1;
    while (p < v)
        p <<= 1;
    return p;
}

}  // namespace

extern "C" RIKFAD_API int rikfad_quadratic_run(int64_t batch, int64_t m, int64_t n, const float *A,
                                               float *X, float *P, float *R, float *C, double step,
                                               const rikfad_hparams *hp, int64_t nsteps,
                                               const int64_t *record, int64_t nrecord, float *energy,
                                               void *stream)
{
    if (batch < 0 || batch > ((int64_t)1 << 24))
        return q_fail(RIKFAD_ERR_ARG, "batch must be in [0, 2^24]");
    if (m < 1 || n < 1 || m * n > kQMaxDim)
        return q_fail(RIKFAD_ERR_ARG, "need m >= 1, n >= 1 and m * n <= 32");
    if (nsteps < 0 || nrecord < 0)
        return q_fail(RIKFAD_ERR_ARG, "nsteps and nrecord must be >= 0");
    if (hp == nullptr)
        return q_fail(RIKFAD_ERR_ARG, "hp is NULL");
    if (!(std::isfinite(hp->alpha) && hp->alpha > 0) || !(hp->mu > 0) ||
        !(std::isfinite(hp->gamma) && hp->gamma >= 0) ||
        !(std::isfinite(hp->eps_stab) && hp->eps_stab >= 0))
        return q_fail(RIKFAD_ERR_ARG, "hyperparameters out of range");
    if (!(std::isfinite(step) && step > 0))
        return q_fail(RIKFAD_ERR_ARG, "step must be finite and > 0");
    if (batch > 0 && (A == nullptr || X == nullptr || P == nullptr || R == nullptr || C == nullptr))
        return q_fail(RIKFAD_ERR_ARG, "NULL state pointer");
    if (batch > 0 && nrecord > 0 && (record == nullptr || energy == nullptr))
        return q_fail(RIKFAD_ERR_ARG, "NULL record or energy pointer");
    if ((uintptr_t)A % 4 || (uintptr_t)X % 4 || (uintptr_t)P % 4 || (uintptr_t)R % 4 ||
        (uintptr_t)C % 4 || (uintptr_t)energy % 4 || (uintptr_t)record % 8)
        return q_fail(RIKFAD_ERR_ALIGN, "misaligned pointer");
    if (batch == 0)
        return RIKFAD_OK;

    QuadParams q{};
    q.batch = batch;
    q.m = (int)m;
    q.n = (int)n;
    q.d = (int)(m * n);
    q.A = A;
    q.X = X;
    q.P = P;
    q.R = R;
    q.C = C;
    q.record = nrecord > 0 ? record : nullptr;
    q.nrecord = nrecord;
    q.energy = energy;
    q.h = (float)step;
    q.half_h = (float)(-0.5 * step);
    q.eg = (float)std::expm1(-hp->gamma * step);
    q.decay = (float)std::exp(-hp->alpha * step);
    q.gain = std::isinf(hp->mu) ? 0.f : (float)(-std::expm1(-hp->alpha * step) / (hp->mu * hp->alpha));
    q.eps = (float)hp->eps_stab;

    // Launches of per_launch steps: 2^16, or the largest power of two that
    // keeps a launch within 2^31 system-steps (at least 128 for batch <=
    // 2^24), so that no launch runs for more than about a second.
    int64_t per_launch = (int64_t)1 << 16;
    while (per_launch > 128 && per_launch * batch > ((int64_t)1 << 31))
        per_launch >>= 1;

    const int mb = pow2_ceil((int)m), nb = pow2_ceil((int)n);   // mb nb <= 64 when m n <= 32
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e;
    switch (mb) {
    case 1: e = dispatch_nb<1>(nb, q, nsteps, per_launch, s); break;
    case 2: e = dispatch_nb<2>(nb, q, nsteps, per_launch, s); break;
    case 4: e = dispatch_nb<4>(nb, q, nsteps, per_launch, s); break;
    case 8: e = dispatch_nb<8>(nb, q, nsteps, per_launch, s); break;
    case 16: e = dispatch_nb<16>(nb, q, nsteps, per_launch, s); break;
    default: e = dispatch_nb<32>(nb, q, nsteps, per_launch, s); break;
    }
    if (e != cudaSuccess)
        return q_fail(RIKFAD_ERR_CUDA, cudaGetErrorString(e));
    return RIKFAD_OK;
}
