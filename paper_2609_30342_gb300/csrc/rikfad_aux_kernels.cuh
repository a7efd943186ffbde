// rikfad_aux_kernels.cuh -- the kernels around the step kernel: the factor
// finalise (run after every step), the canonical-momentum pass (checkpoints,
// tests) and the denominator read-back.  Included by rikfad.cu only.
#pragma once
#include "rikfad_kernels.cuh"

namespace rikfad {

struct DenParams {
    const TensorDev *tensors;
    const float *spart;
    float *out;
    int ntensors;
    CheckBounds chk;           // read by checked builds only
};

struct CanonParams {
    const TensorDev *tensors;
    const PanelDev *panels;
    const PieceDev *pieces;
    const int32_t *block_piece;
    const float *const *src;
    float *const *dst;
    const float *fac;
    const float *spart;
    float ex_prev;
    float damp_prev;
    float eps;
    CheckBounds chk;           // read by checked builds only
};

struct FinParams {
    const TensorDev *tensors;
    const PanelDev *panels;
    const FinItemDev *items;
    const int64_t *slot_off;
    float *fac;
    const float *rowpart;
    const float *colpart;
    float *spart;
    float decay;
    float gain;
    int resum_only;            // 1: only recompute the partial sums of R
    Guard guard;
    CheckBounds chk;           // read by checked builds only
};

// Checks of one finalise item (checked builds): its tensor, rows or panel
// and slots, and the offsets they lead to.
__device__ __forceinline__ bool fin_item_ok(const FinParams &f, const FinItemDev &it, const TensorDev &td)
{
    (void)f; (void)it; (void)td;
    const CheckBounds &cb = f.chk;
    (void)cb;
    if (!RK_DEV_CHECK(cb, td.cols > 0 && td.fac_off >= 0 && td.fac_off + td.rows + td.cols <= cb.fac_floats,
                      kChkFactors))
        return false;
    if (it.kind == kFinRows)
        return RK_DEV_CHECK(cb, it.begin >= 0 && it.begin <= it.end && it.end <= td.rows, kChkRows) &&
               RK_DEV_CHECK(cb, it.chunk >= 0 && it.chunk < td.spart_cnt && td.spart_off >= 0 &&
                                    (int64_t)td.spart_off + td.spart_cnt <= cb.spart_floats, kChkSpart) &&
               RK_DEV_CHECK(cb, f.resum_only || (td.rowpart_off >= 0 &&
                                    td.rowpart_off + (int64_t)td.npanels * td.rows <= cb.rowpart_floats),
                            kChkRowpart);
    if (!RK_DEV_CHECK(cb, it.kind == kFinCols, kChkKind) ||
        !RK_DEV_CHECK(cb, it.panel >= td.panel0 && it.panel < td.panel0 + td.npanels && it.panel >= 0 &&
                              it.panel < cb.npanels, kChkPanel))
        return false;
    if (f.resum_only)
        return true;
    const PanelDev pd = f.panels[it.panel];
    const int ns = pd.slot_end - pd.slot_begin;
    (void)ns;                  // read by the checks only
    return RK_DEV_CHECK(cb, pd.tensor == it.tensor && pd.col0 >= 0 &&
                                (int64_t)pd.col0 + pd.width <= td.cols, kChkCols) &&
           RK_DEV_CHECK(cb, it.begin >= 0 && it.begin <= it.end && it.end <= pd.width, kChkCols) &&
           RK_DEV_CHECK(cb, pd.slot_begin >= 0 && ns >= 0 && pd.slot_end <= cb.nslots &&
                                (it.chunk != 0 || ns <= kFinSplitSlots), kChkColpart) &&
           RK_DEV_CHECK(cb, ns == 0 || (f.slot_off[pd.slot_begin] >= 0 &&
                                        f.slot_off[pd.slot_begin] + (int64_t)ns * pd.width <= cb.colpart_floats),
                        kChkColpart);
}


// ---------------------------------------------------- finalise kernel
//
// R_{n+1} = e^{-alpha h} R_n + k sum_panels rowpart,
// C_{n+1} = e^{-alpha h} C_n + k sum_slots colpart,
// and the partial sums of R_{n+1} that give 1^T R_{n+1}.
//
// A row item is kFinThreads rows, one thread per row.  A column item of a
// panel with few slots is up to 256 columns, one thread per column adding the
// slots in order; a panel with many slots (more than kFinSplitSlots) gets
// items of kFinColChunk (32) columns: warp w adds the slots slot_begin + w,
// + 8, ... for the 32 columns (coalesced 128-byte rows of the partials), then
// warp 0 adds the eight warp sums in order.
__global__ void __launch_bounds__(kFinThreads) rikfad_finalize_kernel(FinParams f)
{
    __shared__ float wsum[kFinThreads / 32];
    __shared__ float csum[kFinThreads / 32][32];
    if (!RK_DEV_CHECK(f.chk, (int)blockIdx.x < f.chk.nfin, kChkFinItem))
        return;
    const FinItemDev it = f.items[blockIdx.x];
    if (!RK_DEV_CHECK(f.chk, it.tensor >= 0 && it.tensor < f.chk.ntensors, kChkTensor))
        return;
    const TensorDev td = f.tensors[it.tensor];
    wait_for_predecessor();
    allow_successor_launch();
    if (!fin_item_ok(f, it, td))
        return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (it.kind == kFinRows) {
        const int64_t i = it.begin + threadIdx.x;
        float val = 0.f;
        if (i < it.end) {
            float *R = f.fac + td.fac_off;
            if (f.resum_only) {
                val = R[i];
            } else {
                float acc = 0.f;
                const float *rp = f.rowpart + td.rowpart_off + i;
#pragma unroll 4
                for (int k = 0; k < td.npanels; ++k)
                    acc += rp[(int64_t)k * td.rows];
                val = fmaf(f.gain, acc, f.decay * R[i]);
                R[i] = val;
            }
            if (!isfinite(val))
                report_nonfinite(f.guard, it.tensor);
        }
        val = warp_sum(val);
        if (lane == 0)
            wsum[warp] = val;
        __syncthreads();
        if (threadIdx.x < 32) {
            float v = threadIdx.x < kFinThreads / 32 ? wsum[threadIdx.x] : 0.f;
            v = warp_sum(v);
            if (threadIdx.x == 0) {
                f.spart[td.spart_off + it.chunk] = v;
                if (!isfinite(v))       // finite R whose sum overflows
                    report_nonfinite(f.guard, it.tensor);
            }
        }
    } else if (!f.resum_only && it.chunk == 0) {
        // A panel's slots are consecutive in colpart, pd.width apart (the
        // planner checks this), so every slot's load is issued at once and
        // the sum is still taken in slot order.
        const PanelDev pd = f.panels[it.panel];
        const int64_t c = it.begin + threadIdx.x;
        if (c < it.end) {
            const int ns = pd.slot_end - pd.slot_begin;
            const float *cp = f.colpart + (ns > 0 ? f.slot_off[pd.slot_begin] : 0) + c;
            float v[kFinSplitSlots];
#pragma unroll
            for (int u = 0; u < kFinSplitSlots; ++u)
                v[u] = u < ns ? cp[(int64_t)u * pd.width] : 0.f;
            float acc = 0.f;
#pragma unroll
            for (int u = 0; u < kFinSplitSlots; ++u)
                if (u < ns)
                    acc += v[u];
            float *C = f.fac + td.fac_off + td.rows + pd.col0;
            const float cn = fmaf(f.gain, acc, f.decay * C[c]);
            C[c] = cn;
            if (!isfinite(cn))
                report_nonfinite(f.guard, it.tensor);
        }
    } else if (!f.resum_only) {
        const PanelDev pd = f.panels[it.panel];
        const int64_t c = it.begin + lane;
        float acc = 0.f;
        if (c < it.end) {
            const float *cp = f.colpart + f.slot_off[pd.slot_begin] + c;
#pragma unroll 4
            for (int s = warp; s < pd.slot_end - pd.slot_begin; s += kFinThreads / 32)
                acc += cp[(int64_t)s * pd.width];
        }
        csum[warp][lane] = acc;
        __syncthreads();
        if (warp == 0 && c < it.end) {
            float t = 0.f;
#pragma unroll
            for (int k = 0; k < kFinThreads / 32; ++k)
                t += csum[k][lane];
            float *C = f.fac + td.fac_off + td.rows + pd.col0;
            const float cn = fmaf(f.gain, t, f.decay * C[c]);
            C[c] = cn;
            if (!isfinite(cn))
                report_nonfinite(f.guard, it.tensor);
        }
    }
}

// ------------------------------------------- canonical momentum kernel
//
// dst = src exp(-(h_prev/2) xi~) e^{-gamma h_prev} for matrices (the same
// expression, in the same rounding order, as the start of the next step);
// vectors already hold P_{n+1} and are copied when dst != src.
__global__ void __launch_bounds__(kThreads) rikfad_canonical_kernel(CanonParams c)
{
    __shared__ float Cs[kPanelMax];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    wait_for_predecessor();
    allow_successor_launch();
    if (!RK_DEV_CHECK(c.chk, (int)blockIdx.x < c.chk.nblocks, kChkBlock))
        return;
    const int q0 = c.block_piece[blockIdx.x], q1 = c.block_piece[blockIdx.x + 1];
    if (!block_ok(c.chk, blockIdx.x, q0, q1))
        return;
    for (int q = q0; q < q1; ++q) {
        const PieceDev pc = c.pieces[q];
        if (!piece_tensor_ok(c.chk, pc))
            continue;
        const TensorDev td = c.tensors[pc.tensor];
        const float *S = c.src[pc.tensor];
        float *D = c.dst[pc.tensor];
        if (pc.kind == kElements) {
            if (S != D && vector_piece_ok(c.chk, pc, td, D, nullptr, S, false))
                for (int64_t e = pc.begin + threadIdx.x; e < pc.end; e += kThreads)
                    D[e] = S[e];
            continue;
        }
        if (!piece_panel_ok(c.chk, pc, td))
            continue;
        const PanelDev pd = c.panels[pc.panel];
        if (!matrix_piece_ok(c.chk, pc, td, pd, D, nullptr, S, false))
            continue;
        if (td.full) {      // element-wise friction: P already holds P_{n+1}
            if (S != D)
                for (int64_t row = pc.begin + warp; row < pc.end; row += kWarps)
                    for (int j = lane; j < pd.width; j += 32)
                        D[row * td.cols + pd.col0 + j] = S[row * td.cols + pd.col0 + j];
            continue;
        }
        const float *C = c.fac + td.fac_off + td.rows + pd.col0;
        for (int j = threadIdx.x; j < pd.width; j += kThreads)
            Cs[j] = C[j];
        const float inv = inv_denominator(row_total(c.spart, td), c.eps);
        __syncthreads();
        const float *R = c.fac + td.fac_off;
        for (int64_t row = pc.begin + warp; row < pc.end; row += kWarps) {
            const float a_prev = c.ex_prev * (R[row] * inv);
            const int64_t base = row * td.cols + pd.col0;
            if (td.vec) {
                // 16-byte aligned rows and panels: the whole panel row is
                // loaded first (at most kPanelMax / 128 float4 per lane), so
                // every load is in flight before the first in-place store.
                constexpr int kV = kPanelMax / 128;
                const float4 *s4 = reinterpret_cast<const float4 *>(S + base);
                float4 *d4 = reinterpret_cast<float4 *>(D + base);
                const int w4 = pd.width / 4;
                float4 v[kV];
#pragma unroll
                for (int k = 0; k < kV; ++k)
                    if (lane + 32 * k < w4)
                        v[k] = __ldcs(s4 + lane + 32 * k);
#pragma unroll
                for (int k = 0; k < kV; ++k) {
                    const int j4 = lane + 32 * k;
                    if (j4 < w4) {
                        const int j = 4 * j4;
                        v[k].x = (v[k].x * exp2f(a_prev * Cs[j])) * c.damp_prev;
                        v[k].y = (v[k].y * exp2f(a_prev * Cs[j + 1])) * c.damp_prev;
                        v[k].z = (v[k].z * exp2f(a_prev * Cs[j + 2])) * c.damp_prev;
                        v[k].w = (v[k].w * exp2f(a_prev * Cs[j + 3])) * c.damp_prev;
                        __stcs(d4 + j4, v[k]);
                    }
                }
            } else {
                for (int j = lane; j < pd.width; j += 32)
                    D[base + j] = (S[base + j] * exp2f(a_prev * Cs[j])) * c.damp_prev;
            }
        }
        __syncthreads();
    }
}

// 1^T R of every matrix (0 for vectors), same summation order as the kernels.
// d.out may be page-locked host memory mapped into the device's address
// space (the enqueued read-back writes there directly).
__global__ void rikfad_denominators_kernel(DenParams d)
{
    wait_for_predecessor();
    allow_successor_launch();
    const int t = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
    if (t >= d.ntensors)
        return;
    const TensorDev td = d.tensors[t];
    if (!RK_DEV_CHECK(d.chk, td.spart_off >= 0 && (int64_t)td.spart_off + td.spart_cnt <= d.chk.spart_floats,
                      kChkSpart))
        return;
    const float s = td.cols == 0 ? 0.f : row_total(d.spart, td);
    if ((threadIdx.x & 31) == 0)
        d.out[t] = s;
}

}  // namespace rikfad
