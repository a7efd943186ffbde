// rikfad_sweep.cuh -- the in-order ("sweep") schedule of the R-iKFAD step
// (opt-in: RIKFAD_SCHEDULE=sweep; the default is the static schedule).
//
// Persistent blocks take units from a global counter in memory order, so at
// any moment the whole GPU streams through a narrow window of HBM.  A bare
// stream probe gained ~6% on GB300 this way, but here every unit also needs
// an acquire/release arrival and block barriers; measured on GPT2-S the
// sweep reaches 83% of the copy peak against 93.6% for the static schedule,
// so it is not the default.  A
// matrix unit is up to kUnitRows rows of one column panel, one row per warp,
// processed by the same per-row code as the static schedule.  Each unit
// writes its column partial sums of [P^(1)]^2 to its own slot; the partials
// of a panel are combined up a static kTreeFan-ary tree, in a fixed order, by
// the block that completes a node's last child, and the consumed slots are
// dropped from L2 without being written back (discard.global.L2), so the
// partials cost L2 bandwidth only.  The block that completes a tensor's last
// panel applies the factor filter (R, C, the partial sums of R) in the same
// launch, so a step is one kernel.  Sums are in a fixed order whatever block
// does them: results are bitwise reproducible.
//
// No block ever waits on another: completion is detected with one atomic per
// arrival, and the last arriver does the work.  The last block to leave
// resets the unit counter for the next launch.
#pragma once
#include "rikfad_kernels.cuh"

namespace rikfad {

// Blocks per SM the sweep kernel's registers are sized for (4: 64 registers).
#ifndef RIKFAD_SWEEP_MIN_BLOCKS
#define RIKFAD_SWEEP_MIN_BLOCKS 4
#endif

struct SweepParams {
    const UnitDev *units;
    const NodeDev *nodes;
    const PanelTreeDev *trees;
    int64_t nunits;
    float *partials;
    float *spart;                  // partial sums of R (written by tensor finishers)
    int32_t *node_count;
    int32_t *tensor_count;
    unsigned long long *fetch;
    unsigned int *exits;
};

__device__ __forceinline__ void discard_l2_line(const float *p)
{
    asm volatile("discard.global.L2 [%0], 128;" ::"l"(p) : "memory");
}

__device__ __forceinline__ int atomic_add_acq_rel_gpu(int32_t *p, int v)
{
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// One arrival of this block at a counter that completes after `expected`
// arrivals; returns (to every thread) whether this block was the last.  The
// block barrier orders every thread's earlier writes before thread 0's
// release; thread 0's acquire and the second barrier order the last
// arrival's later reads after every other arrival's writes.  No thread waits
// for its own streaming stores.
__device__ __forceinline__ bool block_arrive(int32_t *counter, int32_t expected, int *flag)
{
    __syncthreads();
    if (threadIdx.x == 0)
        *flag = atomic_add_acq_rel_gpu(counter, 1) == expected - 1;
    __syncthreads();
    return *flag != 0;
}

// Factor filter of one tensor once all its units are done (same arithmetic
// and order as rikfad_finalize_kernel for R and its partial sums).
__device__ __forceinline__ void finish_tensor(const StepParams &a, const SweepParams &s, int t,
                                              float *wsum)
{
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const TensorDev td = a.tensors[t];
    float *R = a.fac + td.fac_off;
    for (int ch = 0; ch < td.spart_cnt; ++ch) {
        const int64_t i = (int64_t)ch * kThreads + tid;
        float val = 0.f;
        if (i < td.rows) {
            float acc = 0.f;
            const float *rp = a.rowpart + td.rowpart_off + i;
            for (int k = 0; k < td.npanels; ++k)
                acc += __ldcg(rp + (int64_t)k * td.rows);
            val = fmaf(a.gain, acc, a.decay * R[i]);
            R[i] = val;
            if (!isfinite(val))
                report_nonfinite(a.guard, t);
        }
        val = warp_sum(val);
        if (lane == 0)
            wsum[warp] = val;
        __syncthreads();
        if (tid < 32) {
            float v = tid < kWarps ? wsum[tid] : 0.f;
            v = warp_sum(v);
            if (tid == 0) {
                s.spart[td.spart_off + ch] = v;
                if (!isfinite(v))
                    report_nonfinite(a.guard, t);
            }
        }
        __syncthreads();
    }
    for (int k = 0; k < td.npanels; ++k) {
        const PanelDev pd = a.panels[td.panel0 + k];
        const PanelTreeDev tr = s.trees[td.panel0 + k];
        float *C = a.fac + td.fac_off + td.rows + pd.col0;
        for (int c = tid; c < pd.width; c += kThreads) {
            const float sum = td.rows > 0 ? __ldcg(s.partials + tr.root_off + c) : 0.f;
            const float cn = fmaf(a.gain, sum, a.decay * C[c]);
            C[c] = cn;
            if (!isfinite(cn))
                report_nonfinite(a.guard, t);
        }
        if (td.rows > 0) {
            __syncthreads();
            for (int l = tid; l < tr.slot / 32; l += kThreads)
                discard_l2_line(s.partials + tr.root_off + (int64_t)l * 32);
        }
    }
    if (tid == 0)
        s.tensor_count[t] = 0;
    __syncthreads();
}

// Combine tree node `node` (this block was its last arrival) and climb while
// this block keeps being the last arrival; at a panel's root, count the panel
// at its tensor and finish the tensor if it was the last panel.
__device__ __forceinline__ void climb(const StepParams &a, const SweepParams &s, int node, int t,
                                      int *flag, float *wsum)
{
    const int tid = threadIdx.x;
    for (;;) {
        const NodeDev nd = s.nodes[node];
        const int slot = s.trees[nd.panel].slot;
        const int wn = a.panels[nd.panel].width;
        for (int c = tid; c < wn; c += kThreads) {
            float acc = 0.f;
            for (int k = 0; k < nd.nchildren; ++k)
                acc += __ldcg(s.partials + nd.first_child_off + (int64_t)k * slot + c);
            s.partials[nd.off + c] = acc;
        }
        __syncthreads();
        const int lines = nd.nchildren * slot / 32;
        for (int l = tid; l < lines; l += kThreads)
            discard_l2_line(s.partials + nd.first_child_off + (int64_t)l * 32);
        if (tid == 0)
            s.node_count[node] = 0;
        if (nd.parent < 0) {
            if (block_arrive(&s.tensor_count[t], a.tensors[t].npanels, flag))
                finish_tensor(a, s, t, wsum);
            return;
        }
        node = nd.parent;
        if (!block_arrive(&s.node_count[node], s.nodes[node].nchildren, flag))
            return;
    }
}

template <typename GT, bool REUSE>
__global__ void __launch_bounds__(kThreads, RIKFAD_SWEEP_MIN_BLOCKS)
    rikfad_sweep_kernel(StepParams a, SweepParams s)
{
    __shared__ __align__(16) float Cs[kPanelMax];
    __shared__ __align__(16) float red[kWarps * kPanelMax];
    __shared__ long long s_unit;
    __shared__ int s_flag;
    __shared__ float wsum[kWarps];
    const int tid = threadIdx.x;
    int cached_panel = -1;
    float inv = 0.f;
    if (tid == 0)
        s_unit = (long long)atomicAdd(s.fetch, 1ull);
    for (;;) {
        __syncthreads();
        const long long u = s_unit;
        __syncthreads();
        if (u >= s.nunits)
            break;
        // Take the next ticket now; its latency overlaps this unit.
        if (tid == 0)
            s_unit = (long long)atomicAdd(s.fetch, 1ull);
        const UnitDev un = s.units[u];
        const TensorDev td = a.tensors[un.tensor];
        if (un.kind == kUnitVector) {
            PieceDev pc{};
            pc.kind = kElements;
            pc.tensor = un.tensor;
            pc.begin = un.begin;
            pc.end = un.end;
            vector_piece<GT>(a, pc, td);
            continue;
        }
        if (un.kind == kUnitFactorsOnly) {      // a matrix with no rows: C only decays
            finish_tensor(a, s, un.tensor, wsum);
            continue;
        }
        const PanelDev pd = a.panels[un.panel];
        const int w = pd.width;
        if (un.panel != cached_panel) {
            const float *C = a.fac + td.fac_off + td.rows + pd.col0;
            for (int c = tid; c < w; c += kThreads)
                Cs[c] = C[c];
            inv = inv_denominator(row_total(a.spart, td), a.eps);
            cached_panel = un.panel;
            __syncthreads();
        }
        PieceDev pc{};
        pc.kind = kMatrixRows;
        pc.tensor = un.tensor;
        pc.panel = un.panel;
        pc.begin = un.begin;
        pc.end = un.end;
        if (td.vec)
            matrix_piece_vec<GT, REUSE, false>(a, pc, td, pd, Cs, red, inv);
        else
            matrix_piece_scalar<GT, REUSE, false>(a, pc, td, pd, Cs, red, inv);
        __syncthreads();
        // Column partial of the unit: its rows' squares, warps in order.
        const int nrows = (int)(un.end - un.begin);
        float *leaf = s.partials + un.leaf_off;
        for (int c = tid; c < w; c += kThreads) {
            float acc = 0.f;
            for (int k = 0; k < nrows; ++k)
                acc += red[k * kPanelMax + c];
            leaf[c] = acc;
        }
        // Count this unit at its tree node; the last arrival combines the node
        // and climbs while it keeps being the last.
        if (block_arrive(&s.node_count[un.parent], s.nodes[un.parent].nchildren, &s_flag))
            climb(a, s, un.parent, un.tensor, &s_flag, wsum);
    }
    // The last block to leave resets the unit counter for the next launch
    // (every block has taken its final, out-of-range ticket by now).
    if (tid == 0) {
        __threadfence();
        if (atomicAdd(s.exits, 1u) == gridDim.x - 1) {
            *s.fetch = 0ull;
            *s.exits = 0u;
            __threadfence();
        }
    }
}

}  // namespace rikfad
