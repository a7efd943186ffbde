// rikfad_checks.cuh -- device-side checks of the work plan (checked builds).
//
// A library compiled with -DRIKFAD_CHECKED verifies, before every access a
// plan entry drives, that the entry lies within the extents the planner
// produced (CheckBounds): block and piece indices, tensor and panel
// indices, row and column ranges, offsets into the factor, row-partial,
// column-partial and denominator buffers, and the pointer-table entries
// (non-null, aligned for the vector loads).  A failed check increments an
// error counter and skips the access: nothing traps and nothing waits.  In
// other builds every check compiles to `true` and its operands are never
// evaluated.
#pragma once
#include <stdint.h>

#include "rikfad_plan.hpp"

namespace rikfad {

enum CheckCode : int32_t {
    kChkBlock = 1,      // block index or its piece range
    kChkTensor = 2,     // tensor index
    kChkKind = 3,       // piece or item kind
    kChkPanel = 4,      // panel index, or the panel's tensor
    kChkRows = 5,       // row or element range
    kChkCols = 6,       // column range of a panel
    kChkFactors = 7,    // R, C or friction offset
    kChkRowpart = 8,    // row-partial offset
    kChkColpart = 9,    // column-partial slot or offset
    kChkSpart = 10,     // partial sums of R
    kChkPointer = 11,   // NULL pointer-table entry
    kChkAlign = 12,     // pointer not 16-byte aligned for the 8-wide path
    kChkFinItem = 13,   // finalise item
};

#ifdef RIKFAD_CHECKED
__device__ __forceinline__ bool check_ok(const CheckBounds &cb, bool cond, int code)
{
    if (!cond) {
        atomicAdd(cb.errors, 1);
        atomicCAS(cb.errors + 1, 0, code);
    }
    return cond;
}
#define RK_DEV_CHECK(cb, cond, code) ::rikfad::check_ok((cb), (cond), (code))
#else
#define RK_DEV_CHECK(cb, cond, code) true
#endif

__device__ __forceinline__ bool aligned16(const void *p)
{
    return ((uintptr_t)p & 15u) == 0;
}

// Checks of one piece of a block's share: its tensor, panel, slot and row
// (element) range, the buffer offsets they lead to, and the tensor's
// pointers.  `td` and `pd` are only read after the indices that select them
// have passed (the caller loads them through piece_tensor_ok / piece_panel_ok).
__device__ __forceinline__ bool piece_tensor_ok(const CheckBounds &cb, const PieceDev &pc)
{
    return RK_DEV_CHECK(cb, pc.tensor >= 0 && pc.tensor < cb.ntensors, kChkTensor) &&
           RK_DEV_CHECK(cb, pc.kind == kMatrixRows || pc.kind == kElements, kChkKind);
}

__device__ __forceinline__ bool piece_panel_ok(const CheckBounds &cb, const PieceDev &pc,
                                               const TensorDev &td)
{
    return RK_DEV_CHECK(cb, td.cols > 0, kChkKind) &&
           RK_DEV_CHECK(cb, pc.panel >= td.panel0 && pc.panel < td.panel0 + td.npanels &&
                                pc.panel >= 0 && pc.panel < cb.npanels, kChkPanel);
}

// x, g, p: the tensor's pointer-table entries.  slots: whether the piece
// writes a column partial (the step kernel) or not (the canonical pass).
__device__ __forceinline__ bool matrix_piece_ok(const CheckBounds &cb, const PieceDev &pc,
                                                const TensorDev &td, const PanelDev &pd,
                                                const void *x, const void *g, const void *p,
                                                bool slots)
{
    (void)cb; (void)pc; (void)td; (void)pd; (void)x; (void)g; (void)p; (void)slots;
    bool ok = RK_DEV_CHECK(cb, pd.tensor == pc.tensor, kChkPanel) &&
              RK_DEV_CHECK(cb, pc.begin >= 0 && pc.begin <= pc.end && pc.end <= td.rows, kChkRows) &&
              RK_DEV_CHECK(cb, pd.col0 >= 0 && pd.width >= 1 && pd.width <= kPanelMax &&
                                   (int64_t)pd.col0 + pd.width <= td.cols, kChkCols) &&
              RK_DEV_CHECK(cb, td.fac_off >= 0 && td.fac_off + td.rows + td.cols <= cb.fac_floats,
                           kChkFactors) &&
              RK_DEV_CHECK(cb, !td.full || (td.xi_off >= 0 &&
                                            td.xi_off + td.rows * td.cols <= cb.fac_floats), kChkFactors) &&
              RK_DEV_CHECK(cb, td.spart_off >= 0 && (int64_t)td.spart_off + td.spart_cnt <= cb.spart_floats,
                           kChkSpart);
    if (ok && slots)
        ok = RK_DEV_CHECK(cb, td.rowpart_off >= 0 &&
                                  td.rowpart_off + (int64_t)td.npanels * td.rows <= cb.rowpart_floats,
                          kChkRowpart) &&
             RK_DEV_CHECK(cb, pc.slot >= pd.slot_begin && pc.slot < pd.slot_end && pc.slot >= 0 &&
                                  pc.slot < cb.nslots, kChkColpart) &&
             RK_DEV_CHECK(cb, pc.colpart_off >= 0 && pc.colpart_off + pd.width <= cb.colpart_floats,
                          kChkColpart);
    if (ok && pc.begin < pc.end)
        ok = RK_DEV_CHECK(cb, x != nullptr && p != nullptr && (g != nullptr || !slots), kChkPointer) &&
             RK_DEV_CHECK(cb, !td.vec || ((td.cols & 7) == 0 && (pd.col0 & 7) == 0 && (pd.width & 7) == 0 &&
                                          aligned16(x) && aligned16(p) && (!slots || aligned16(g))),
                          kChkAlign);
    return ok;
}

__device__ __forceinline__ bool vector_piece_ok(const CheckBounds &cb, const PieceDev &pc,
                                                const TensorDev &td, const void *x, const void *g,
                                                const void *p, bool has_grad)
{
    (void)cb; (void)pc; (void)td; (void)x; (void)g; (void)p; (void)has_grad;
    bool ok = RK_DEV_CHECK(cb, td.cols == 0, kChkKind) &&
              RK_DEV_CHECK(cb, pc.begin >= 0 && pc.begin <= pc.end && pc.end <= td.rows &&
                                   (pc.begin & 7) == 0, kChkRows) &&
              RK_DEV_CHECK(cb, td.fac_off >= 0 && td.fac_off + td.rows <= cb.fac_floats, kChkFactors);
    if (ok && pc.begin < pc.end)
        ok = RK_DEV_CHECK(cb, x != nullptr && p != nullptr && (g != nullptr || !has_grad), kChkPointer) &&
             RK_DEV_CHECK(cb, aligned16(x) && aligned16(p) && (!has_grad || aligned16(g)), kChkAlign);
    return ok;
}

// A block's piece range [q0, q1).
__device__ __forceinline__ bool block_ok(const CheckBounds &cb, int b, int q0, int q1)
{
    (void)cb; (void)b; (void)q0; (void)q1;
    return RK_DEV_CHECK(cb, b >= 0 && b < cb.nblocks, kChkBlock) &&
           RK_DEV_CHECK(cb, q0 >= 0 && q0 <= q1 && q1 <= cb.npieces, kChkBlock);
}

}  // namespace rikfad
