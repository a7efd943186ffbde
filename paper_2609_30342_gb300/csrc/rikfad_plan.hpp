// rikfad_plan.hpp -- work plan of the fused R-iKFAD step, shared by the host
// planner and the kernels.  Plain structs only; no CUDA types.
//
// The step over a whole parameter list is one streaming pass.  The planner
// cuts that pass into one contiguous share per thread block ("CTA") of
// nearly equal HBM traffic:
//   * a matrix is split into column panels of at most kPanelMax columns;
//     every row of a panel is one unit of work (a warp updates it and emits
//     its sum of squares);
//   * a non-matrix tensor is a run of elements.
// A block's share is a list of "pieces": a row range of one panel, or an
// element range of one vector.  Each matrix piece owns one "slot" of column
// partial sums, so the column sums of [P^(1)]^2 are reduced in a fixed order
// (slot order), without atomics: runs are bitwise reproducible.
#pragma once
#include <stdint.h>

namespace rikfad {

constexpr int kThreads = 256;        // threads of the step kernel
constexpr int kWarps = kThreads / 32;
constexpr int kPanelMax = 1024;      // widest column panel (floats staged in shared memory)
constexpr int kChunk = 256;          // columns one warp covers per pass (32 lanes x 8)
constexpr int kFinThreads = 256;     // threads of the finalise kernel (= rows per partial sum)
constexpr int kFinColChunk = 32;     // columns per split column item (8 warps share its slots)
constexpr int kFinSplitSlots = 8;    // panels with more slots than this get split column items
constexpr int kElemGranule = 8;      // element pieces start on multiples of 8 elements
constexpr int64_t kMinBlockBytes = 64 * 1024;   // smallest share worth a block
// The planner balances blocks on time, not bytes alone: each row of a matrix
// panel costs its compulsory bytes plus kRowCost bytes' worth of fixed work
// (loading R_i, the exponent scale, the row-sum shuffle, the row-partial
// store).  Measured on GB300, step-kernel bandwidth on single matrices of
// width w follows w * 18 / (w * 18 + 250) to within 2% from w = 64 to 2048;
// without the term, blocks holding narrow panels (a 1600-wide matrix's
// 64-column tail) finish last.
constexpr int64_t kRowCost = 256;

enum PieceKind : int32_t { kMatrixRows = 0, kElements = 1 };
enum FinKind : int32_t { kFinRows = 0, kFinCols = 1 };

struct TensorDev {
    int64_t rows;         // m (matrix) or element count (vector)
    int64_t cols;         // n, or 0 for a vector
    int64_t fac_off;      // R at fac_off (m floats), C at fac_off + m (n floats);
                          // vector: friction at fac_off (rows floats)
    int64_t rowpart_off;  // row sums of panel k at rowpart_off + k * rows
    int32_t npanels;
    int32_t panel0;       // index of the first panel
    int32_t spart_off;    // partial sums of R, one per kFinThreads rows
    int32_t spart_cnt;
    int32_t vec;          // 1: 8-wide vector loads (cols % 8 == 0)
    int32_t full;         // 1: matrix with element-wise friction (full iKFAD) whose R, C are
                          //    shadow factors fed by the same momentum (diagnostics)
    int64_t xi_off;       // full: friction of the m x n elements at fac + xi_off (row-major)
};

struct PanelDev {
    int32_t tensor;
    int32_t col0;
    int32_t width;
    int32_t nch;          // ceil(width / kChunk)
    int32_t slot_begin;   // column partial slots of this panel: [slot_begin, slot_end)
    int32_t slot_end;
};

struct PieceDev {
    int32_t kind;
    int32_t tensor;
    int32_t panel;        // matrix pieces
    int32_t slot;         // matrix pieces
    int64_t begin;        // first row (matrix) or element (vector)
    int64_t end;
    int64_t colpart_off;  // matrix pieces: offset of the slot's width floats
};

struct FinItemDev {
    int32_t kind;
    int32_t tensor;
    int32_t panel;        // kFinCols
    int32_t chunk;        // kFinRows: index of the partial sum of R within the tensor;
                          // kFinCols: 1 = split item (warps share the slots), 0 = one thread per column
    int64_t begin;        // kFinRows: rows; kFinCols: columns relative to the panel
    int64_t end;
};

// Extents every plan index and offset must stay within.  Kernels of a build
// with RIKFAD_CHECKED verify each index against these before using it; a
// failed check is counted in errors[0] (errors[1] keeps the code of the
// first) and the access it guarded is skipped.  Other builds never read them.
struct CheckBounds {
    int32_t ntensors;
    int32_t npanels;
    int32_t npieces;
    int32_t nblocks;
    int32_t nfin;
    int32_t nslots;
    int64_t fac_floats;
    int64_t rowpart_floats;
    int64_t colpart_floats;
    int64_t spart_floats;
    int32_t *errors;
};

// ------------------------------------------------------------------------
// In-order schedule ("sweep"): persistent blocks take small units of work
// from a global counter in memory order, so the whole GPU streams through a
// narrow window of HBM at a time.  A matrix unit is up to kUnitRows rows of
// one panel (one row per warp); a vector unit is up to kUnitElems elements.
// Column partial sums of the units of a panel are combined up a static
// kTreeFan-ary tree, in fixed order, by the block that completes a node's
// last child; the block that completes a tensor's last panel updates R, C
// and the partial sums of R in the same launch.
constexpr int kUnitRows = kWarps;        // 8
constexpr int64_t kUnitElems = 4096;
constexpr int kTreeFan = 16;

enum UnitKind : int32_t { kUnitMatrix = 0, kUnitVector = 1, kUnitFactorsOnly = 2 };

struct UnitDev {
    int32_t kind;
    int32_t tensor;
    int32_t panel;        // matrix units
    int32_t parent;       // matrix units: tree node that combines this unit's partial
    int64_t begin;        // first row (matrix) or element (vector)
    int64_t end;
    int64_t leaf_off;     // matrix units: float offset of this unit's column partial
};

struct NodeDev {
    int32_t nchildren;
    int32_t parent;       // -1: root of its panel
    int32_t panel;
    int32_t pad_;
    int64_t first_child_off;  // children's partials are contiguous, PanelTreeDev::slot floats apart
    int64_t off;              // this node's partial
};

struct PanelTreeDev {
    int32_t slot;         // floats between consecutive partials of this panel (width rounded up to 32)
    int32_t pad_;
    int64_t root_off;     // partial of the panel's root node (column sums of the whole panel)
};

}  // namespace rikfad
