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
constexpr int kFinColChunk = 32;     // columns per finalise column item
constexpr int kElemGranule = 8;      // element pieces start on multiples of 8 elements
constexpr int64_t kMinBlockBytes = 64 * 1024;   // smallest share worth a block

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
    int32_t pad_;
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
    int32_t chunk;        // kFinRows: index of the partial sum of R within the tensor
    int64_t begin;        // kFinRows: rows; kFinCols: columns relative to the panel
    int64_t end;
};

}  // namespace rikfad
