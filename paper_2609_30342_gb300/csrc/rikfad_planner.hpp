// rikfad_planner.hpp -- host-side construction of the work plan (no CUDA).
#pragma once
#include <string>
#include <vector>

#include "rikfad.h"
#include "rikfad_plan.hpp"

namespace rikfad {

struct Plan {
    std::vector<TensorDev> tensors;
    std::vector<PanelDev> panels;
    std::vector<PieceDev> pieces;
    std::vector<int32_t> block_piece;   // block b owns pieces [block_piece[b], block_piece[b+1])
    std::vector<int64_t> slot_off;      // colpart offset of every slot
    std::vector<FinItemDev> fin_items;
    int64_t fac_floats = 0;             // factors + element-wise friction (padded)
    int64_t rowpart_floats = 0;
    int64_t colpart_floats = 0;
    int32_t spart_floats = 0;
    int nblocks = 0;                    // blocks of the step kernel (0 when there is no work)
    int64_t total_bytes = 0;            // compulsory HBM bytes of one step (planner's cost model)

    // In-order schedule (see rikfad_plan.hpp)
    std::vector<UnitDev> units;
    std::vector<NodeDev> nodes;
    std::vector<PanelTreeDev> trees;    // one per panel
    int64_t partial_floats = 0;         // unit and node partials
};

// Add the in-order schedule (units, reduction trees) to a plan built by
// build_plan.  Matrices keep their order; vectors come last.
void build_sweep(const rikfad_shape *shapes, int ntensors, Plan &plan);

// Validate the shape list; returns "" or an error message.
std::string check_shapes(const rikfad_shape *shapes, int ntensors);

// Build the plan for at most max_blocks blocks.  grad_bytes is 2 or 4.
// Returns "" on success or an error message.
// full_matrices: every matrix keeps element-wise friction (m x n floats)
// and its R, C become shadow factors (full iKFAD with R-iKFAD's factors
// carried alongside).
std::string build_plan(const rikfad_shape *shapes, int ntensors, int grad_bytes, int max_blocks,
                       Plan &plan, bool full_matrices = false);

// Bytes of one step that HBM must move for one element (compulsory traffic):
// matrix element: read grad + X + P, write X + P; vector element: + friction
// read and write.
inline int64_t matrix_elem_bytes(int grad_bytes) { return grad_bytes + 16; }
inline int64_t vector_elem_bytes(int grad_bytes) { return grad_bytes + 24; }

}  // namespace rikfad
