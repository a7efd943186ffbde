// rikfad_planner.cpp -- host-side work plan of the fused R-iKFAD step.
#include "rikfad_planner.hpp"

#include <algorithm>
#include <cstdint>
#include <cstdio>
#include <limits>

namespace rikfad {

namespace {

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
int64_t round_up(int64_t a, int64_t b) { return ceil_div(a, b) * b; }

struct Unit {
    int32_t kind;
    int32_t tensor;
    int32_t panel;
    int64_t len;    // rows or elements
    int64_t cost;   // cost per row or element: its bytes, plus kRowCost for a matrix row
    int64_t gran;   // cut granularity
    int64_t bytes;  // compulsory bytes per row or element
};

}  // namespace

std::string check_shapes(const rikfad_shape *shapes, int ntensors)
{
    if (ntensors < 0)
        return "ntensors is negative";
    if (ntensors > 0 && shapes == nullptr)
        return "shapes is NULL";
    const int64_t kMaxCols = std::numeric_limits<int32_t>::max() / 2;
    for (int t = 0; t < ntensors; ++t) {
        const int64_t m = shapes[t].rows, n = shapes[t].cols;
        char buf[160];
        if (m < 0 || n < 0) {
            snprintf(buf, sizeof buf, "tensor %d: negative shape (%lld, %lld)", t, (long long)m,
                     (long long)n);
            return buf;
        }
        if (n > kMaxCols) {
            snprintf(buf, sizeof buf, "tensor %d: cols %lld exceeds %lld", t, (long long)n,
                     (long long)kMaxCols);
            return buf;
        }
        if (n > 0 && m > (std::numeric_limits<int64_t>::max() / 64) / n) {
            snprintf(buf, sizeof buf, "tensor %d: rows x cols overflows", t);
            return buf;
        }
    }
    return "";
}

std::string build_plan(const rikfad_shape *shapes, int ntensors, int grad_bytes, int max_blocks,
                       Plan &plan, bool full_matrices)
{
    std::string err = check_shapes(shapes, ntensors);
    if (!err.empty())
        return err;
    if (grad_bytes != 2 && grad_bytes != 4)
        return "gradient element size must be 2 or 4 bytes";
    if (max_blocks < 1)
        return "block budget must be >= 1";
    Plan p;
    std::vector<Unit> units;

    // Per-tensor layout: factor storage, column panels, row partials.
    int64_t fac = 0, rowpart = 0;
    int64_t spart = 0;
    for (int t = 0; t < ntensors; ++t) {
        TensorDev td{};
        td.rows = shapes[t].rows;
        td.cols = shapes[t].cols;
        td.fac_off = fac;
        td.panel0 = -1;
        if (td.cols == 0) {
            td.vec = 1;
            fac += round_up(td.rows, 8);
            if (td.rows > 0)
                units.push_back({kElements, t, -1, td.rows, vector_elem_bytes(grad_bytes),
                                 kElemGranule, vector_elem_bytes(grad_bytes)});
        } else {
            td.vec = (td.cols % 8 == 0) ? 1 : 0;
            fac += round_up(td.rows + td.cols, 8);
            if (full_matrices) {
                td.full = 1;
                td.xi_off = fac;
                fac += round_up(td.rows * td.cols, 8);
            }
            // Panels of at most kPanelMax columns.  On the 8-wide path a warp
            // moves one 256-column chunk per round trip, so every panel but
            // the last is a whole number of chunks: the matrix then takes the
            // fewest chunks, ceil(cols / 256) per row (two 800-wide panels of
            // a 1600-wide matrix would take 8, 1024 + 576 take 7).
            int64_t np = ceil_div(td.cols, kPanelMax);
            int64_t w = ceil_div(td.cols, np);
            if (td.vec)
                w = std::min<int64_t>(kPanelMax, round_up(w, kChunk));
            np = ceil_div(td.cols, w);
            std::vector<int64_t> widths;
            for (int64_t k = 0; k < np; ++k)
                widths.push_back(std::min<int64_t>(w, td.cols - k * w));
            // A last panel wider than kPanelMax / 2 whose tail past whole
            // chunks is at most half a chunk gives that tail a panel of its
            // own, which the kernel runs with several rows per warp (1600 =
            // 1024 + 512 + 64 takes 6.25 round trips per row, 1024 + 576
            // takes 7).
            if (td.vec) {
                const int64_t r = widths.back(), tail = r % kChunk;
                if (r > kPanelMax / 2 && tail > 0 && tail <= kChunk / 2) {
                    widths.back() = r - tail;
                    widths.push_back(tail);
                }
            }
            np = (int64_t)widths.size();
            td.npanels = (int32_t)np;
            td.panel0 = (int32_t)p.panels.size();
            int64_t col0 = 0;
            for (int64_t k = 0; k < np; ++k) {
                PanelDev pd{};
                pd.tensor = t;
                pd.col0 = (int32_t)col0;
                pd.width = (int32_t)widths[k];
                col0 += widths[k];
                pd.nch = (int32_t)ceil_div(pd.width, kChunk);
                pd.slot_begin = pd.slot_end = 0;
                if (td.rows > 0) {
                    const int64_t b = pd.width * (full_matrices ? vector_elem_bytes(grad_bytes)
                                                                : matrix_elem_bytes(grad_bytes));
                    units.push_back({kMatrixRows, t, (int32_t)p.panels.size(), td.rows, b + kRowCost, 1, b});
                }
                p.panels.push_back(pd);
            }
            td.rowpart_off = rowpart;
            rowpart += td.rows * np;
            td.spart_off = (int32_t)spart;
            td.spart_cnt = (int32_t)ceil_div(td.rows, kFinThreads);
            spart += td.spart_cnt;
        }
        p.tensors.push_back(td);
    }
    if (spart > std::numeric_limits<int32_t>::max())
        return "too many rows";
    p.fac_floats = fac;
    p.rowpart_floats = rowpart;
    p.spart_floats = (int32_t)spart;

    int64_t total = 0, total_bytes = 0;
    for (const Unit &u : units) {
        total += u.len * u.cost;
        total_bytes += u.len * u.bytes;
    }
    p.total_bytes = total_bytes;

    // Cut the unit sequence into nblocks shares of nearly equal cost.
    p.block_piece.push_back(0);
    if (total > 0) {
        const int64_t G = std::min<int64_t>(max_blocks, std::max<int64_t>(1, ceil_div(total, kMinBlockBytes)));
        p.nblocks = (int)G;
        int64_t block = 0, acc = 0;
        auto boundary = [&](int64_t b) { return (int64_t)((__int128)total * (b + 1) / G); };
        int64_t bound = boundary(0);
        int64_t colpart = 0;
        for (const Unit &u : units) {
            int64_t pos = 0;
            while (pos < u.len) {
                int64_t take;
                if (block == G - 1) {
                    take = u.len - pos;
                } else {
                    const int64_t room = bound - acc;
                    take = room > 0 ? ceil_div(room, u.cost) : 1;
                    take = round_up(take, u.gran);
                    take = std::min(take, u.len - pos);
                }
                PieceDev pc{};
                pc.kind = u.kind;
                pc.tensor = u.tensor;
                pc.panel = u.panel;
                pc.begin = pos;
                pc.end = pos + take;
                pc.slot = -1;
                pc.colpart_off = 0;
                if (u.kind == kMatrixRows) {
                    PanelDev &pd = p.panels[u.panel];
                    const int32_t slot = (int32_t)p.slot_off.size();
                    if (pd.slot_end == pd.slot_begin)
                        pd.slot_begin = slot;
                    pd.slot_end = slot + 1;
                    pc.slot = slot;
                    pc.colpart_off = colpart;
                    p.slot_off.push_back(colpart);
                    colpart += pd.width;
                }
                p.pieces.push_back(pc);
                acc += take * u.cost;
                pos += take;
                while (acc >= bound && block < G - 1) {
                    ++block;
                    p.block_piece.push_back((int32_t)p.pieces.size());
                    bound = boundary(block);
                }
            }
        }
        while ((int64_t)p.block_piece.size() < G + 1)
            p.block_piece.push_back((int32_t)p.pieces.size());
        p.colpart_floats = colpart;
    }

    // The finalise kernel addresses a panel's slots from its first one: they
    // must be consecutive and one panel width apart in colpart.
    for (const PanelDev &pd : p.panels)
        for (int32_t s = pd.slot_begin; s < pd.slot_end; ++s)
            if (p.slot_off[s] != p.slot_off[pd.slot_begin] + (int64_t)(s - pd.slot_begin) * pd.width)
                return "internal: slots of a panel are not contiguous";

    // Finalise work: R in chunks of kFinThreads rows (each also yields one
    // partial sum of R), C in chunks of kFinColChunk columns of each panel.
    for (int t = 0; t < ntensors; ++t) {
        const TensorDev &td = p.tensors[t];
        if (td.cols == 0)
            continue;
        for (int32_t c = 0; c < td.spart_cnt; ++c) {
            FinItemDev it{};
            it.kind = kFinRows;
            it.tensor = t;
            it.panel = -1;
            it.chunk = c;
            it.begin = (int64_t)c * kFinThreads;
            it.end = std::min<int64_t>(td.rows, it.begin + kFinThreads);
            p.fin_items.push_back(it);
        }
        for (int32_t k = 0; k < td.npanels; ++k) {
            const PanelDev &pd = p.panels[td.panel0 + k];
            // Many slots: 32-column items whose 8 warps split the slots; few
            // slots: one thread per column, 256 columns per item.
            const bool split = pd.slot_end - pd.slot_begin > kFinSplitSlots;
            const int64_t step = split ? kFinColChunk : kFinThreads;
            for (int64_t c0 = 0; c0 < pd.width; c0 += step) {
                FinItemDev it{};
                it.kind = kFinCols;
                it.tensor = t;
                it.panel = td.panel0 + k;
                it.chunk = split ? 1 : 0;
                it.begin = c0;
                it.end = std::min<int64_t>(pd.width, c0 + step);
                p.fin_items.push_back(it);
            }
        }
    }
    plan = std::move(p);
    return "";
}

void build_sweep(const rikfad_shape *shapes, int ntensors, Plan &plan)
{
    Plan &p = plan;
    p.units.clear();
    p.nodes.clear();
    p.trees.assign(p.panels.size(), PanelTreeDev{});
    int64_t off = 0;
    for (int t = 0; t < ntensors; ++t) {
        const TensorDev &td = p.tensors[t];
        if (td.cols == 0)
            continue;
        if (td.rows == 0) {
            UnitDev u{};
            u.kind = kUnitFactorsOnly;
            u.tensor = t;
            u.panel = -1;
            u.parent = -1;
            p.units.push_back(u);
            continue;
        }
        const int64_t first_unit = (int64_t)p.units.size();
        const int64_t nrb = ceil_div(td.rows, kUnitRows);
        // Units in memory order: row block major, panel minor.
        for (int64_t rb = 0; rb < nrb; ++rb)
            for (int32_t k = 0; k < td.npanels; ++k) {
                UnitDev u{};
                u.kind = kUnitMatrix;
                u.tensor = t;
                u.panel = td.panel0 + k;
                u.begin = rb * kUnitRows;
                u.end = std::min<int64_t>(td.rows, u.begin + kUnitRows);
                p.units.push_back(u);
            }
        // One tree per panel over its nrb units.
        for (int32_t k = 0; k < td.npanels; ++k) {
            const int32_t panel = td.panel0 + k;
            const int64_t slot = round_up(p.panels[panel].width, 32);
            PanelTreeDev &tr = p.trees[panel];
            tr.slot = (int32_t)slot;
            // leaves: the panel's units, in row order
            const int64_t leaf0 = off;
            for (int64_t rb = 0; rb < nrb; ++rb) {
                UnitDev &u = p.units[first_unit + rb * td.npanels + k];
                u.leaf_off = leaf0 + rb * slot;
            }
            off += nrb * slot;
            // internal levels until one node remains (a single leaf still gets a root)
            int64_t count = nrb, child_off = leaf0;
            std::vector<int32_t> child_ids;      // node ids of the previous level (empty: leaves)
            for (;;) {
                const int64_t nn = ceil_div(count, kTreeFan);
                const int64_t level_off = off;
                std::vector<int32_t> ids;
                for (int64_t j = 0; j < nn; ++j) {
                    NodeDev nd{};
                    nd.nchildren = (int32_t)std::min<int64_t>(kTreeFan, count - j * kTreeFan);
                    nd.parent = -1;
                    nd.panel = panel;
                    nd.first_child_off = child_off + j * kTreeFan * slot;
                    nd.off = level_off + j * slot;
                    const int32_t id = (int32_t)p.nodes.size();
                    p.nodes.push_back(nd);
                    ids.push_back(id);
                    for (int64_t c = j * kTreeFan; c < j * kTreeFan + nd.nchildren; ++c) {
                        if (child_ids.empty())
                            p.units[first_unit + c * td.npanels + k].parent = id;
                        else
                            p.nodes[child_ids[c]].parent = id;
                    }
                }
                off += nn * slot;
                if (nn == 1) {
                    tr.root_off = p.nodes[ids[0]].off;
                    break;
                }
                child_ids = ids;
                child_off = level_off;
                count = nn;
            }
        }
    }
    // vectors last
    for (int t = 0; t < ntensors; ++t) {
        const TensorDev &td = p.tensors[t];
        if (td.cols != 0)
            continue;
        for (int64_t b = 0; b < td.rows; b += kUnitElems) {
            UnitDev u{};
            u.kind = kUnitVector;
            u.tensor = t;
            u.panel = -1;
            u.parent = -1;
            u.begin = b;
            u.end = std::min<int64_t>(td.rows, b + kUnitElems);
            p.units.push_back(u);
        }
    }
    p.partial_floats = off;
    (void)shapes;
}

}  // namespace rikfad
