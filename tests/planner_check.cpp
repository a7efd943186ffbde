// Host-side check of the in-order schedule built by build_sweep: every unit,
// tree node and partial offset is in range, every node gets exactly its
// declared number of children, every panel has one root, and the units
// cover every row of every panel and every element of every vector exactly
// once.  Compiled with g++ against the planner source by
// tests/test_planner_sweep.py; prints "OK" or the first violation.
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "rikfad_planner.hpp"

using namespace rikfad;

static int fail(const char *what, long long a, long long b)
{
    std::printf("FAIL %s (%lld, %lld)\n", what, a, b);
    return 1;
}

static int check(const std::vector<rikfad_shape> &shapes)
{
    Plan p;
    std::string err = build_plan(shapes.data(), (int)shapes.size(), 2, 304, p);
    if (!err.empty()) {
        std::printf("FAIL build_plan: %s\n", err.c_str());
        return 1;
    }
    build_sweep(shapes.data(), (int)shapes.size(), p);
    const int64_t P = p.partial_floats;
    std::vector<int> children(p.nodes.size(), 0);
    std::vector<std::vector<int>> rows_seen(p.panels.size());
    for (size_t k = 0; k < p.panels.size(); ++k)
        rows_seen[k].assign(p.tensors[p.panels[k].tensor].rows, 0);
    std::vector<std::vector<int>> elems_seen(shapes.size());
    for (size_t t = 0; t < shapes.size(); ++t)
        if (shapes[t].cols == 0)
            elems_seen[t].assign(shapes[t].rows, 0);
    std::vector<int> factor_only(shapes.size(), 0);
    bool vectors_started = false;
    for (size_t u = 0; u < p.units.size(); ++u) {
        const UnitDev &un = p.units[u];
        if (un.tensor < 0 || un.tensor >= (int)shapes.size())
            return fail("unit tensor", (long long)u, un.tensor);
        const TensorDev &td = p.tensors[un.tensor];
        if (un.kind == kUnitVector) {
            vectors_started = true;
            if (td.cols != 0 || un.begin < 0 || un.end > td.rows || un.begin >= un.end)
                return fail("vector unit range", un.begin, un.end);
            if (un.begin % 8)
                return fail("vector unit alignment", (long long)u, un.begin);
            for (int64_t e = un.begin; e < un.end; ++e)
                elems_seen[un.tensor][e]++;
            continue;
        }
        if (vectors_started)
            return fail("matrix unit after a vector unit", (long long)u, 0);
        if (un.kind == kUnitFactorsOnly) {
            if (td.rows != 0 || td.cols == 0)
                return fail("factor-only unit on a non-empty matrix", un.tensor, td.rows);
            factor_only[un.tensor]++;
            continue;
        }
        if (un.kind != kUnitMatrix)
            return fail("unit kind", (long long)u, un.kind);
        if (un.panel < td.panel0 || un.panel >= td.panel0 + td.npanels)
            return fail("unit panel", (long long)u, un.panel);
        if (un.begin < 0 || un.end > td.rows || un.begin >= un.end || un.end - un.begin > kUnitRows)
            return fail("unit rows", un.begin, un.end);
        const PanelDev &pd = p.panels[un.panel];
        const PanelTreeDev &tr = p.trees[un.panel];
        if (tr.slot < pd.width || tr.slot % 32)
            return fail("slot", tr.slot, pd.width);
        if (un.leaf_off < 0 || un.leaf_off + tr.slot > P || un.leaf_off % 32)
            return fail("leaf offset", un.leaf_off, P);
        if (un.parent < 0 || un.parent >= (int)p.nodes.size())
            return fail("unit parent", (long long)u, un.parent);
        const NodeDev &nd = p.nodes[un.parent];
        if (nd.panel != un.panel)
            return fail("parent panel", nd.panel, un.panel);
        const int64_t idx = (un.leaf_off - nd.first_child_off) / tr.slot;
        if ((un.leaf_off - nd.first_child_off) % tr.slot || idx < 0 || idx >= nd.nchildren)
            return fail("leaf not among its parent's children", un.leaf_off, nd.first_child_off);
        children[un.parent]++;
        for (int64_t r = un.begin; r < un.end; ++r)
            rows_seen[un.panel][r]++;
    }
    std::vector<int> roots(p.panels.size(), 0);
    for (size_t i = 0; i < p.nodes.size(); ++i) {
        const NodeDev &nd = p.nodes[i];
        const PanelTreeDev &tr = p.trees[nd.panel];
        if (nd.nchildren < 1 || nd.nchildren > kTreeFan)
            return fail("node fan-in", (long long)i, nd.nchildren);
        if (nd.first_child_off < 0 || nd.first_child_off + (int64_t)nd.nchildren * tr.slot > P)
            return fail("node children range", nd.first_child_off, P);
        if (nd.off < 0 || nd.off + tr.slot > P || nd.off % 32)
            return fail("node offset", nd.off, P);
        if (nd.off >= nd.first_child_off && nd.off < nd.first_child_off + (int64_t)nd.nchildren * tr.slot)
            return fail("node overlaps its children", nd.off, nd.first_child_off);
        if (nd.parent < 0) {
            roots[nd.panel]++;
            if (tr.root_off != nd.off)
                return fail("root offset", tr.root_off, nd.off);
        } else {
            if (nd.parent >= (int)p.nodes.size() || p.nodes[nd.parent].panel != nd.panel)
                return fail("node parent", (long long)i, nd.parent);
            const NodeDev &pa = p.nodes[nd.parent];
            const int64_t idx = (nd.off - pa.first_child_off) / tr.slot;
            if ((nd.off - pa.first_child_off) % tr.slot || idx < 0 || idx >= pa.nchildren)
                return fail("node not among its parent's children", nd.off, pa.first_child_off);
            children[nd.parent]++;
        }
    }
    for (size_t i = 0; i < p.nodes.size(); ++i)
        if (children[i] != p.nodes[i].nchildren)
            return fail("node child count", (long long)i, children[i]);
    for (size_t k = 0; k < p.panels.size(); ++k) {
        const int64_t m = p.tensors[p.panels[k].tensor].rows;
        if (m > 0 && roots[k] != 1)
            return fail("roots per panel", (long long)k, roots[k]);
        for (int64_t r = 0; r < m; ++r)
            if (rows_seen[k][r] != 1)
                return fail("row coverage", (long long)k, r);
    }
    for (size_t t = 0; t < shapes.size(); ++t) {
        if (shapes[t].cols == 0) {
            for (int64_t e = 0; e < shapes[t].rows; ++e)
                if (elems_seen[t][e] != 1)
                    return fail("element coverage", (long long)t, e);
        } else if (shapes[t].rows == 0 && factor_only[t] != 1) {
            return fail("empty matrix needs one factor-only unit", (long long)t, factor_only[t]);
        }
    }
    return 0;
}

int main()
{
    std::vector<std::vector<rikfad_shape>> cases;
    // GPT2-S-like list (q/k/v separate), in module order
    std::vector<rikfad_shape> g;
    g.push_back({50257, 768});
    g.push_back({1024, 768});
    for (int b = 0; b < 12; ++b) {
        g.push_back({768, 0});
        g.push_back({768, 0});
        for (int q = 0; q < 4; ++q) {
            g.push_back({768, 768});
            g.push_back({768, 0});
        }
        g.push_back({768, 0});
        g.push_back({768, 0});
        g.push_back({3072, 768});
        g.push_back({3072, 0});
        g.push_back({768, 3072});
        g.push_back({768, 0});
    }
    g.push_back({768, 0});
    g.push_back({768, 0});
    cases.push_back(g);
    cases.push_back({{1, 1}, {1, 7}, {3, 5}, {257, 129}, {0, 4}, {5, 0}, {0, 0}, {13, 0}, {9, 2048},
                     {2, 3000}, {4096, 8}, {100, 1032}, {4097, 0}, {8, 1040}, {1025, 1}});
    cases.push_back({{50304, 4096}});
    cases.push_back({{4096, 14336}});
    cases.push_back({{65536, 1024}, {300000, 0}});
    cases.push_back({});
    for (size_t i = 0; i < cases.size(); ++i) {
        if (check(cases[i])) {
            std::printf("case %zu\n", i);
            return 1;
        }
    }
    std::printf("OK\n");
    return 0;
}
