// planner.cu -- choice of every tensor's upper/lower split over a tree of
// binary EinSums (paper Sec. 7 and Sec. 8.1).  Host code only.
//
// * Tuple counts of a decomposition follow Eq. eqn-count from the tensor's
//   statistics T and V (Sec. 7.1).
// * A vertex costs C_join + C_agg, an edge whose producer and consumer split
//   the tensor differently costs C_repart (Sec. 7.2).
// * Alg. 1 visits the vertices in topological order and keeps, for every
//   vertex and every output split, the cheapest ways to produce it; this
//   version keeps the k cheapest, so the runner-up plans come out too.
// * Statistics of intermediate tensors that the caller does not supply are
//   estimated as Alg. 2 prescribes: textbook join and group-by estimates over
//   the fully relational (scalar) form of the program.
//
// Readings: a label takes one class within an EinSum (both inputs and the
// output agree on it); the aggregation estimate multiplies over the output's
// promoted labels; C_krnel is c_flop times the kernel's multiply-adds (two
// flops per combination of the expression's lower labels) and C_add is c_add
// times the elements of an output tile; input tensors are free in any split
// and are read as their consumer wants them; ties keep the first plan found,
// subsets enumerated by increasing bit mask.  The memory constraint of
// Sec. 8.2 is a bound on the bytes of the three tiles one kernel call touches.
//
// ucl_plan_dag is Sec. 8.2's heuristic for programs whose results are used
// more than once.  The DAG is cut into trees at every EinSum result used more
// than once (and at every output): such a result roots its own tree, every
// other EinSum vertex joins its one consumer's tree.  Trees are optimised by
// the same dynamic programme in increasing order of their root, each reading
// the results earlier trees decided as inputs whose split is fixed (another
// split costs C_repart).  A result used twice is not merged into one of its
// consumers' trees: that can make the order between trees cyclic.
#include <algorithm>
#include <cmath>
#include <vector>

#include "internal.cuh"

namespace {

constexpr int kMaxPlanLabels = 12;   // labels of one tensor (2^12 splits)

struct PVertex {
    int left = -1, right = -1;
    std::vector<char> lab;            // labels in order
    std::vector<int64_t> ext;         // extent per label
    int bytes = 2;
    double T = 0;
    std::vector<double> V;            // per label
    int64_t fixed = -1;               // leaves: the split the tensor is stored in, -1 = free
};

struct Entry {
    double cost;
    uint32_t upW;                     // this vertex's output split (for bookkeeping)
    uint32_t upU, upV;                // how it reads its inputs (leaves: unused)
    uint32_t lprod, rprod;            // producer output splits
    int lidx, ridx;                   // entries of the producers' lists
};

int find(const std::vector<char> &lab, char c) {
    for (size_t q = 0; q < lab.size(); ++q)
        if (lab[q] == c) return (int)q;
    return -1;
}

bool has(uint32_t mask, int q) { return q >= 0 && (mask >> q & 1u); }

double tuple_count(const PVertex &x, uint32_t up) {
    double n = 1.0;
    for (size_t q = 0; q < x.lab.size(); ++q)
        if (up >> q & 1u) n *= x.V[q];
    if (n <= 0 || x.T <= 0) return 0.0;
    return n * -std::expm1(-x.T / n);
}

// Tile sizes are products of extents, in double so that no split of large
// labels overflows (exact below 2^53).
double tile_bytes(const PVertex &x, uint32_t up) {
    double tile = 1.0;
    for (size_t q = 0; q < x.lab.size(); ++q)
        if (!(up >> q & 1u)) tile *= (double)x.ext[q];
    return (double)x.bytes * tile;
}

double tuple_bytes(const PVertex &x, uint32_t up, int key_bytes) {
    double tile = 1.0;
    int nk = 0;
    for (size_t q = 0; q < x.lab.size(); ++q) {
        if (up >> q & 1u) ++nk;
        else tile *= (double)x.ext[q];
    }
    return (double)(key_bytes * nk) + (double)x.bytes * tile;
}

struct Ctx {
    std::vector<PVertex> g;
    ucl_cost_model cm;
};

double join_tuples(const PVertex &U, uint32_t upU, const PVertex &Vv, uint32_t upV) {
    double den = 1.0;
    for (size_t q = 0; q < U.lab.size(); ++q) {
        if (!(upU >> q & 1u)) continue;
        const int p = find(Vv.lab, U.lab[q]);
        if (has(upV, p)) den *= std::max(U.V[q], Vv.V[p]);
    }
    return tuple_count(U, upU) * tuple_count(Vv, upV) / den;
}

double vertex_cost(const Ctx &cx, int i, uint32_t upW, uint32_t upU, uint32_t upV) {
    const PVertex &W = cx.g[i], &U = cx.g[W.left], &Vv = cx.g[W.right];
    const ucl_cost_model &cm = cx.cm;
    const double tj = join_tuples(U, upU, Vv, upV);
    // C_join
    const double size = tuple_bytes(U, upU, cm.key_bytes) + tuple_bytes(Vv, upV, cm.key_bytes);
    double flops = 2.0;
    for (size_t q = 0; q < U.lab.size(); ++q)
        if (!(upU >> q & 1u)) flops *= (double)U.ext[q];
    for (size_t q = 0; q < Vv.lab.size(); ++q)
        if (!(upV >> q & 1u) && find(U.lab, Vv.lab[q]) < 0) flops *= (double)Vv.ext[q];
    const double cjoin = tj * (size * cm.xfer + cm.flop * flops + cm.fixed);
    // C_agg
    double p = 1.0;
    for (size_t q = 0; q < W.lab.size(); ++q) {
        if (!(upW >> q & 1u)) continue;
        const int a = find(U.lab, W.lab[q]), b = find(Vv.lab, W.lab[q]);
        if (has(upU, a) && has(upV, b)) p *= std::min(U.V[a], Vv.V[b]);
        else if (has(upU, a)) p *= U.V[a];
        else p *= Vv.V[b];
    }
    const double ta = std::min(0.5 * tj, p);
    double elems = 1.0;
    for (size_t q = 0; q < W.lab.size(); ++q)
        if (!(upW >> q & 1u)) elems *= (double)W.ext[q];
    const double wsize = tuple_bytes(W, upW, cm.key_bytes);
    const double cagg = (tj - ta) * (wsize * cm.xfer + cm.add * elems + cm.fixed);
    return cjoin + cagg;
}

double repart_cost(const Ctx &cx, int i, uint32_t up_in, uint32_t up_out) {
    if (up_in == up_out) return 0.0;
    const PVertex &x = cx.g[i];
    const uint32_t un = up_in | up_out;
    const double t = 2.0 * tuple_count(x, un) - tuple_count(x, up_in) - tuple_count(x, up_out);
    return t * (tuple_bytes(x, un, cx.cm.key_bytes) * cx.cm.xfer + cx.cm.fixed);
}

// X's split agrees with W's on every label they share.
bool consistent(const PVertex &X, uint32_t upX, const PVertex &W, uint32_t upW) {
    for (size_t q = 0; q < X.lab.size(); ++q) {
        const int p = find(W.lab, X.lab[q]);
        if (p >= 0 && (bool)(upX >> q & 1u) != (bool)(upW >> p & 1u)) return false;
    }
    return true;
}

// Alg. 2: statistics of W = sum U x V from its inputs'.
void estimate_stats(PVertex &W, const PVertex &U, const PVertex &Vv) {
    double den = 1.0;
    for (size_t q = 0; q < U.lab.size(); ++q) {
        const int p = find(Vv.lab, U.lab[q]);
        if (p >= 0) den *= std::max(U.V[q], Vv.V[p]);
    }
    const double tj = U.T * Vv.T / den;
    W.V.assign(W.lab.size(), 0.0);
    double prod = 1.0;
    for (size_t q = 0; q < W.lab.size(); ++q) {
        const int a = find(U.lab, W.lab[q]), b = find(Vv.lab, W.lab[q]);
        if (a >= 0 && b >= 0) W.V[q] = std::min(U.V[a], Vv.V[b]);
        else if (a >= 0) W.V[q] = U.V[a];
        else W.V[q] = Vv.V[b];
        prod *= W.V[q];
    }
    W.T = std::min(tj, prod);
    for (double &v : W.V) v = std::min(v, W.T);
}

bool by_cost(const Entry &a, const Entry &b) { return a.cost < b.cost; }

using Table = std::vector<std::vector<std::vector<Entry>>>;   // [vertex][output split] -> k cheapest

// Alg. 1 with k-best lists over the tree cx.g (topological order, last vertex
// the root, every vertex but the root consumed once).  Leaves cost nothing in
// any split, or a repartition from the split they are stored in.
void run_dp(const Ctx &cx, int k, Table &C) {
    const int n = (int)cx.g.size();
    C.assign(n, {});
    for (int i = 0; i < n; ++i) {
        const PVertex &W = cx.g[i];
        const uint32_t nW = 1u << W.lab.size();
        C[i].resize(nW);
        if (W.left < 0) {
            for (uint32_t s = 0; s < nW; ++s) C[i][s].push_back(Entry{0.0, s, 0, 0, 0, 0, -1, -1});
            continue;
        }
        const PVertex &U = cx.g[W.left], &Vv = cx.g[W.right];
        const uint32_t nU = 1u << U.lab.size(), nV = 1u << Vv.lab.size();
        std::vector<Entry> sideU, sideV, cands;
        auto side = [&](int child, uint32_t up_in, std::vector<Entry> &opts) {
            opts.clear();
            const PVertex &x = cx.g[child];
            if (x.left < 0) {
                const double c0 = x.fixed >= 0 ? repart_cost(cx, child, (uint32_t)x.fixed, up_in) : 0.0;
                opts.push_back(Entry{c0, up_in, 0, 0, up_in, 0, 0, -1});
                return;
            }
            for (uint32_t p = 0; p < C[child].size(); ++p) {
                const double r = repart_cost(cx, child, p, up_in);
                for (size_t e = 0; e < C[child][p].size(); ++e)
                    opts.push_back(Entry{C[child][p][e].cost + r, up_in, 0, 0, p, 0, (int)e, -1});
            }
            std::stable_sort(opts.begin(), opts.end(), by_cost);
            if ((int)opts.size() > k) opts.resize(k);
        };
        for (uint32_t upW = 0; upW < nW; ++upW) {
            cands.clear();
            for (uint32_t upU = 0; upU < nU; ++upU) {
                if (!consistent(U, upU, W, upW)) continue;
                for (uint32_t upV = 0; upV < nV; ++upV) {
                    if (!consistent(Vv, upV, W, upW) || !consistent(Vv, upV, U, upU)) continue;
                    if (cx.cm.max_call_bytes > 0 &&
                        tile_bytes(U, upU) + tile_bytes(Vv, upV) + tile_bytes(W, upW) > cx.cm.max_call_bytes)
                        continue;
                    const double here = vertex_cost(cx, i, upW, upU, upV);
                    side(W.left, upU, sideU);
                    side(W.right, upV, sideV);
                    for (const Entry &a : sideU)
                        for (const Entry &b : sideV)
                            cands.push_back(Entry{here + a.cost + b.cost, upW, upU, upV, a.lprod, b.lprod, a.lidx,
                                                  b.lidx});
                }
            }
            std::stable_sort(cands.begin(), cands.end(), by_cost);
            if ((int)cands.size() > k) cands.resize(k);
            C[i][upW] = cands;
        }
    }
}

// The k cheapest entries of the root, cheapest first.
std::vector<Entry> root_best(const Table &C, int k) {
    std::vector<Entry> best;
    const int root = (int)C.size() - 1;
    for (uint32_t s = 0; s < C[root].size(); ++s)
        for (const Entry &e : C[root][s]) best.push_back(e);
    std::stable_sort(best.begin(), best.end(), by_cost);
    if ((int)best.size() > k) best.resize(k);
    return best;
}

// Walk one plan down from the root: every vertex's output split (a leaf's:
// the split its consumer reads) and every EinSum's read splits.
void unroll(const Ctx &cx, const Table &C, const Entry &top, uint32_t *up, uint32_t (*in_up)[2]) {
    const int root = (int)cx.g.size() - 1;
    std::vector<std::pair<int, Entry>> stack{{root, top}};
    while (!stack.empty()) {
        const int i = stack.back().first;
        const Entry e = stack.back().second;
        stack.pop_back();
        up[i] = e.upW;
        const PVertex &W = cx.g[i];
        if (W.left < 0) continue;
        in_up[i][0] = e.upU;
        in_up[i][1] = e.upV;
        if (cx.g[W.left].left < 0) up[W.left] = e.upU;
        else stack.push_back({W.left, C[W.left][e.lprod][e.lidx]});
        if (cx.g[W.right].left < 0) up[W.right] = e.upV;
        else stack.push_back({W.right, C[W.right][e.rprod][e.ridx]});
    }
}

// Labels, extents and statistics of every vertex.  tree: every tensor but the
// last consumed exactly once, by two distinct producers; else any DAG in
// topological order.
ucl_status parse(int n_vertices, const ucl_plan_vertex *vertices, const char *label_names,
                 const int64_t *label_bounds, int n_labels, bool tree, Ctx &cx) {
    cx.g.assign(n_vertices, PVertex{});
    std::vector<int> consumed(n_vertices, 0);
    for (int i = 0; i < n_vertices; ++i) {
        const ucl_plan_vertex &v = vertices[i];
        PVertex &x = cx.g[i];
        if (!v.labels) return UCL_ERR_ARG;
        for (const char *c = v.labels; *c; ++c) {
            if (find(x.lab, *c) >= 0) return UCL_ERR_SPEC;
            int pos = -1;
            for (int l = 0; l < n_labels; ++l)
                if (label_names[l] == *c) pos = l;
            if (pos < 0 || label_bounds[pos] < 1) return UCL_ERR_SHAPE;
            x.lab.push_back(*c);
            x.ext.push_back(label_bounds[pos]);
            if ((int)x.lab.size() > kMaxPlanLabels) return UCL_ERR_UNSUPPORTED;
        }
        if (v.dtype_bytes < 1) return UCL_ERR_ARG;
        x.bytes = v.dtype_bytes;
        x.left = v.left;
        x.right = v.right;
        if ((v.left < 0) != (v.right < 0)) return UCL_ERR_ARG;
        if (v.left < 0) {
            if (!v.distinct || !(v.nnz >= 0)) return UCL_ERR_ARG;
            x.T = v.nnz;
            x.V.assign(v.distinct, v.distinct + x.lab.size());
            continue;
        }
        if (v.left >= i || v.right >= i) return UCL_ERR_ARG;
        if (tree && (v.left == v.right || consumed[v.left]++ || consumed[v.right]++)) return UCL_ERR_ARG;
        const PVertex &U = cx.g[v.left], &Vv = cx.g[v.right];
        for (char c : x.lab)
            if (find(U.lab, c) < 0 && find(Vv.lab, c) < 0) return UCL_ERR_SPEC;
        if (v.distinct && v.nnz >= 0) {
            x.T = v.nnz;
            x.V.assign(v.distinct, v.distinct + x.lab.size());
        } else {
            estimate_stats(x, U, Vv);
        }
    }
    return UCL_OK;
}

}  // namespace

extern "C" {

ucl_status ucl_plan(int n_vertices, const ucl_plan_vertex *vertices, const char *label_names,
                    const int64_t *label_bounds, int n_labels, const ucl_cost_model *cost_model, int k,
                    ucl_plan_choice *out, int *n_out) {
    if (n_out) *n_out = 0;
    if (n_vertices < 1 || n_vertices > UCL_PLAN_MAX_VERTICES || !vertices || !label_names || !label_bounds ||
        n_labels < 0 || !cost_model || k < 1 || !out || !n_out)
        return UCL_ERR_ARG;
    Ctx cx;
    cx.cm = *cost_model;
    const ucl_status st = parse(n_vertices, vertices, label_names, label_bounds, n_labels, true, cx);
    if (st) return st;
    Table C;
    run_dp(cx, k, C);
    const std::vector<Entry> best = root_best(C, k);
    for (size_t b = 0; b < best.size(); ++b) {
        ucl_plan_choice &pc = out[b];
        memset(&pc, 0, sizeof(pc));
        pc.cost = best[b].cost;
        unroll(cx, C, best[b], pc.up, pc.in_up);
    }
    *n_out = (int)best.size();
    return UCL_OK;
}

ucl_status ucl_plan_dag(int n_vertices, const ucl_plan_vertex *vertices, const char *label_names,
                        const int64_t *label_bounds, int n_labels, const ucl_cost_model *cost_model,
                        ucl_plan_choice *out, int *tree_root) {
    if (n_vertices < 1 || n_vertices > UCL_PLAN_MAX_VERTICES || !vertices || !label_names || !label_bounds ||
        n_labels < 0 || !cost_model || !out)
        return UCL_ERR_ARG;
    Ctx cx;
    cx.cm = *cost_model;
    ucl_status st = parse(n_vertices, vertices, label_names, label_bounds, n_labels, false, cx);
    if (st) return st;
    // consuming edges of every vertex, and the tree of every EinSum vertex
    std::vector<std::vector<int>> uses(n_vertices);
    for (int i = 0; i < n_vertices; ++i)
        if (cx.g[i].left >= 0) {
            uses[cx.g[i].left].push_back(i);
            uses[cx.g[i].right].push_back(i);
        }
    std::vector<int> tree(n_vertices, -1);
    for (int i = n_vertices - 1; i >= 0; --i)
        if (cx.g[i].left >= 0) tree[i] = uses[i].size() == 1 ? tree[uses[i][0]] : i;
    ucl_plan_choice res;
    memset(&res, 0, sizeof(res));
    std::vector<int> where(n_vertices, -1);
    for (int r = 0; r < n_vertices; ++r) {
        if (tree[r] != r) continue;
        // the tree rooted at r: its EinSum vertices in order, and one leaf per
        // edge that enters it (an input, or a result an earlier tree decided)
        Ctx sub;
        sub.cm = cx.cm;
        std::vector<int> members;
        auto leaf = [&](int p) {
            PVertex x = cx.g[p];
            x.fixed = x.left >= 0 ? (int64_t)res.up[p] : -1;
            x.left = x.right = -1;
            sub.g.push_back(x);
            return (int)sub.g.size() - 1;
        };
        for (int i = 0; i <= r; ++i) {
            if (tree[i] != r) continue;
            PVertex x = cx.g[i];
            const int a = tree[x.left] == r ? where[x.left] : leaf(x.left);
            const int b = tree[x.right] == r ? where[x.right] : leaf(x.right);
            x.left = a;
            x.right = b;
            sub.g.push_back(x);
            where[i] = (int)sub.g.size() - 1;
            members.push_back(i);
        }
        Table C;
        run_dp(sub, 1, C);
        const std::vector<Entry> best = root_best(C, 1);
        if (best.empty()) return UCL_ERR_UNSUPPORTED;   // no split within the memory bound
        std::vector<uint32_t> up(sub.g.size(), 0), in_flat(2 * sub.g.size(), 0);
        unroll(sub, C, best[0], up.data(), reinterpret_cast<uint32_t(*)[2]>(in_flat.data()));
        res.cost += best[0].cost;
        for (int i : members) {
            res.up[i] = up[where[i]];
            res.in_up[i][0] = in_flat[2 * where[i]];
            res.in_up[i][1] = in_flat[2 * where[i] + 1];
        }
    }
    // an input's entry: the split its first consumer (lowest index, left
    // operand first) reads
    for (int i = 0; i < n_vertices; ++i) {
        if (cx.g[i].left >= 0 || uses[i].empty()) continue;
        const int c = uses[i][0];
        res.up[i] = cx.g[c].left == i ? res.in_up[c][0] : res.in_up[c][1];
    }
    *out = res;
    if (tree_root)
        for (int i = 0; i < n_vertices; ++i) tree_root[i] = tree[i];
    return UCL_OK;
}

}  // extern "C"
