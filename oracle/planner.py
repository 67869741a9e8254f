"""Oracle for the sparsity-aware decomposition planner (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke`` and the CPU leg of ``bench.py`` may
use this module; it shares nothing with the executor or its planner.

It restates, in plain Python and in the paper's order:

* the statistics of Sec. 7.1: T(U), the number of non-zero entries of a
  tensor, and V(l, U), the number of slices along label l holding a non-zero;
* the tuple-count estimate of Eq. eqn-count for a decomposition with
  promoted labels up(U);
* the join, aggregation and repartition costs of Sec. 7.2;
* GetStats (Alg. 2): statistics of an intermediate tensor from those of its
  inputs by textbook relational estimates over purely relational (scalar)
  versions of the tensors;
* ComputeMinCostForTree (Alg. 1): the dynamic programme over a tree of binary
  EinSums, keeping for every vertex and output decomposition the cheapest way
  to produce it;
* the heuristic of Sec. 8.2 for programs whose results are consumed more than
  once: split the DAG into trees in which no result is used twice, optimise
  them one after another with Alg. 1, each treating the decompositions already
  chosen as fixed;
* an exhaustive enumeration of every plan, which the tests use to pin the
  dynamic programme (and its k-best extension) independently of its recursion.

Readings where the paper is silent or inconsistent:

* P1 A label shared by both inputs takes one class in both (upper in both or
  lower in both): a label has one case in a UCL expression, so ↑U and ↑V
  agree on ℓU ∩ ℓV, besides agreeing with ↑W on the labels they share with it.
* P2 The aggregation estimate multiplies the distinct counts over the output's
  promoted labels ↑W (the grouping labels its text describes); the printed
  subscript names the aggregated labels instead.
* P3 C_krnel = c_flop × the multiply-adds of one kernel call (2 flops for
  every combination of the expression's lower labels); C_add = c_add × the
  elements of one output tile.
* P4 Input tensors cost nothing in any decomposition (Alg. 1's initialisation)
  and are never repartitioned: they are materialised as their consumer reads
  them.  The k-best lists therefore never contain a plan that repartitions an
  input, which would only add cost to another plan.
* P5 GetStats: the join of scalar relations has T(U)·T(V) / Π max(V_U, V_V)
  tuples over the shared labels; a label's distinct count after the join is
  the smaller of its counts on the two sides (or its only side's); the
  aggregation onto ℓW keeps min(T_join, Π V) tuples, and no distinct count
  exceeds the tuple count.
* P6 Ties between plans of equal cost keep the first found, enumerating
  subsets of a label list by increasing bit mask (bit q = the q-th label).
* P7 The memory constraint of Sec. 8.2 bounds what one kernel call touches:
  with a positive ``max_call_bytes``, an EinSum may only read and write tiles
  whose bytes (U's tile + V's tile + W's tile, at each tensor's element
  size) total at most that; choices above it are left out of the search.
* P8 The trees of Sec. 8.2's multi-use heuristic are cut at every EinSum
  result used more than once (and at every result no EinSum uses, an
  output): such a result roots its own tree, and every other EinSum vertex
  joins the tree of its one consumer.  Trees are optimised in increasing
  order of their root, so every result a tree reads from another tree is
  already decided.  Its consumers read it as an input whose decomposition is
  fixed: reading it in another split costs C_repart (an input tensor of the
  program stays free in any split, P4).  The paper asks for maximal trees; a
  result used twice could also join one of its consumers' trees, but that
  choice can make the order between trees cyclic (two trees each reading a
  result the other decides), so it is not taken.  A result that one EinSum
  reads as both operands counts as used twice.
"""
from __future__ import annotations

import itertools
import math
from dataclasses import dataclass, field

import numpy as np


@dataclass
class CostModel:
    """Per-unit costs of Sec. 7.2 (seconds per byte, flop, added element and tuple)."""

    xfer: float = 1.0
    flop: float = 0.0
    add: float = 0.0
    fixed: float = 0.0
    key_bytes: int = 4
    max_call_bytes: float = 0.0     # reading P7; 0: no bound


@dataclass
class Stats:
    T: float                       # non-zero entries, T(U)
    V: dict = field(default_factory=dict)   # label -> V(l, U)


@dataclass
class Vertex:
    """One vertex of an EinSum tree: an input tensor (left = right = None) or a
    binary EinSum W = Σ U × V over the labels it does not keep."""

    labels: str
    dtype_bytes: int = 2
    left: int | None = None
    right: int | None = None
    stats: Stats | None = None     # inputs: required; EinSums: estimated when None
    fixed_up: tuple | None = None  # inputs only: the split the tensor is already stored in
                                   # (reading P8); None = free in any split (reading P4)


# ------------------------------------------------------------------ Sec. 7.1

def dense_stats(arr, labels) -> Stats:
    """T(U) and V(l, U) of a dense tensor whose axes carry ``labels`` in order:
    a slice along l counts when it holds at least one non-zero entry."""
    nz = np.asarray(arr) != 0
    V = {}
    for q, l in enumerate(labels):
        other = tuple(a for a in range(nz.ndim) if a != q)
        V[l] = int(np.count_nonzero(nz.any(axis=other))) if other else int(np.count_nonzero(nz))
    return Stats(float(np.count_nonzero(nz)), V)


def relation_stats(keys, bounds, tiles, labels) -> Stats:
    """Statistics of the tensor a tensor-relation stores.  ``labels`` names the
    key columns then the tile dimensions, in order.  The dense tensor, with
    axes in that order, is formed and measured (small inputs only)."""
    keys = np.asarray(keys, dtype=np.int64).reshape(len(tiles), len(bounds))
    tiles = np.asarray(tiles)
    dense = np.zeros(tuple(int(b) for b in bounds) + tiles.shape[1:], dtype=np.float64)
    for t in range(len(tiles)):
        dense[tuple(keys[t])] = tiles[t]
    return dense_stats(dense, labels)


def relation_stats_direct(keys, bounds, tiles):
    """The same statistics straight from the tuples, for relations too large
    to form densely: (T, [V of each key column] + [V of each tile dim]).  A
    key value counts when a tuple carrying it has a non-zero element; a tile
    index counts when some tuple has a non-zero element at it."""
    tiles = np.asarray(tiles)
    n = tiles.shape[0]
    keys = np.asarray(keys, dtype=np.int64).reshape(n, len(bounds))
    nz = tiles != 0
    T = int(np.count_nonzero(nz))
    live = nz.reshape(n, -1).any(axis=1) if n else np.zeros(0, bool)
    V = [int(len(np.unique(keys[live, c]))) for c in range(len(bounds))]
    for q in range(1, tiles.ndim):
        other = tuple(a for a in range(tiles.ndim) if a != q)
        V.append(int(np.count_nonzero(nz.any(axis=other))) if n else 0)
    return T, V


def drop_zero_tiles(keys, tiles):
    """The tuples whose tile holds a non-zero element, in their order (the
    zero-tuple elimination Sec. 4.2 allows)."""
    tiles = np.asarray(tiles)
    keep = (tiles.reshape(len(tiles), -1) != 0).any(axis=1) if len(tiles) else np.zeros(0, bool)
    return np.asarray(keys)[keep], tiles[keep]


def tuple_count(s: Stats, up) -> float:
    """Eq. eqn-count: n(↑U)·(1 − exp(−T(U)/n(↑U))), n(↑U) = Π V(l, U) over ↑U."""
    n = 1.0
    for l in up:
        n *= s.V[l]
    if n <= 0 or s.T <= 0:
        return 0.0
    return n * -math.expm1(-s.T / n)      # 1 − e^(−x) without cancellation for small x


def tuple_bytes(labels, up, bounds, dtype_bytes, key_bytes) -> float:
    """sizeof of one tuple: its key columns plus its tile."""
    tile = 1
    for l in labels:
        if l not in up:
            tile *= bounds[l]
    return key_bytes * len(up) + dtype_bytes * tile


# ------------------------------------------------------------------ Sec. 7.2

def join_tuples(sU, upU, sV, upV) -> float:
    """T_join: the textbook join estimate over the labels promoted on both sides."""
    den = 1.0
    for l in upU:
        if l in upV:
            den *= max(sU.V[l], sV.V[l])
    return tuple_count(sU, upU) * tuple_count(sV, upV) / den


def agg_tuples(sU, upU, sV, upV, upW, tj) -> float:
    """T_agg: min(T_join / 2, Π over ↑W of the label's distinct count) (reading P2)."""
    p = 1.0
    for l in upW:
        if l in upU and l in upV:
            p *= min(sU.V[l], sV.V[l])
        elif l in upU:
            p *= sU.V[l]
        else:
            p *= sV.V[l]
    return min(0.5 * tj, p)


def kernel_flops(lU, upU, lV, upV, bounds) -> float:
    lower = [l for l in lU if l not in upU] + [l for l in lV if l not in upV and l not in lU]
    f = 2.0
    for l in lower:
        f *= bounds[l]
    return f


def join_cost(cm, bounds, vU, upU, sU, vV, upV, sV) -> float:
    """C_join = T_join · [(sizeof Ū + sizeof V̄)·C_xfer + C_krnel + C_fixed]."""
    tj = join_tuples(sU, upU, sV, upV)
    size = (tuple_bytes(vU.labels, upU, bounds, vU.dtype_bytes, cm.key_bytes) +
            tuple_bytes(vV.labels, upV, bounds, vV.dtype_bytes, cm.key_bytes))
    krnel = cm.flop * kernel_flops(vU.labels, upU, vV.labels, upV, bounds)
    return tj * (size * cm.xfer + krnel + cm.fixed)


def agg_cost(cm, bounds, vW, upW, sU, upU, sV, upV) -> float:
    """C_agg = (T_join − T_agg) · [sizeof W̄ · C_xfer + C_add + C_fixed]."""
    tj = join_tuples(sU, upU, sV, upV)
    ta = agg_tuples(sU, upU, sV, upV, upW, tj)
    elems = 1
    for l in vW.labels:
        if l not in upW:
            elems *= bounds[l]
    size = tuple_bytes(vW.labels, upW, bounds, vW.dtype_bytes, cm.key_bytes)
    return (tj - ta) * (size * cm.xfer + cm.add * elems + cm.fixed)


def repart_cost(cm, bounds, v, s, up_in, up_out) -> float:
    """C_repart = (2·T(↑in ∪ ↑out) − T(↑in) − T(↑out)) · (sizeof W̄_int · C_xfer + C_fixed);
    nothing when the two decompositions promote the same labels."""
    if set(up_in) == set(up_out):
        return 0.0
    union = [l for l in v.labels if l in up_in or l in up_out]
    t = 2.0 * tuple_count(s, union) - tuple_count(s, up_in) - tuple_count(s, up_out)
    return t * (tuple_bytes(v.labels, union, bounds, v.dtype_bytes, cm.key_bytes) * cm.xfer + cm.fixed)


# ------------------------------------------------------------------- Alg. 2

def estimate_stats(sU, lU, sV, lV, lW) -> Stats:
    """Statistics of W = Σ U × V from those of U and V (reading P5)."""
    den = 1.0
    for l in lU:
        if l in lV:
            den *= max(sU.V[l], sV.V[l])
    tj = sU.T * sV.T / den
    V = {}
    for l in lW:
        if l in lU and l in lV:
            V[l] = min(sU.V[l], sV.V[l])
        elif l in lU:
            V[l] = sU.V[l]
        else:
            V[l] = sV.V[l]
    p = 1.0
    for l in lW:
        p *= V[l]
    T = min(tj, p)
    return Stats(T, {l: min(V[l], T) for l in lW})


def all_stats(graph):
    """Statistics of every vertex: the given ones, else GetStats estimates."""
    out = []
    for v in graph:
        if v.stats is not None:
            out.append(v.stats)
        else:
            if v.left is None:
                raise ValueError("an input tensor needs statistics")
            out.append(estimate_stats(out[v.left], graph[v.left].labels, out[v.right], graph[v.right].labels,
                                      v.labels))
    return out


# ------------------------------------------------------------------- Alg. 1

def subsets(labels):
    """Every subset of a label list, by increasing bit mask (reading P6)."""
    n = len(labels)
    for m in range(1 << n):
        yield tuple(labels[q] for q in range(n) if m >> q & 1)


def consistent(lX, upX, lW, upW):
    """Every label X shares with W is promoted in X iff it is promoted in W."""
    return all((l in upX) == (l in upW) for l in lX if l in lW)


def _check_tree(graph):
    used = {}
    for i, v in enumerate(graph):
        if (v.left is None) != (v.right is None):
            raise ValueError("a vertex has one input")
        if v.left is not None:
            for p in (v.left, v.right):
                if not 0 <= p < i:
                    raise ValueError("vertices must be in topological order")
                if p in used:
                    raise ValueError("a tensor is consumed twice (not a tree)")
                used[p] = i
            lU, lV = graph[v.left].labels, graph[v.right].labels
            if any(l not in lU and l not in lV for l in v.labels):
                raise ValueError("an output label appears in no input")


def _vertex_terms(graph, stats, bounds, cm, i, upW, upU, upV):
    v = graph[i]
    vU, vV = graph[v.left], graph[v.right]
    sU, sV = stats[v.left], stats[v.right]
    return (join_cost(cm, bounds, vU, upU, sU, vV, upV, sV) +
            agg_cost(cm, bounds, v, upW, sU, upU, sV, upV))


def tile_bytes(v, up, bounds) -> float:
    return tuple_bytes(v.labels, up, bounds, v.dtype_bytes, 0)


def _input_choices(graph, i, upW, bounds=None, cm=None):
    v = graph[i]
    vU, vV = graph[v.left], graph[v.right]
    lU, lV = vU.labels, vV.labels
    for upU in subsets(lU):
        if not consistent(lU, upU, v.labels, upW):
            continue
        for upV in subsets(lV):
            if consistent(lV, upV, v.labels, upW) and consistent(lV, upV, lU, upU):
                if cm is not None and cm.max_call_bytes > 0 and (
                        tile_bytes(vU, upU, bounds) + tile_bytes(vV, upV, bounds) + tile_bytes(v, upW, bounds)
                        > cm.max_call_bytes):
                    continue
                yield upU, upV


def optimize(graph, bounds, cm: CostModel, k: int = 1):
    """Alg. 1 extended to keep the k cheapest ways of producing every vertex in
    every output decomposition.  Returns the k cheapest plans of the whole tree
    as (cost, plan), plan = {vertex: (↑W, ↑U, ↑V)} for EinSum vertices and
    {vertex: ↑} for inputs.  The last vertex is the root."""
    _check_tree(graph)
    stats = all_stats(graph)
    C = []   # C[i][↑W] = sorted list of (cost, plan)
    for i, v in enumerate(graph):
        if v.left is None:
            C.append({up: [(_leaf_cost(v, stats[i], bounds, cm, up), {i: up})] for up in subsets(v.labels)})
            continue
        table = {}
        for upW in subsets(v.labels):
            cands = []
            for upU, upV in _input_choices(graph, i, upW, bounds, cm):
                here = _vertex_terms(graph, stats, bounds, cm, i, upW, upU, upV)
                sides = []
                for child, up_in_consumer in ((v.left, upU), (v.right, upV)):
                    opts = []
                    if graph[child].left is None:
                        opts = list(C[child][up_in_consumer])           # reading P4
                    else:
                        for up_prod, lst in C[child].items():
                            r = repart_cost(cm, bounds, graph[child], stats[child], up_prod, up_in_consumer)
                            opts.extend((c + r, p) for c, p in lst)
                    opts.sort(key=lambda e: e[0])
                    sides.append(opts[:k])
                for (cu, pu), (cv, pv) in itertools.product(*sides):
                    plan = dict(pu)
                    plan.update(pv)
                    plan[i] = (upW, upU, upV)
                    cands.append((here + cu + cv, plan))
            cands.sort(key=lambda e: e[0])
            table[upW] = cands[:k]
        C.append(table)
    root = C[-1]
    best = sorted((e for lst in root.values() for e in lst), key=lambda e: e[0])
    return best[:k]


def _leaf_cost(v, s, bounds, cm, up) -> float:
    """Reading an input tensor in split ``up``: free (P4), or a repartition
    from the split it is already stored in (P8)."""
    if v.fixed_up is None:
        return 0.0
    return repart_cost(cm, bounds, v, s, tuple(v.fixed_up), tuple(up))


def plan_cost(graph, bounds, cm: CostModel, plan) -> float:
    """Cost of one complete plan, term by term."""
    stats = all_stats(graph)
    total = 0.0
    for i, v in enumerate(graph):
        if v.left is None:
            continue
        upW, upU, upV = plan[i]
        total += _vertex_terms(graph, stats, bounds, cm, i, upW, upU, upV)
        for child, up_in in ((v.left, upU), (v.right, upV)):
            if graph[child].left is not None:
                total += repart_cost(cm, bounds, graph[child], stats[child], plan[child][0], up_in)
            else:
                total += _leaf_cost(graph[child], stats[child], bounds, cm, up_in)
    return total


def enumerate_plans(graph, bounds, cm: CostModel):
    """Every plan of the tree with its cost, by exhaustive search (tests only)."""
    _check_tree(graph)
    ein = [i for i, v in enumerate(graph) if v.left is not None]
    per_vertex = []
    for i in ein:
        opts = []
        for upW in subsets(graph[i].labels):
            for upU, upV in _input_choices(graph, i, upW, bounds, cm):
                opts.append((upW, upU, upV))
        per_vertex.append(opts)
    out = []
    for combo in itertools.product(*per_vertex):
        plan = dict(zip(ein, combo))
        for i in ein:
            v = graph[i]
            for child, up in ((v.left, plan[i][1]), (v.right, plan[i][2])):
                if graph[child].left is None:
                    plan[child] = up
        out.append((plan_cost(graph, bounds, cm, plan), plan))
    out.sort(key=lambda e: e[0])
    return out


def dense_tree(graph, dense_inputs):
    """Evaluate an EinSum tree densely in fp64 from its input tensors (each
    a numpy array with axes in its vertex's label order): every EinSum vertex
    is its definition, Σ over the labels absent from the output of U × V,
    computed by numpy.einsum.  Returns every vertex's tensor."""
    val = {}
    for i, v in enumerate(graph):
        if v.left is None:
            val[i] = np.asarray(dense_inputs[i], dtype=np.float64)
        else:
            lU, lV = graph[v.left].labels, graph[v.right].labels
            val[i] = np.einsum(f"{lU},{lV}->{v.labels}", val[v.left], val[v.right])
    return val


# ------------------------------------------------- Sec. 8.2, results used twice

def check_dag(graph):
    """Topological order, two producers per EinSum, output labels present."""
    for i, v in enumerate(graph):
        if (v.left is None) != (v.right is None):
            raise ValueError("a vertex has one input")
        if v.left is not None:
            for p in (v.left, v.right):
                if not 0 <= p < i:
                    raise ValueError("vertices must be in topological order")
            lU, lV = graph[v.left].labels, graph[v.right].labels
            if any(l not in lU and l not in lV for l in v.labels):
                raise ValueError("an output label appears in no input")
        elif v.stats is None:
            raise ValueError("an input tensor needs statistics")


def dag_trees(graph):
    """Reading P8: the tree (its root vertex) of every EinSum vertex, and the
    consuming edges (consumer, side) of every vertex."""
    uses = {i: [] for i in range(len(graph))}
    for i, v in enumerate(graph):
        if v.left is not None:
            uses[v.left].append((i, 0))
            uses[v.right].append((i, 1))
    tree = {}
    for i in reversed(range(len(graph))):
        if graph[i].left is None:
            continue
        tree[i] = tree[uses[i][0][0]] if len(uses[i]) == 1 else i
    return tree, uses


def optimize_dag(graph, bounds, cm: CostModel):
    """Sec. 8.2: optimise the trees of ``dag_trees`` one after another with
    Alg. 1 (k = 1).  Returns (cost, plan, tree) with plan[i] = (↑W, ↑U, ↑V) for
    every EinSum vertex (how it writes its result and reads its inputs)."""
    check_dag(graph)
    tree, _ = dag_trees(graph)
    stats = all_stats(graph)
    plan = {}
    total = 0.0
    for r in sorted(set(tree.values())):
        members = sorted(i for i in tree if tree[i] == r)
        sub, where = [], {}

        def leaf(p):
            # one leaf per consuming edge; a result decided by an earlier tree
            # keeps the split that tree chose
            v = graph[p]
            fixed = plan[p][0] if v.left is not None else None
            sub.append(Vertex(v.labels, v.dtype_bytes, stats=stats[p], fixed_up=fixed))
            return len(sub) - 1

        for i in members:
            v = graph[i]
            a = where[v.left] if v.left in where else leaf(v.left)
            b = where[v.right] if v.right in where else leaf(v.right)
            sub.append(Vertex(v.labels, v.dtype_bytes, a, b, stats=stats[i]))
            where[i] = len(sub) - 1
        best = optimize(sub, bounds, cm, k=1)
        if not best:
            raise ValueError("no decomposition of a tree satisfies the memory bound")
        cost, sp = best[0]
        total += cost
        for i in members:
            plan[i] = sp[where[i]]
    return total, plan, tree


def dag_plan_cost(graph, bounds, cm: CostModel, plan) -> float:
    """Cost of a DAG plan term by term: every EinSum's join and aggregation,
    plus a repartition on every edge whose producer (an EinSum) wrote another
    split than its consumer reads.  Inputs of the program are free (P4)."""
    stats = all_stats(graph)
    total = 0.0
    for i, v in enumerate(graph):
        if v.left is None:
            continue
        upW, upU, upV = plan[i]
        total += _vertex_terms(graph, stats, bounds, cm, i, upW, upU, upV)
        for child, up_in in ((v.left, upU), (v.right, upV)):
            if graph[child].left is not None:
                total += repart_cost(cm, bounds, graph[child], stats[child], plan[child][0], up_in)
    return total


def enumerate_dag_plans(graph, bounds, cm: CostModel):
    """Every plan of a DAG with its cost, by exhaustive search (tests only)."""
    check_dag(graph)
    ein = [i for i, v in enumerate(graph) if v.left is not None]
    per_vertex = [[(upW, upU, upV) for upW in subsets(graph[i].labels)
                   for upU, upV in _input_choices(graph, i, upW, bounds, cm)] for i in ein]
    out = []
    for combo in itertools.product(*per_vertex):
        plan = dict(zip(ein, combo))
        out.append((dag_plan_cost(graph, bounds, cm, plan), plan))
    out.sort(key=lambda e: e[0])
    return out
