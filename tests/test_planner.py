"""The native planner (ucl_plan, host C++) against the planner oracle: the k
cheapest plans of random EinSum trees, their costs and their validity.  Host
logic only, so these run without a GPU."""
from __future__ import annotations

import numpy as np
import pytest

from oracle import planner as P
from paper_2603_08957_gb300 import UclError, plan, plan_dag


def _tree(rng, shape):
    bounds = {l: int(rng.choice([2, 4, 8, 16, 64, 1000])) for l in "abcdefgh"}

    def leaf(labels):
        T = float(rng.uniform(1, np.prod([float(bounds[l]) for l in labels])))
        return P.Vertex(labels, int(rng.choice([2, 4])), stats=P.Stats(
            T, {l: float(rng.integers(1, bounds[l] + 1)) for l in labels}))

    if shape == "chain":          # message passing: (X × Y) × Z
        g = [leaf("fab"), leaf("abcd"), P.Vertex("cdf", 2, 0, 1), leaf("fg"), P.Vertex("cdg", 4, 2, 3)]
    elif shape == "two_layer":    # ((X × Y) × W1) × Y' × W2
        g = [leaf("fab"), leaf("abcd"), P.Vertex("cdf", 2, 0, 1), leaf("fg"), P.Vertex("cdg", 2, 2, 3),
             leaf("cdeh"), P.Vertex("ehg", 2, 4, 5), leaf("gf"), P.Vertex("ehf", 4, 6, 7)]
    elif shape == "transpose":
        g = [leaf("ab"), leaf("bc"), P.Vertex("ca", 2, 0, 1), leaf("ad"), P.Vertex("cd", 4, 2, 3)]
    else:
        g = [leaf("ab"), leaf("bc"), P.Vertex("ac", 2, 0, 1), leaf("cd"), leaf("de"), P.Vertex("ce", 2, 3, 4),
             P.Vertex("ae", 4, 2, 5)]
    cm = P.CostModel(xfer=float(rng.uniform(1e-12, 1e-9)), flop=float(rng.uniform(1e-15, 1e-12)),
                     add=float(rng.uniform(0, 1e-12)), fixed=float(rng.uniform(0, 1e-7)))
    return g, bounds, cm


def _native(g, bounds, cm, k, measured=False):
    verts = []
    for v in g:
        d = {"labels": v.labels, "dtype_bytes": v.dtype_bytes}
        if v.left is None:
            d.update(T=v.stats.T, V=v.stats.V)
        else:
            d.update(left=v.left, right=v.right)
            if measured and v.stats is not None:
                d.update(T=v.stats.T, V=v.stats.V)
        verts.append(d)
    return plan(verts, bounds, {"xfer": cm.xfer, "flop": cm.flop, "add": cm.add, "fixed": cm.fixed,
                                "max_call_bytes": cm.max_call_bytes}, k=k)


def _as_oracle_plan(g, per):
    out = {}
    for i, v in enumerate(g):
        if v.left is None:
            out[i] = tuple(per[i])
        else:
            out[i] = tuple(tuple(x) for x in per[i])
    return out


@pytest.mark.parametrize("shape", ["chain", "two_layer", "transpose", "bushy"])
@pytest.mark.parametrize("seed", range(5))
def test_native_k_best_matches_oracle(shape, seed):
    rng = np.random.default_rng(1000 + seed)
    g, bounds, cm = _tree(rng, shape)
    k = 8
    ref = P.optimize(g, bounds, cm, k=k)
    got = _native(g, bounds, cm, k)
    assert len(got) == len(ref)
    assert [c for c, _ in got] == pytest.approx([c for c, _ in ref], rel=1e-12)
    for (c, per), (rc, rplan) in zip(got, ref):
        mine = _as_oracle_plan(g, per)
        # the oracle's cost of the native plan is the native cost
        assert P.plan_cost(g, bounds, cm, mine) == pytest.approx(c, rel=1e-12)
    # where costs are not tied, the plans are the same
    for j, ((c, per), (rc, rplan)) in enumerate(zip(got, ref)):
        tied = any(abs(c - got[m][0]) <= 1e-12 * abs(c) for m in range(len(got)) if m != j)
        if not tied:
            assert _as_oracle_plan(g, per) == rplan


@pytest.mark.parametrize("seed", range(3))
def test_memory_bound_matches_oracle(seed):
    rng = np.random.default_rng(2000 + seed)
    g, bounds, cm = _tree(rng, "two_layer")
    cm.max_call_bytes = float(rng.choice([256.0, 4096.0, 65536.0]))
    ref = P.optimize(g, bounds, cm, k=5)
    got = _native(g, bounds, cm, 5)
    assert [c for c, _ in got] == pytest.approx([c for c, _ in ref], rel=1e-12)
    for c, per in got:
        plan_ = _as_oracle_plan(g, per)
        for i, v in enumerate(g):
            if v.left is not None:
                upW, upU, upV = plan_[i]
                tot = (P.tile_bytes(g[v.left], upU, bounds) + P.tile_bytes(g[v.right], upV, bounds) +
                       P.tile_bytes(v, upW, bounds))
                assert tot <= cm.max_call_bytes


def test_measured_intermediate_statistics_are_used():
    rng = np.random.default_rng(7)
    g, bounds, cm = _tree(rng, "chain")
    g[2].stats = P.Stats(1234.0, {"c": 3.0, "d": 5.0, "f": 7.0})
    ref = P.optimize(g, bounds, cm, k=3)
    got = _native(g, bounds, cm, 3, measured=True)
    assert [c for c, _ in got] == pytest.approx([c for c, _ in ref], rel=1e-12)


def test_plan_rejects_bad_trees():
    bounds = {"a": 4, "b": 4}
    leaf = {"labels": "ab", "T": 3.0, "V": {"a": 2, "b": 2}}
    cm = {"xfer": 1.0}
    with pytest.raises(UclError):      # consumed twice
        plan([leaf, {"labels": "a", "left": 0, "right": 0}], bounds, cm)
    with pytest.raises(UclError):      # output label in no input
        plan([leaf, leaf, {"labels": "ac", "left": 0, "right": 1}], {"a": 4, "b": 4, "c": 2}, cm)
    with pytest.raises(UclError):      # label without a bound
        plan([{"labels": "ax", "T": 1.0, "V": {"a": 1, "x": 1}}], bounds, cm)
    with pytest.raises(UclError):      # not topological
        plan([leaf, {"labels": "a", "left": 2, "right": 0}, leaf], bounds, cm)


# --------------------------------------- Sec. 8.2: results used more than once

def _native_dag(g, bounds, cm):
    verts = []
    for v in g:
        d = {"labels": v.labels, "dtype_bytes": v.dtype_bytes}
        if v.left is None:
            d.update(T=v.stats.T, V=v.stats.V)
        else:
            d.update(left=v.left, right=v.right)
        verts.append(d)
    return plan_dag(verts, bounds, {"xfer": cm.xfer, "flop": cm.flop, "add": cm.add, "fixed": cm.fixed,
                                    "max_call_bytes": cm.max_call_bytes})


def _random_dag(rng, n_ein):
    """Inputs, then n_ein EinSums on earlier vertices; results are read again
    on purpose (also as both operands of one EinSum)."""
    bounds = {l: int(rng.choice([2, 4, 8, 16, 64, 1000])) for l in "abcdefg"}

    def stats_for(lab):
        T = float(rng.uniform(1, np.prod([float(bounds[l]) for l in lab])))
        return P.Stats(T, {l: float(rng.integers(1, bounds[l] + 1)) for l in lab})

    g = []
    for _ in range(int(rng.integers(3, 6))):
        lab = "".join(rng.choice(list("abcdefg"), size=int(rng.integers(1, 4)), replace=False))
        g.append(P.Vertex(lab, int(rng.choice([2, 4])), stats=stats_for(lab)))
    n_in = len(g)
    for j in range(n_ein):
        i = len(g)
        r = rng.random()
        if j > 0 and r < 0.15:
            a = b = int(rng.integers(n_in, i))            # one result as both operands
        elif j > 0 and r < 0.6:
            a, b = i - 1, int(rng.integers(0, i - 1))
        else:
            a, b = (int(x) for x in rng.choice(i, size=2, replace=False))
        pool = sorted(set(g[a].labels) | set(g[b].labels))
        lab = "".join(rng.choice(pool, size=int(rng.integers(1, min(4, len(pool)) + 1)), replace=False))
        g.append(P.Vertex(lab, int(rng.choice([2, 4])), a, b))
    cm = P.CostModel(xfer=float(rng.uniform(1e-12, 1e-9)), flop=float(rng.uniform(1e-15, 1e-12)),
                     add=float(rng.uniform(0, 1e-12)), fixed=float(rng.uniform(0, 1e-7)))
    return g, bounds, cm


@pytest.mark.parametrize("seed", range(25))
def test_native_dag_matches_oracle(seed):
    rng = np.random.default_rng(3000 + seed)
    g, bounds, cm = _random_dag(rng, int(rng.integers(2, 9)))
    if seed % 5 == 4:
        cm.max_call_bytes = float(rng.choice([4096.0, 1e6]))
    try:
        ref_cost, ref_plan, ref_tree = P.optimize_dag(g, bounds, cm)
    except ValueError:
        with pytest.raises(UclError):
            _native_dag(g, bounds, cm)
        return
    cost, per, roots = _native_dag(g, bounds, cm)
    assert cost == pytest.approx(ref_cost, rel=1e-12)
    assert {i: r for i, r in enumerate(roots) if r >= 0} == ref_tree
    mine = {i: tuple(tuple(x) for x in per[i]) for i, v in enumerate(g) if v.left is not None}
    # the oracle's term-by-term cost of the native plan is the native cost
    assert P.dag_plan_cost(g, bounds, cm, mine) == pytest.approx(cost, rel=1e-12)
    # an input's entry is the split its first consumer reads
    for i, v in enumerate(g):
        if v.left is None:
            cons = [(c, s) for c, w in enumerate(g) if w.left is not None for s, p in enumerate((w.left, w.right))
                    if p == i]
            if cons:
                c, s = cons[0]
                assert tuple(per[i]) == tuple(mine[c][1 + s])


def test_native_dag_on_the_gnn_two_layer_program():
    """Y is read by both message-passing EinSums: inputs may be read twice and
    stay free; one tree, the same plan as the tree planner's."""
    rng = np.random.default_rng(17)
    g, bounds, cm = _tree(rng, "two_layer")
    ref = P.optimize(g, bounds, cm, k=1)[0]
    cost, per, roots = _native_dag(g, bounds, cm)
    assert cost == pytest.approx(ref[0], rel=1e-12)
    assert {i: roots[i] for i in range(len(g)) if g[i].left is not None} == {2: 8, 4: 8, 6: 8, 8: 8}


def test_native_dag_errors():
    rng = np.random.default_rng(23)
    g, bounds, cm = _random_dag(rng, 4)
    cm.max_call_bytes = 1.0                     # no tile fits: no plan for the first tree
    with pytest.raises(ValueError):
        P.optimize_dag(g, bounds, cm)
    with pytest.raises(UclError):
        _native_dag(g, bounds, cm)
    bounds2 = {"a": 4, "b": 4}
    leaf = {"labels": "ab", "T": 3.0, "V": {"a": 2, "b": 2}}
    ok = plan_dag([leaf, {"labels": "a", "left": 0, "right": 0}], bounds2, {"xfer": 1.0})
    assert ok[2] == [-1, 1]                     # one input read as both operands is allowed here
    with pytest.raises(UclError):               # not topological
        plan_dag([leaf, {"labels": "a", "left": 2, "right": 0}, leaf], bounds2, {"xfer": 1.0})
    with pytest.raises(UclError):               # output label in no input
        plan_dag([leaf, leaf, {"labels": "ac", "left": 0, "right": 1}], {"a": 4, "b": 4, "c": 2}, {"xfer": 1.0})
