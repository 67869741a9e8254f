"""Pins of the planner oracle (oracle/planner.py) against brute force, closed
forms and invariants that the paper's definitions fix (Sec. 7.1, 7.2, Alg. 1,
Alg. 2).  CPU only."""
from __future__ import annotations

import itertools
import math
import random

import numpy as np
import pytest

from oracle import planner as P


# ----------------------------------------------------------- statistics

def _brute_stats(arr, labels):
    """T and V by visiting every index tuple (pure Python)."""
    T = 0
    seen = {l: set() for l in labels}
    for idx in itertools.product(*[range(e) for e in arr.shape]):
        if arr[idx] != 0:
            T += 1
            for q, l in enumerate(labels):
                seen[l].add(idx[q])
    return T, {l: len(s) for l, s in seen.items()}


@pytest.mark.parametrize("shape", [(7,), (5, 6), (3, 4, 5), (2, 3, 2, 4)])
@pytest.mark.parametrize("density", [0.0, 0.05, 0.4, 1.0])
def test_dense_stats_brute_force(shape, density):
    rng = np.random.default_rng(len(shape) * 100 + int(density * 10))
    arr = rng.standard_normal(shape) * (rng.random(shape) < density)
    labels = "abcd"[: len(shape)]
    s = P.dense_stats(arr, labels)
    T, V = _brute_stats(arr, labels)
    assert s.T == T and s.V == V


def test_relation_stats_any_decomposition():
    # the statistics belong to the tensor, not to how it is decomposed
    rng = np.random.default_rng(3)
    dense = rng.standard_normal((4, 6, 5)) * (rng.random((4, 6, 5)) < 0.2)
    ref = P.dense_stats(dense, "abc")
    for up in range(1, 3):
        keys = np.array(list(itertools.product(*[range(e) for e in dense.shape[:up]])), dtype=np.int32)
        tiles = dense.reshape((-1,) + dense.shape[up:])
        s = P.relation_stats(keys, dense.shape[:up], tiles, "abc")
        assert s.T == ref.T and s.V == ref.V


def test_relation_stats_direct_matches_dense():
    rng = np.random.default_rng(11)
    for up in range(0, 3):
        dense = rng.standard_normal((5, 3, 4)) * (rng.random((5, 3, 4)) < 0.15)
        dense[1] = 0.0                                     # a key value with only zero tiles
        dense[..., 2] = -0.0                               # a tile index holding only negative zeros
        keys = np.array(list(itertools.product(*[range(e) for e in dense.shape[:up]])), dtype=np.int32)
        tiles = dense.reshape((-1,) + dense.shape[up:])
        T, V = P.relation_stats_direct(keys.reshape(len(tiles), up), dense.shape[:up], tiles)
        ref = P.dense_stats(dense, "abc")
        assert T == ref.T and V == [ref.V[c] for c in "abc"]
    T, V = P.relation_stats_direct(np.zeros((0, 1), np.int32), (4,), np.zeros((0, 3)))
    assert T == 0 and V == [0, 0]


def test_drop_zero_tiles_keeps_the_tensor():
    rng = np.random.default_rng(12)
    dense = rng.standard_normal((6, 4)) * (rng.random((6, 4)) < 0.2)
    keys = np.arange(6, dtype=np.int32)[:, None]
    k, t = P.drop_zero_tiles(keys, dense)
    back = np.zeros_like(dense)
    back[k[:, 0]] = t
    assert np.array_equal(back, dense) and all(np.any(x) for x in t)


# ----------------------------------------------------- Eq. eqn-count

def test_tuple_count_limits():
    s = P.Stats(1e9, {"a": 10, "b": 20})
    assert P.tuple_count(s, ("a", "b")) == pytest.approx(200.0)       # T ≫ n: every tuple present
    s = P.Stats(5.0, {"a": 1e6, "b": 1e6})
    assert P.tuple_count(s, ("a", "b")) == pytest.approx(5.0, rel=1e-9)  # n ≫ T: one tuple per entry
    s = P.Stats(3.0, {"a": 4})
    assert P.tuple_count(s, ()) == pytest.approx(1 - math.exp(-3.0))   # no promoted label: one tuple
    assert P.tuple_count(P.Stats(0.0, {"a": 4}), ("a",)) == 0.0


def test_tuple_count_uniform_monte_carlo():
    # T non-zeros placed uniformly at random: the tuple count of a decomposition
    # is the number of occupied (a, b) cells, whose expectation the estimate gives
    rng = np.random.default_rng(0)
    shape, T = (50, 40, 30), 2000
    counts = []
    for _ in range(20):
        flat = rng.choice(np.prod(shape), size=T, replace=False)
        a, b, c = np.unravel_index(flat, shape)
        arr = np.zeros(shape)
        arr[a, b, c] = 1.0
        s = P.dense_stats(arr, "abc")
        occupied = len(set(zip(a.tolist(), b.tolist())))
        counts.append((occupied, P.tuple_count(s, ("a", "b"))))
    occ = np.mean([c[0] for c in counts])
    est = np.mean([c[1] for c in counts])
    assert abs(est - occ) / occ < 0.03


# ---------------------------------------------------------- Sec. 7.2

def _dense(labels, bounds):
    T = float(np.prod([bounds[l] for l in labels]))
    return P.Stats(T * 1e3, {l: bounds[l] for l in labels})   # saturated: every tuple present


def test_join_estimate_matches_join_of_full_relations():
    bounds = {"J": 6, "K": 5, "j": 4}
    sU, sV = _dense("J", bounds), _dense("JK", bounds)
    # U keyed J (6 tuples), V keyed (J, K) (30 tuples): each U tuple meets 5 V tuples
    actual = sum(1 for u in range(6) for (j, k) in itertools.product(range(6), range(5)) if u == j)
    assert P.join_tuples(sU, ("J",), sV, ("J", "K")) == pytest.approx(actual)
    # no shared promoted label: the cross product
    assert P.join_tuples(sU, ("J",), sV, ("K",)) == pytest.approx(6 * 5)


def test_agg_estimate_counts_groups_of_full_relations():
    bounds = {"J": 6, "K": 5}
    sU, sV = _dense("J", bounds), _dense("JK", bounds)
    tj = P.join_tuples(sU, ("J",), sV, ("J", "K"))
    groups = len({k for (j, k) in itertools.product(range(6), range(5))})
    assert P.agg_tuples(sU, ("J",), sV, ("J", "K"), ("K",), tj) == pytest.approx(groups)


def test_repart_cost_invariants():
    bounds = {"a": 8, "b": 16, "c": 4}
    v = P.Vertex("abc", 2)
    s = P.Stats(300.0, {"a": 8, "b": 12, "c": 4})
    cm = P.CostModel(xfer=1e-3, fixed=0.5)
    subs = list(P.subsets("abc"))
    for x, y in itertools.product(subs, subs):
        cxy = P.repart_cost(cm, bounds, v, s, x, y)
        assert cxy >= -1e-9
        assert cxy == pytest.approx(P.repart_cost(cm, bounds, v, s, y, x))   # same intermediate both ways
        if set(x) == set(y):
            assert cxy == 0.0
        if set(x) < set(y):
            # only the decomposition step runs: T(out) − T(in) new tuples
            per = P.tuple_bytes("abc", y, bounds, 2, 4) * cm.xfer + cm.fixed
            assert cxy == pytest.approx((P.tuple_count(s, y) - P.tuple_count(s, x)) * per)


# ------------------------------------------------------------ Alg. 2

def test_estimate_stats_dense_product_is_exact():
    bounds = {"i": 3, "j": 4, "k": 5}
    sU = P.dense_stats(np.ones((3, 4)), "ij")
    sV = P.dense_stats(np.ones((4, 5)), "jk")
    sW = P.estimate_stats(sU, "ij", sV, "jk", "ik")
    ref = P.dense_stats(np.ones((3, 4)) @ np.ones((4, 5)), "ik")
    assert sW.T == ref.T and sW.V == ref.V


# ------------------------------------------------------------ Alg. 1

def _valid(graph, plan):
    """Independent validity check of one plan: every label has one class
    within each EinSum (inputs and output agree)."""
    for i, v in enumerate(graph):
        if v.left is None:
            continue
        upW, upU, upV = plan[i]
        lU, lV = graph[v.left].labels, graph[v.right].labels
        for l in set(lU) | set(lV):
            classes = set()
            for lab, up in ((lU, upU), (lV, upV), (v.labels, upW)):
                if l in lab:
                    classes.add(l in up)
            if len(classes) != 1:
                return False
    return True


def _random_tree(rng, shape):
    bounds = {l: rng.choice([2, 4, 8, 16, 64]) for l in "abcdefg"}

    def leaf(labels):
        T = float(rng.uniform(1, np.prod([bounds[l] for l in labels])))
        return P.Vertex(labels, int(rng.choice([2, 4])), stats=P.Stats(
            T, {l: float(rng.integers(1, bounds[l] + 1)) for l in labels}))

    if shape == "chain":      # ((X × Y) × Z), the message-passing shape
        g = [leaf("fab"), leaf("abcd"), P.Vertex("cdf", 2, 0, 1), leaf("fg"), P.Vertex("cdg", 4, 2, 3)]
    elif shape == "transpose":  # (X × Y)^T × Z
        g = [leaf("ab"), leaf("bc"), P.Vertex("ca", 2, 0, 1), leaf("ad"), P.Vertex("cd", 4, 2, 3)]
    else:                     # two products joined: (X × Y) × (Z × Q)
        g = [leaf("ab"), leaf("bc"), P.Vertex("ac", 2, 0, 1), leaf("cd"), leaf("de"), P.Vertex("ce", 2, 3, 4),
             P.Vertex("ae", 4, 2, 5)]
    cm = P.CostModel(xfer=rng.uniform(0, 1e-3), flop=rng.uniform(0, 1e-4), add=rng.uniform(0, 1e-3),
                     fixed=rng.uniform(0, 10))
    return g, bounds, cm


@pytest.mark.parametrize("shape", ["chain", "transpose", "bushy"])
@pytest.mark.parametrize("seed", range(4))
def test_dp_matches_exhaustive_search(shape, seed):
    rng = np.random.default_rng(seed)
    g, bounds, cm = _random_tree(rng, shape)
    every = P.enumerate_plans(g, bounds, cm)
    assert all(_valid(g, p) for _, p in every)
    best = P.optimize(g, bounds, cm, k=6)
    assert [c for c, _ in best] == pytest.approx([c for c, _ in every[:6]], rel=1e-12)
    for c, plan in best:
        assert _valid(g, plan)
        assert P.plan_cost(g, bounds, cm, plan) == pytest.approx(c, rel=1e-12)
    # the k plans are distinct
    keys = {tuple(sorted((i, repr(x)) for i, x in p.items())) for _, p in best}
    assert len(keys) == len(best)


def test_memory_bound_exhaustive():
    rng = np.random.default_rng(3)
    g, bounds, cm = _random_tree(rng, "chain")
    every = P.enumerate_plans(g, bounds, cm)
    cm.max_call_bytes = 2048.0
    bounded = P.enumerate_plans(g, bounds, cm)
    ok = [(c, p) for c, p in every if all(
        P.tile_bytes(g[v.left], p[i][1], bounds) + P.tile_bytes(g[v.right], p[i][2], bounds) +
        P.tile_bytes(v, p[i][0], bounds) <= 2048.0 for i, v in enumerate(g) if v.left is not None)]
    assert [c for c, _ in bounded] == [c for c, _ in ok]
    best = P.optimize(g, bounds, cm, k=4)
    assert [c for c, _ in best] == pytest.approx([c for c, _ in bounded[:4]], rel=1e-12)


def test_plan_count_closed_form():
    # each label takes one class per EinSum: 2^|ℓU ∪ ℓV| plans per vertex
    rng = np.random.default_rng(1)
    g, bounds, cm = _random_tree(rng, "chain")
    n1 = 2 ** len(set("fab") | set("abcd"))
    n2 = 2 ** len(set("cdf") | set("fg"))
    assert len(P.enumerate_plans(g, bounds, cm)) == n1 * n2


def test_planted_consistency_mistake_is_caught(monkeypatch):
    # a planted mistake: only the output's labels constrain the inputs
    rng = np.random.default_rng(1)
    g, bounds, cm = _random_tree(rng, "chain")
    orig = P.consistent
    monkeypatch.setattr(P, "consistent", lambda lX, upX, lW, upW: True if lW != g[2].labels and lW != g[4].labels
                        else orig(lX, upX, lW, upW))
    every = P.enumerate_plans(g, bounds, cm)
    assert len(every) != 2 ** 6 * 2 ** 5 or not all(_valid(g, p) for _, p in every)


def test_tree_checks():
    s = P.Stats(1.0, {"a": 1})
    with pytest.raises(ValueError):
        P.optimize([P.Vertex("a", stats=s), P.Vertex("a", 2, 0, 0)], {"a": 1}, P.CostModel())
    with pytest.raises(ValueError):
        P.optimize([P.Vertex("a", stats=s), P.Vertex("a", stats=s), P.Vertex("b", 2, 0, 1)], {"a": 1, "b": 1},
                   P.CostModel())


def test_dense_tree_brute_force():
    from tests.ucl_testutil import brute_force
    rng = np.random.default_rng(5)
    X, Y, Z = rng.standard_normal((2, 3)), rng.standard_normal((3, 2, 2)), rng.standard_normal((2, 3))
    g = [P.Vertex("ab", stats=P.Stats(1, {})), P.Vertex("bcd", stats=P.Stats(1, {})), P.Vertex("cda", 4, 0, 1),
         P.Vertex("ae", stats=P.Stats(1, {})), P.Vertex("ce", 4, 2, 3)]
    val = P.dense_tree(g, {0: X, 1: Y, 3: Z})
    T = brute_force("ab,bcd->cda", [X, Y])
    np.testing.assert_allclose(val[2], T, rtol=1e-12)
    np.testing.assert_allclose(val[4], brute_force("cda,ae->ce", [T, Z]), rtol=1e-12)


# ------------------------------------------- Sec. 8.2: results used twice

def _rand_dag(rng, n_ein, bounds_choice=(2, 3, 4, 8), labels="abcde", max_lab=3, reuse=True):
    """A random EinSum DAG: three or four inputs, then n_ein binary EinSums on
    earlier vertices; with ``reuse`` some intermediate is consumed twice."""
    bounds = {l: int(rng.choice(bounds_choice)) for l in labels}

    def stats_for(lab):
        T = float(rng.uniform(1, np.prod([float(bounds[l]) for l in lab])))
        return P.Stats(T, {l: float(rng.integers(1, bounds[l] + 1)) for l in lab})

    g = []
    for _ in range(int(rng.integers(3, 5))):
        lab = "".join(rng.choice(list(labels), size=int(rng.integers(1, max_lab + 1)), replace=False))
        g.append(P.Vertex(lab, int(rng.choice([2, 4])), stats=stats_for(lab)))
    n_in = len(g)
    for j in range(n_ein):
        i = len(g)
        if reuse and j == n_ein - 1 and n_ein >= 2:
            a, b = n_in, i - 1          # the first intermediate is read again
        else:
            a, b = (int(x) for x in rng.choice(i, size=2, replace=False))
            if j > 0 and rng.random() < 0.6:
                a = i - 1
        pool = sorted(set(g[a].labels) | set(g[b].labels))
        k = int(rng.integers(1, min(max_lab, len(pool)) + 1))
        lab = "".join(rng.choice(pool, size=k, replace=False))
        g.append(P.Vertex(lab, int(rng.choice([2, 4])), a, b))
    return g, bounds


def _cm(rng, repart=True):
    return P.CostModel(xfer=float(rng.uniform(1e-9, 1e-6)) if repart else 0.0,
                       flop=float(rng.uniform(1e-12, 1e-9)), add=float(rng.uniform(0, 1e-9)),
                       fixed=float(rng.uniform(0, 1e-6)) if repart else 0.0)


def _rand_tree(rng, bushy):
    """A tree: a chain ((A B) C) D, or a bushy (A B) (C D), random labels."""
    bounds = {l: int(rng.choice([2, 3, 4, 8])) for l in "abcde"}

    def leaf(lab):
        T = float(rng.uniform(1, np.prod([float(bounds[l]) for l in lab])))
        return P.Vertex(lab, int(rng.choice([2, 4])), stats=P.Stats(
            T, {l: float(rng.integers(1, bounds[l] + 1)) for l in lab}))

    def lab():
        return "".join(rng.choice(list("abcde"), size=int(rng.integers(1, 4)), replace=False))

    def ein(g, a, b):
        pool = sorted(set(g[a].labels) | set(g[b].labels))
        out = "".join(rng.choice(pool, size=int(rng.integers(1, min(3, len(pool)) + 1)), replace=False))
        g.append(P.Vertex(out, int(rng.choice([2, 4])), a, b))

    g = [leaf(lab()), leaf(lab())]
    ein(g, 0, 1)                               # 2
    g.append(leaf(lab()))                      # 3
    if bushy:
        g.append(leaf(lab()))                  # 4
        ein(g, 3, 4)                           # 5
        ein(g, 2, 5)                           # 6
    else:
        ein(g, 2, 3)                           # 4
        g.append(leaf(lab()))                  # 5
        ein(g, 4, 5)                           # 6
    return g, bounds


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("bushy", [False, True])
def test_dag_on_a_tree_is_alg1(seed, bushy):
    """Without a result used twice the heuristic is Alg. 1 itself: one tree,
    the same cost and the same plan."""
    rng = np.random.default_rng(500 + seed)
    g, bounds = _rand_tree(rng, bushy)
    cm = _cm(rng)
    cost, plan, tree = P.optimize_dag(g, bounds, cm)
    c1, p1 = P.optimize(g, bounds, cm, k=1)[0]
    assert cost == pytest.approx(c1, rel=1e-12)
    assert plan == {i: p1[i] for i in p1 if g[i].left is not None}
    assert set(tree.values()) == {6}


@pytest.mark.parametrize("seed", range(12))
def test_dag_trees_cut_at_results_used_twice(seed):
    rng = np.random.default_rng(600 + seed)
    g, _ = _rand_dag(rng, int(rng.integers(3, 7)))
    tree, uses = P.dag_trees(g)
    ein = [i for i, v in enumerate(g) if v.left is not None]
    assert sorted(tree) == ein
    for i in ein:
        n_use = len(uses[i])
        if n_use != 1:
            assert tree[i] == i                         # an output or a result used twice roots a tree
        else:
            assert tree[i] == tree[uses[i][0][0]]      # else it joins its consumer's tree
    for r in set(tree.values()):
        members = [i for i in ein if tree[i] == r]
        assert max(members) == r
        # inside a tree no result is read twice
        reads = [p for i in members for p in (g[i].left, g[i].right) if p in members]
        assert len(reads) == len(set(reads)) == len(members) - 1
        # what a tree reads from other trees are roots decided before it
        for i in members:
            for p in (g[i].left, g[i].right):
                if g[p].left is not None and tree[p] != r:
                    assert tree[p] == p < r


@pytest.mark.parametrize("seed", range(10))
def test_dag_plan_cost_and_local_optimality(seed):
    """The reported cost is the plan's cost term by term, and each tree's
    choices are the cheapest for that tree with the earlier trees' splits
    held fixed (exhaustive over the tree's own vertices)."""
    rng = np.random.default_rng(700 + seed)
    g, bounds = _rand_dag(rng, int(rng.integers(2, 5)))
    cm = _cm(rng)
    cost, plan, tree = P.optimize_dag(g, bounds, cm)
    assert cost == pytest.approx(P.dag_plan_cost(g, bounds, cm, plan), rel=1e-12)
    stats = P.all_stats(g)
    for r in set(tree.values()):
        members = sorted(i for i in tree if tree[i] == r)

        def tree_cost(choice):
            tot = 0.0
            for i in members:
                upW, upU, upV = choice[i]
                tot += P._vertex_terms(g, stats, bounds, cm, i, upW, upU, upV)
                for p, up_in in ((g[i].left, upU), (g[i].right, upV)):
                    if g[p].left is not None:
                        up_p = choice[p][0] if p in choice else plan[p][0]
                        tot += P.repart_cost(cm, bounds, g[p], stats[p], up_p, up_in)
            return tot

        opts = [[(upW, upU, upV) for upW in P.subsets(g[i].labels)
                 for upU, upV in P._input_choices(g, i, upW, bounds, cm)] for i in members]
        best = min(tree_cost(dict(zip(members, c))) for c in itertools.product(*opts))
        assert tree_cost({i: plan[i] for i in members}) == pytest.approx(best, rel=1e-12)


@pytest.mark.parametrize("seed", range(8))
def test_dag_heuristic_against_exhaustive(seed):
    """Exhaustive search over the whole DAG: the heuristic never beats the
    optimum, and with free repartition (no C_xfer, no C_fixed) the trees are
    independent, so it finds the optimum."""
    rng = np.random.default_rng(800 + seed)
    g, bounds = _rand_dag(rng, 3, labels="abcd", max_lab=3)
    every = P.enumerate_dag_plans(g, bounds, _cm(np.random.default_rng(seed)))
    cm = _cm(np.random.default_rng(seed))
    cost, plan, _ = P.optimize_dag(g, bounds, cm)
    assert cost >= every[0][0] * (1 - 1e-12)
    cm0 = _cm(np.random.default_rng(seed), repart=False)
    cost0, plan0, _ = P.optimize_dag(g, bounds, cm0)
    best0 = P.enumerate_dag_plans(g, bounds, cm0)[0][0]
    assert cost0 == pytest.approx(best0, rel=1e-12)


def test_dag_fixed_split_costs_a_repartition():
    """A result decided by an earlier tree is read for free in its own split
    and for C_repart in another (reading P8); a planted mistake that reads it
    for free in every split is caught by the exhaustive check above."""
    rng = np.random.default_rng(9)
    s = P.Stats(50.0, {"a": 8.0, "b": 6.0})
    bounds = {"a": 8, "b": 8}
    cm = _cm(rng)
    leaf = P.Vertex("ab", 2, stats=s, fixed_up=("a",))
    assert P._leaf_cost(leaf, s, bounds, cm, ("a",)) == 0.0
    for up in (("b",), (), ("a", "b")):
        assert P._leaf_cost(leaf, s, bounds, cm, up) == pytest.approx(
            P.repart_cost(cm, bounds, leaf, s, ("a",), up), rel=0) and P._leaf_cost(leaf, s, bounds, cm, up) > 0
    free = P.Vertex("ab", 2, stats=s)
    assert all(P._leaf_cost(free, s, bounds, cm, up) == 0.0 for up in P.subsets("ab"))
