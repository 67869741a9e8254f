"""GPU parity of the planner's statistics and zero-tuple elimination against
the oracle, and plans chosen by ucl_plan executed end to end: every one of
the cheapest plans computes the same tensor as the dense definition."""
import numpy as np
import pytest
import torch

import workloads
from oracle import planner as P
from paper_2603_08957_gb300 import Context, plan, plan_dag, program
from tests.parity import gpu_rel
from tests.ucl_testutil import decompose, random_sparse, recompose

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = Context(0)
    yield c
    c.close()


def _exact(a, dtype):
    t = torch.from_numpy(np.asarray(a, dtype=np.float64))
    return t.to(dtype).to(torch.float64).numpy()


STATS_CASES = [
    # (dense shape, promoted axes, density)
    ((40, 64, 64), (0,), 0.01),        # message-passing tiles, mostly empty
    ((12, 9, 16, 16), (0, 1), 0.2),    # two key columns
    ((7, 5, 3), (0,), 0.3),            # odd inner extent: one element per load
    ((6, 8, 4, 2), (1,), 0.5),         # promoted label between tile dims
    ((300,), (0,), 0.5),               # scalar tiles
    ((128, 1000), (), 0.9),            # one key-less dense tuple
    ((5, 6, 7), (0, 1, 2), 0.4),       # scalars keyed by every label
]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("shape,promoted,density", STATS_CASES)
def test_stats_and_drop_zero_match_oracle(ctx, shape, promoted, density, dtype):
    rng = np.random.default_rng(abs(hash((shape, promoted))) % 2**31)
    dense = random_sparse(rng, shape, density=density, block_axes=range(len(shape)))
    if dense.size > 10:
        dense.flat[rng.integers(0, dense.size, 3)] = -0.0      # negative zeros are zeros
    dense = _exact(dense, dtype)
    labels = "abcd"[: len(shape)]
    up = {labels[a] for a in promoted}
    keys, bounds, tiles = decompose(dense, labels, up, drop_zero=False)
    rel = gpu_rel(ctx, (keys.astype(np.int32), tuple(int(b) for b in bounds), torch.from_numpy(tiles).to(dtype)))
    T, V = ctx.stats(rel)
    wT, wV = P.relation_stats_direct(keys, bounds, tiles)
    assert (T, V) == (wT, wV)
    kept = ctx.drop_zero_tiles(rel)
    wk, wt = P.drop_zero_tiles(keys, tiles)
    gk, gt = kept.download()
    assert kept.n == len(wk)
    assert np.array_equal(gk.reshape(wk.shape), wk)
    assert np.array_equal(gt.to(torch.float64).numpy().reshape(wt.shape), wt)


def test_stats_nan_empty_and_zero(ctx):
    t = torch.zeros((4, 8), dtype=torch.bfloat16)
    t[2, 5] = float("nan")
    rel = gpu_rel(ctx, (np.arange(4, dtype=np.int32)[:, None], (4,), t))
    assert ctx.stats(rel) == (1, [1, 1])
    assert ctx.drop_zero_tiles(rel).n == 1
    zero = gpu_rel(ctx, (np.arange(3, dtype=np.int32)[:, None], (9,), torch.zeros((3, 2, 2))))
    assert ctx.stats(zero) == (0, [0, 0, 0])
    assert ctx.drop_zero_tiles(zero).n == 0
    empty = gpu_rel(ctx, (np.zeros((0, 1), np.int32), (9,), torch.zeros((0, 2))))
    assert ctx.stats(empty) == (0, [0, 0])
    out = ctx.drop_zero_tiles(empty)
    assert out.n == 0 and out.bounds == (9,) and out.shape == (2,)


def test_stats_wide_key_bound(ctx):
    rng = np.random.default_rng(2)
    keys = np.sort(rng.choice(1 << 24, size=5000, replace=False)).astype(np.int32)[:, None]
    tiles = rng.standard_normal((5000, 16)) * (rng.random((5000, 16)) < 0.1)
    tiles = _exact(tiles, torch.float32)
    rel = gpu_rel(ctx, (keys, (1 << 24,), torch.from_numpy(tiles).float()))
    assert ctx.stats(rel) == P.relation_stats_direct(keys, (1 << 24,), tiles)


def test_stats_full_size_message_passing(ctx):
    """Y of the message-passing workload (R-MAT, 1.6M edges in ~373k 64x64
    tiles) and X (128 x 100000): statistics against the oracle; a
    repartition that creates empty tuples, then zero-tuple elimination."""
    w = workloads.gnn_chain(seed=0, n=100_000, device="cpu")
    for name in ("X", "Y"):
        k, b, t = w[name]
        rel = gpu_rel(ctx, w[name])
        bits = t.view(torch.int16).numpy() & 0x7FFF      # bf16 non-zero test on the bit pattern
        assert ctx.stats(rel) == P.relation_stats_direct(k, b, bits)
    Y = gpu_rel(ctx, w["Y"])
    rows = ctx.repartition("JKjk->JKj|k", Y)             # one tuple per (J, K, j): mostly empty rows
    kept = ctx.drop_zero_tiles(rows)
    src, dst = w["edges"]
    # one kept tuple per distinct (source vertex, destination block) pair
    pairs = np.unique((src.astype(np.int64) << 20) | (dst.astype(np.int64) // 64))
    assert kept.n == len(pairs)
    T, V = ctx.stats(kept)
    assert T == len(np.unique((src.astype(np.int64) << 20) | dst.astype(np.int64)))


# ------------------------------------------------------- plans, end to end

def _chain_tree(w):
    """Message passing as an EinSum tree over lower-case labels: X[f,a,b]
    (a = vertex block J, b = index j within it), Y[a,b,c,d] (c = K, d = k),
    T = Σ_ab X Y [c,d,f], out = Σ_f T Z [c,d,g]; T and out in fp32."""
    return [
        {"labels": "fab"},
        {"labels": "abcd"},
        {"labels": "cdf", "left": 0, "right": 1, "dtype_bytes": 4},
        {"labels": "fg"},
        {"labels": "cdg", "left": 2, "right": 3, "dtype_bytes": 4},
    ]


def test_cheapest_plans_compute_the_same_tensor(ctx):
    n, t = 4096, 64
    w = workloads.gnn_chain(seed=3, n=n, degree=8, device="cpu")
    nt = -(-n // t)
    bounds = {"f": 128, "a": nt, "b": t, "c": nt, "d": t, "g": 128}
    verts = _chain_tree(w)
    stored = {0: (gpu_rel(ctx, w["X"]), "a"), 1: (gpu_rel(ctx, w["Y"]), "ac"), 3: (gpu_rel(ctx, w["Z"]), "")}
    # statistics measured on the GPU, per label in each tensor's label order
    for i, (rel, up) in stored.items():
        T, V = ctx.stats(rel)
        lab = verts[i]["labels"]
        order = [c for c in lab if c in up] + [c for c in lab if c not in up]
        verts[i].update(T=T, V=dict(zip(order, V)))
    cm = {"xfer": 1 / 6.7e12, "flop": 1 / 1.0e15, "add": 0.0, "fixed": 2e-9, "max_call_bytes": 256e3}
    plans = plan(verts, bounds, cm, k=4)
    assert len(plans) == 4 and plans[0][0] <= plans[-1][0]
    # the dense definition, from the same bf16 inputs
    X = recompose(w["X"][0], w["X"][2].to(torch.float64).numpy(), "fab", {"a"}, bounds)
    Y = recompose(w["Y"][0], w["Y"][2].to(torch.float64).numpy(), "abcd", {"a", "c"}, bounds)
    Z = w["Z"][2][0].to(torch.float64).numpy()
    g = [P.Vertex("fab"), P.Vertex("abcd"), P.Vertex("cdf", 4, 0, 1), P.Vertex("fg"), P.Vertex("cdg", 4, 2, 3)]
    ref = P.dense_tree(g, {0: X, 1: Y, 3: Z})[4]
    absb = P.dense_tree(g, {0: np.abs(X), 1: np.abs(Y), 3: np.abs(Z)})[4]
    for cost, ups in plans:
        ins = program.prepare_inputs(ctx, verts, ups, stored)
        out = program.execute(ctx, verts, ups, ins)
        k, tl = out.download()
        got = recompose(k, tl.to(torch.float64).numpy(), "cdg", set(ups[4][0]), bounds)
        err = np.abs(got - ref)
        assert np.all(err <= 3e-5 * absb + 1e-30), (ups, float(err.max()))
        for i, r in ins.items():
            if r is not stored[i][0]:
                r.destroy()
        out.destroy()


def test_dag_plan_with_a_result_read_twice(ctx):
    """Two heads read the message-passing result T: O1 = T Z, O2 = T W.
    ucl_plan_dag decides T in its own tree, each head reads it in the split it
    chose (repartitioned where they differ); both outputs match the dense
    definition."""
    n, t = 4096, 64
    w = workloads.gnn_chain(seed=4, n=n, degree=8, device="cpu")
    nt = -(-n // t)
    bounds = {"f": 128, "a": nt, "b": t, "c": nt, "d": t, "g": 128, "h": 16}
    gen = torch.Generator().manual_seed(11)
    Wt = (torch.randn((1, 128, 16), generator=gen) * 0.1).to(torch.bfloat16)
    Wrel = (np.zeros((1, 0), dtype=np.int32), (), Wt)
    verts = _chain_tree(w) + [{"labels": "fh"}, {"labels": "cdh", "left": 2, "right": 5, "dtype_bytes": 4}]
    stored = {0: (gpu_rel(ctx, w["X"]), "a"), 1: (gpu_rel(ctx, w["Y"]), "ac"), 3: (gpu_rel(ctx, w["Z"]), ""),
              5: (gpu_rel(ctx, Wrel), "")}
    for i, (rel, up) in stored.items():
        T, V = ctx.stats(rel)
        lab = verts[i]["labels"]
        order = [c for c in lab if c in up] + [c for c in lab if c not in up]
        verts[i].update(T=T, V=dict(zip(order, V)))
    cm = {"xfer": 1 / 6.7e12, "flop": 1 / 1.0e15, "add": 0.0, "fixed": 2e-9, "max_call_bytes": 256e3}
    cost, ups, roots = plan_dag(verts, bounds, cm)
    assert roots == [-1, -1, 2, -1, 4, -1, 6] and cost > 0
    X = recompose(w["X"][0], w["X"][2].to(torch.float64).numpy(), "fab", {"a"}, bounds)
    Y = recompose(w["Y"][0], w["Y"][2].to(torch.float64).numpy(), "abcd", {"a", "c"}, bounds)
    Z = w["Z"][2][0].to(torch.float64).numpy()
    Wd = Wt[0].to(torch.float64).numpy()
    Td, Ta = np.einsum("fab,abcd->cdf", X, Y), np.einsum("fab,abcd->cdf", np.abs(X), np.abs(Y))
    ref = {4: (np.einsum("cdf,fg->cdg", Td, Z), np.einsum("cdf,fg->cdg", Ta, np.abs(Z))),
           6: (np.einsum("cdf,fh->cdh", Td, Wd), np.einsum("cdf,fh->cdh", Ta, np.abs(Wd)))}
    ins = program.prepare_inputs(ctx, verts, ups, stored)
    outs = program.execute_dag(ctx, verts, ups, ins)
    assert sorted(outs) == [4, 6]
    for i, r in outs.items():
        k, tl = r.download()
        got = recompose(k, tl.to(torch.float64).numpy(), verts[i]["labels"], set(ups[i][0]), bounds)
        want, mag = ref[i]
        err = np.abs(got - want)
        assert np.all(err <= 3e-5 * mag + 1e-30), (i, ups, float(err.max()))
        r.destroy()
    for i, r in ins.items():
        if r is not stored[i][0]:
            r.destroy()
