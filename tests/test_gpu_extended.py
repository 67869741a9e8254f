"""GPU parity of the extended EinSum (Sec. 3: aggregate MAX / MIN / SUM of
map(comb(u, v))) against the oracle, softmax as four chained EinSums, and
the sparse-attention chain of the paper's graph-transformer experiment."""
import zlib

import numpy as np
import pytest
import torch

import workloads
from paper_2603_08957_gb300 import Context, UclError
from tests.parity import assert_parity, gpu_rel, oracle_ref
from tests.ucl_testutil import decompose, random_sparse, ucl_operand

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    c = Context(0)
    yield c
    c.close()


def _exact(a, dtype):
    return torch.from_numpy(np.asarray(a, dtype=np.float64)).to(dtype)


def _rels(dense_ops, labels, ups, dtype, rng, shuffle=False, divisor=None):
    """Relations of dense operands under the given promotions.  `divisor`
    (an operand index): give every entry of that operand's stored tiles a
    magnitude of at least 0.5, so that no quotient divides by zero."""
    out = []
    for q, (d, l, u) in enumerate(zip(dense_ops, labels, ups)):
        k, b, t = decompose(d, l, set(u))
        if q == divisor:
            t = np.where(t == 0, 0.75, np.sign(t) * (0.5 + np.abs(t)))
        if shuffle and len(k) > 1:
            p = rng.permutation(len(k))
            k, t = k[p], t[p]
        out.append((k.astype(np.int32), tuple(int(x) for x in b), _exact(t, dtype)))
    return out


EXT_CASES = [
    # (agg, comb, map)
    ("max", "sub", "square"),      # Sec. 3's example
    ("min", "mul", "ident"),
    ("max", "add", "relu"),
    ("sum", "sub", "exp"),
    ("sum", "add", "ident"),
    ("sum", "div", "ident"),       # every divisor in a stored tile has |v| >= 0.5
    ("sum", "div0", "ident"),      # zero divisors kept: inf / NaN entries matched exactly
    ("max", "mul", "exp"),
]

SPLITS = [("ij", "jk", "ik", {"i"}, {"j"}),        # (labels U, V, W, up U, up V)
          ("ij", "jk", "ik", {"i", "j"}, {"j", "k"}),
          ("ij", "jk", "ik", set(), set()),
          ("ij", "jk", "ik", {"j"}, {"j"})]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("agg,comb,mp", EXT_CASES)
@pytest.mark.parametrize("lu,lv,lw,uu,uv", SPLITS)
def test_extended_binary_matches_oracle(ctx, lu, lv, lw, uu, uv, agg, comb, mp, dtype):
    rng = np.random.default_rng(zlib.crc32(repr((agg, comb, mp, lu, sorted(uu), sorted(uv))).encode()))
    U = random_sparse(rng, (24, 20), density=0.6, block_axes=(0, 1))
    V = random_sparse(rng, (20, 36), density=0.6, block_axes=(0, 1))
    uw = (uu | uv) & set(lw)
    spec = ucl_operand(lu, uu) + "," + ucl_operand(lv, uv) + "->" + ucl_operand(lw, uw)
    rels = _rels([U, V], [lu, lv], [uu, uv], dtype, rng, shuffle=True, divisor=1 if comb == "div" else None)
    op = "div" if comb == "div0" else comb
    out = ctx.einsum(spec, gpu_rel(ctx, rels[0]), gpu_rel(ctx, rels[1]), agg=agg, comb=op, map=mp)
    assert ctx.last_stats()["path"] == "simt"
    ref = oracle_ref(spec, rels, agg=agg, comb=op, map=mp)
    assert_parity(out, ref, dtype)
    fin = np.isfinite(ref["out"])
    if comb == "div":
        assert fin.all()
    elif comb == "div0" and not uv & {"j", "k"}:
        # V's tiles hold zeros along the contracted j: the exact inf / NaN
        # pattern was compared above
        assert not fin.all()


@pytest.mark.parametrize("agg", ["max", "min", "sum"])
@pytest.mark.parametrize("mp", ["ident", "relu", "exp", "square"])
def test_extended_unary_matches_oracle(ctx, agg, mp):
    rng = np.random.default_rng(7)
    A = random_sparse(rng, (30, 40, 8), density=0.5, block_axes=(0, 1))
    rels = _rels([A], ["ijk"], [{"i", "j"}], torch.float32, rng)
    for spec in ("IJk->I", "IJk->Ik", "IJk->IJ"):
        out = ctx.einsum(spec, gpu_rel(ctx, rels[0]), agg=agg, map=mp, scale=0.5)
        ref = oracle_ref(spec, rels, agg=agg, map=mp, scale=0.5)
        assert_parity(out, ref, torch.float32, scale=0.5)


def test_extended_max_split_across_units(ctx):
    """One output key with 200k scalar tuples spans every work unit: the
    fixup folds the units' partials with MAX and MIN."""
    rng = np.random.default_rng(8)
    n = 200_000
    keys = np.stack([np.zeros(n, np.int64), np.arange(n)], axis=1).astype(np.int32)
    keys = np.concatenate([keys, np.array([[1, 0], [1, 5]], np.int32)])
    vals = rng.standard_normal(len(keys)).astype(np.float32)
    rel = (keys, (2, n), torch.from_numpy(vals))
    for agg in ("max", "min"):
        out = ctx.einsum("IJ->I", gpu_rel(ctx, rel), agg=agg)
        assert_parity(out, oracle_ref("IJ->I", [rel], agg=agg), torch.float32)


def test_softmax_chain(ctx):
    """Row softmax of attention scores over the neighbours present, as four
    EinSums; each stage against the oracle fed the GPU's previous output."""
    rng = np.random.default_rng(9)
    S = random_sparse(rng, (300, 500), density=0.05) * 4
    rel = _rels([S], ["ij"], [{"i", "j"}], torch.float32, rng)[0]
    R = gpu_rel(ctx, rel)
    M = ctx.einsum("IJ->I", R, agg="max")
    assert_parity(M, oracle_ref("IJ->I", [rel], agg="max"), torch.float32)
    mk, mt = M.download()
    E = ctx.einsum("IJ,I->IJ", R, M, comb="sub", map="exp")
    mrel = (mk, M.bounds, mt)
    assert_parity(E, oracle_ref("IJ,I->IJ", [rel, mrel], comb="sub", map="exp"), torch.float32)
    ek, et = E.download()
    erel = (ek, E.bounds, et)
    D = ctx.einsum("IJ->I", E)
    assert_parity(D, oracle_ref("IJ->I", [erel]), torch.float32)
    dk, dt = D.download()
    P = ctx.einsum("IJ,I->IJ", E, D, comb="div")
    assert_parity(P, oracle_ref("IJ,I->IJ", [erel, (dk, D.bounds, dt)], comb="div"), torch.float32)
    # every row of present entries sums to 1
    pk, pt = P.download()
    sums = np.bincount(pk[:, 0], weights=pt.numpy().astype(np.float64))
    assert np.allclose(sums[np.unique(pk[:, 0])], 1.0, atol=1e-5)


def test_extended_errors(ctx):
    rel = (np.zeros((1, 0), np.int32), (), torch.ones((1, 4, 4)))
    R = gpu_rel(ctx, rel)
    with pytest.raises(UclError, match="UNSUPPORTED"):
        ctx.einsum("ij,jk->ik", R, R, agg="max", path="tc")
    with pytest.raises(UclError, match="UNSUPPORTED"):
        ctx.einsum("ij,jk,kl->il", R, R, R, agg="max")
    from paper_2603_08957_gb300 import _lib
    import ctypes
    bad = _lib.EinsumOpts(1, 0, 1.0, 0, 7, 0, 0)
    arr = (ctypes.c_void_p * 2)(R.handle, R.handle)
    h = ctypes.c_void_p()
    assert ctx.lib.ucl_einsum(ctx.handle, b"ij,jk->ik", 2, arr, ctypes.byref(bad), ctypes.byref(h)) == 1


def test_attention_chain_small(ctx):
    """The sparse-attention chain of the graph-transformer experiment at a
    reduced size, stage by stage against the oracle."""
    w = workloads.graph_attention(seed=2, n=400, feat=300, feat_nnz=12, edges=2000, dk=64, device="cpu")
    env = {k: gpu_rel(ctx, w[k]) for k in ("XQ", "XK", "WQ", "WK", "A")}
    host = {k: w[k] for k in ("XQ", "XK", "WQ", "WK", "A")}
    for name, spec, ins, opts in w["chain"]:
        out = ctx.einsum(spec, *[env[i] for i in ins], **opts)
        ref_opts = {k: v for k, v in opts.items() if k in ("agg", "comb", "map", "scale", "epi")}
        ref = oracle_ref(spec, [host[i] for i in ins], **ref_opts)
        in_dt = torch.bfloat16 if any(host[i][2].dtype == torch.bfloat16 for i in ins) else torch.float32
        assert_parity(out, ref, in_dt, scale=opts.get("scale", 1.0))
        k, t = out.download()
        env[name], host[name] = out, (k, out.bounds, t)
