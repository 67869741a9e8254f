"""GPU parity: the executor (through the C ABI) against the CPU oracle on the
same seeded inputs.  Every test here needs a GB300 and the built library."""
import itertools
import os

import numpy as np
import pytest
import torch

import oracle
import workloads
from paper_2603_08957_gb300 import Context, UclError
from tests.parity import assert_parity, gpu_rel, oracle_parallel, oracle_ref
from tests.ucl_testutil import decompose, golden, random_sparse, ucl_operand

pytestmark = pytest.mark.gpu

GOLD = golden(os.path.join(os.path.dirname(__file__), "golden", "worked_example.txt"))


@pytest.fixture(scope="module")
def ctx():
    c = Context(0)
    yield c
    c.close()


@pytest.fixture(scope="module")
def ctx_even():
    """A context that always splits pair lists evenly into work units, so
    that even small lists have segments spanning units (partials + fixup)."""
    old = os.environ.get("UCL_SEG_UNITS")
    os.environ["UCL_SEG_UNITS"] = "0"
    try:
        c = Context(0)
    finally:
        if old is None:
            del os.environ["UCL_SEG_UNITS"]
        else:
            os.environ["UCL_SEG_UNITS"] = old
    yield c
    c.close()


def _bf16_exact(a):
    """Round a float64 array to bf16 values (both sides then see the same inputs)."""
    return torch.from_numpy(np.asarray(a)).to(torch.bfloat16).to(torch.float64).numpy()


# ------------------------------------------------------ paper's worked example


@pytest.mark.parametrize("path", ["simt", "auto"])
def test_worked_example(ctx, path):
    U, V = GOLD["U"], GOLD["V"]
    relU = (np.array([[0], [2]], np.int32), (4,), torch.tensor(U[[0, 2]], dtype=torch.float32))
    relV = (np.array([[0], [2]], np.int32), (4,), torch.tensor(V[:, [0, 2]].T.copy(), dtype=torch.float32))
    out = ctx.einsum("Ij,jK->IK", gpu_rel(ctx, relU), gpu_rel(ctx, relV), path=path)
    keys, tiles = out.download()
    want = GOLD["W_scalars"]
    assert keys.tolist() == want[:, :2].astype(int).tolist()
    np.testing.assert_allclose(tiles.numpy(), want[:, 2], rtol=1e-6)
    assert ctx.last_stats()["n_pairs"] == 4
    vt = GOLD["V_relational_tuples"]
    relU2 = (np.arange(4, dtype=np.int32)[:, None], (4,), torch.tensor(U.T.copy(), dtype=torch.float32))
    relV2 = (vt[:, :2].astype(np.int32), (4, 4), torch.tensor(vt[:, 2], dtype=torch.float32))
    out = ctx.einsum("iJ,JK->iK", gpu_rel(ctx, relU2), gpu_rel(ctx, relV2), path=path)
    keys, tiles = out.download()
    want = GOLD["W_colvec"]
    assert keys[:, 0].tolist() == want[:, 0].astype(int).tolist()
    np.testing.assert_allclose(tiles.numpy(), want[:, 1:], rtol=1e-6, atol=1e-7)
    assert ctx.last_stats()["n_pairs"] == 6


# ------------------------------------------------- tcgen05 operand layouts

TC_CASES = [
    # (U operand, V operand, output, extents)  U/V tiles in every major order
    ("IJmk", "JKkn", "IKmn", {"m": 128, "k": 64, "n": 64}),    # A K-major, B MN-major
    ("IJmk", "JKnk", "IKmn", {"m": 128, "k": 64, "n": 64}),    # B K-major
    ("IJkm", "JKkn", "IKmn", {"m": 128, "k": 64, "n": 64}),    # A MN-major
    ("IJkm", "JKnk", "IKnm", {"m": 128, "k": 64, "n": 64}),    # both MN/K swapped, transposed output
    ("IJmk", "JKkn", "IKmn", {"m": 128, "k": 16, "n": 16}),    # 32-byte swizzle
    ("IJmk", "JKkn", "IKnm", {"m": 128, "k": 32, "n": 32}),    # 64-byte swizzle
    ("IJmk", "JKkn", "IKmn", {"m": 128, "k": 128, "n": 128}),  # two boxes per row
    ("IJkm", "JKkn", "IKmn", {"m": 128, "k": 128, "n": 256}),  # N = 256
    ("IJmk", "JKkn", "IKmn", {"m": 256, "k": 64, "n": 64}),    # two M blocks
    ("IJkm", "JKkn", "IKnm", {"m": 256, "k": 64, "n": 32}),    # two M blocks, MN-major A
    ("IJnk", "JKmk", "IKnm", {"m": 128, "k": 64, "n": 48}),    # A comes from V
    ("IJkm", "JKkn", "IKmn", {"m": 256, "k": 256, "n": 64}),   # K chunks, MN-major A (row ranges)
    ("IJmk", "JKnk", "IKmn", {"m": 256, "k": 256, "n": 128}),  # K chunks, K-major A and B (column ranges)
    ("IJmk", "JKkn", "IKnm", {"m": 128, "k": 128, "n": 256}),  # K chunks, transposed output
]


@pytest.mark.parametrize("ou,ov,ow,ext", TC_CASES)
def test_tc_gemm_layouts(ctx_even, ou, ov, ow, ext):
    """Block-sparse tiled matmul whose tile kernel is a bf16 GEMM in every
    operand major order, output transpose and swizzle width: 3 x 40 x 2 key
    grid, 240 pairs over 6 output keys (segments split across work units)."""
    ctx = ctx_even
    rng = np.random.default_rng(hash((ou, ov, ow)) % 2**31)
    nI, nJ, nK = 3, 40, 2

    def rel(op, keys, bounds):
        shape = [ext[c] for c in op if c.islower()]
        t = torch.randn([len(keys)] + shape, generator=torch.Generator().manual_seed(int(rng.integers(1 << 30))))
        return (np.array(keys, np.int32), bounds, t.to(torch.bfloat16))

    U = rel(ou, [(i, j) for i in range(nI) for j in range(nJ)], (nI, nJ))
    V = rel(ov, [(j, k) for j in range(nJ) for k in range(nK)], (nJ, nK))
    spec = f"{ou},{ov}->{ow}"
    ref = oracle_ref(spec, [U, V])
    out = ctx.einsum(spec, gpu_rel(ctx, U), gpu_rel(ctx, V), path="tc")
    assert ctx.last_stats()["path"] == "tc"
    assert_parity(out, ref, torch.bfloat16)
    out16 = ctx.einsum(spec, gpu_rel(ctx, U), gpu_rel(ctx, V), path="tc", out_dtype="bf16", epi="relu", scale=2.0)
    ref16 = oracle_ref(spec, [U, V], epi="relu", scale=2.0)
    assert_parity(out16, ref16, torch.bfloat16, scale=2.0)


# ---------------------------------------------------------- random small specs

SPECS = [
    ("ij,jk->ik", {"i": 5, "j": 7, "k": 6}),
    ("ij,jk->ki", {"i": 4, "j": 3, "k": 5}),
    ("ijb,jbk->ik", {"i": 3, "j": 4, "b": 2, "k": 5}),
    ("bij,bjk->bik", {"b": 3, "i": 4, "j": 5, "k": 2}),
    ("ij,j->i", {"i": 6, "j": 5}),
    ("i,j->ij", {"i": 5, "j": 4}),
    ("ij,ij->i", {"i": 5, "j": 3}),
    ("ijk->ki", {"i": 3, "j": 4, "k": 5}),
    ("ijk,jr,kr->ir", {"i": 3, "j": 4, "k": 2, "r": 5}),   # MTTKRP: star join
    ("ij,jk,kl->il", {"i": 3, "j": 4, "k": 3, "l": 2}),    # chain: C joins through B
    ("i,j,k->ijk", {"i": 3, "j": 2, "k": 4}),               # no shared labels: cross products
]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("spec,ext", SPECS)
def test_random_splits(ctx, spec, ext, dtype):
    rng = np.random.default_rng(abs(hash(spec)) % 2**31)
    lhs, out = spec.split("->")
    ops = lhs.split(",")
    arrs = [random_sparse(rng, [ext[c] for c in op], density=0.6, block_axes=range(len(op))) for op in ops]
    if dtype == torch.bfloat16:
        arrs = [_bf16_exact(a) for a in arrs]
    labels = sorted(ext)
    subsets = [set(s) for k in range(len(labels) + 1) for s in itertools.combinations(labels, k)]
    for promoted in subsets:
        rels = [decompose(a, op, promoted) for op, a in zip(ops, arrs)]
        rels = [(k, tuple(b), torch.from_numpy(t).to(dtype)) for k, b, t in rels]
        uspec = ",".join(ucl_operand(op, promoted) for op in ops) + "->" + ucl_operand(out, promoted)
        ref = oracle_ref(uspec, rels)
        got = ctx.einsum(uspec, *[gpu_rel(ctx, r) for r in rels])
        assert_parity(got, ref, dtype)


# ------------------------------------------------------------------ workloads


def test_blocksparse_fp32_full(ctx):
    """Block-sparse fp32 matmul, 1024 x 1024 at 10% tile density times a dense
    1024 x 256, 32 x 32 tiles, seed 0: the whole output checked."""
    w = workloads.blocksparse_matmul(seed=0)
    ref = oracle_ref(w["spec"], [w["A"], w["B"]])
    out = ctx.einsum(w["spec"], gpu_rel(ctx, w["A"]), gpu_rel(ctx, w["B"]))
    assert_parity(out, ref, torch.float32)
    st = ctx.last_stats()
    assert st["n_pairs"] == ref["n_pairs"] == 102 * 8


def test_blocksparse_fp32_unsorted_inputs(ctx):
    """Same workload with the tuples of both inputs shuffled: the sort path."""
    w = workloads.blocksparse_matmul(seed=1)
    rng = np.random.default_rng(0)
    shuf = []
    for k, b, t in (w["A"], w["B"]):
        p = rng.permutation(len(k))
        shuf.append((k[p], b, t[torch.from_numpy(p)]))
    ref = oracle_ref(w["spec"], shuf)
    out = ctx.einsum(w["spec"], gpu_rel(ctx, shuf[0]), gpu_rel(ctx, shuf[1]))
    assert_parity(out, ref, torch.float32)


@pytest.mark.parametrize("path", ["simt", "auto"])
def test_gnn_chain_small(ctx, path):
    """(X x Y)^T x Z on a 4096-vertex R-MAT graph, 64 x 64 tiles, bf16:
    stage-local parity for both steps (the second step's oracle input is the
    GPU's first-step output)."""
    w = workloads.gnn_chain(seed=3, n=4096, degree=16)
    X, Y, Z = (gpu_rel(ctx, w[k]) for k in ("X", "Y", "Z"))
    T = ctx.einsum(w["spec1"], X, Y, out_dtype="bf16", path=path)
    ref1 = oracle_ref(w["spec1"], [w["X"], w["Y"]])
    assert_parity(T, ref1, torch.bfloat16)
    keys_t, tiles_t = T.download()
    out = ctx.einsum(w["spec2"], T, Z, path=path)
    ref2 = oracle_ref(w["spec2"], [(keys_t, T.bounds, tiles_t), w["Z"]])
    assert_parity(out, ref2, torch.bfloat16)


@pytest.mark.parametrize("bands", [2, 4, 16])
def test_banded_message_passing(monkeypatch, bands):
    """Banding of the contracted label (forced): the message passing of a
    4096-vertex R-MAT graph with 128-wide embeddings, its pairs contracted
    band after band into fp32 (band, K) partials and summed per K in band
    order.  Both layers' EinSums against the oracle, every output key."""
    monkeypatch.setenv("UCL_BANDS", str(bands))
    c = Context(0)
    monkeypatch.delenv("UCL_BANDS")
    w = workloads.gnn_two_layer(seed=4, n=4096, n_edges=20_000, feat=128, device="cuda")
    X, Y = gpu_rel(c, w["X"]), gpu_rel(c, w["Y"])
    T1 = c.einsum(w["spec1"], X, Y, out_dtype="bf16")
    st = c.last_stats()
    assert st["n_bands"] == bands and st["path"] == "tc"
    assert st["n_band_segments"] > st["n_segments"]
    host = {k: (w[k][0], w[k][1], w[k][2].cpu()) for k in ("X", "Y")}
    assert_parity(T1, oracle_ref(w["spec1"], [host["X"], host["Y"]]), torch.bfloat16)
    # the second message passing reads T1 keyed by the source block
    k1, t1 = T1.download()
    T2 = c.einsum(w["spec3"], T1, Y, out_dtype="f32")
    assert c.last_stats()["n_bands"] == bands
    assert_parity(T2, oracle_ref(w["spec3"], [(k1, T1.bounds, t1), host["Y"]]), torch.bfloat16)
    for r in (X, Y, T1, T2):
        r.destroy()
    c.close()


@pytest.mark.parametrize("window,bands", [(1, 0), (2, 0), (3, 0), (2, 4), (1, 2)])
def test_windowed_message_passing(monkeypatch, window, bands):
    """Windows of 2^w consecutive output keys (forced): pairs ordered by
    (band, K >> w, X tuple), accumulated per key slot in one TMEM buffer, an
    X tile loaded once per run of pairs that read it.  Both message-passing
    EinSums of a small two-layer GNN against the oracle, every output key,
    with units small enough that windows straddle CTAs (partials + fixup)."""
    monkeypatch.setenv("UCL_WINDOW", str(window))
    monkeypatch.setenv("UCL_BANDS", str(bands))
    c = Context(0)
    monkeypatch.delenv("UCL_WINDOW")
    monkeypatch.delenv("UCL_BANDS")
    feat = 128 if window == 3 else 256
    w = workloads.gnn_two_layer(seed=7, n=3000, n_edges=30_000, feat=feat, device="cuda")
    X, Y = gpu_rel(c, w["X"]), gpu_rel(c, w["Y"])
    T1 = c.einsum(w["spec1"], X, Y, out_dtype="bf16")
    st = c.last_stats()
    assert st["path"] == "tc" and st["n_bands"] == max(bands, 1)
    host = {k: (w[k][0], w[k][1], w[k][2].cpu()) for k in ("X", "Y")}
    assert_parity(T1, oracle_ref(w["spec1"], [host["X"], host["Y"]]), torch.bfloat16)
    k1, t1 = T1.download()
    T2 = c.einsum(w["spec3"], T1, Y, out_dtype="f32")
    assert_parity(T2, oracle_ref(w["spec3"], [(k1, T1.bounds, t1), host["Y"]]), torch.bfloat16)
    # the same EinSum without windows: the same key set
    c2 = Context(0)
    T3 = c2.einsum(w["spec1"], gpu_rel(c2, w["X"]), gpu_rel(c2, w["Y"]), out_dtype="bf16")
    assert np.array_equal(T3.download()[0], k1)
    for r in (X, Y, T1, T2):
        r.destroy()
    c.close()


def test_windowed_gnn_full_size_sampled(monkeypatch):
    """The full message-passing EinSum (100000 vertices, 358k Y tiles) with
    windows of 4 keys (forced): every output key, values on sampled keys."""
    monkeypatch.setenv("UCL_WINDOW", "2")
    c = Context(0)
    monkeypatch.delenv("UCL_WINDOW")
    w = workloads.gnn_chain(seed=0, n=100_000)
    X, Y = gpu_rel(c, w["X"]), gpu_rel(c, w["Y"])
    T = c.einsum(w["spec1"], X, Y, out_dtype="bf16")
    ky = w["Y"][0]
    kt = T.download()[0]
    assert np.array_equal(kt, np.unique(ky[:, 1]).astype(np.int32)[:, None])
    cnt = np.bincount(ky[:, 1])
    big = int(np.searchsorted(kt[:, 0], int(np.argmax(cnt))))
    sk = kt[_sample_rows(len(kt), 12, seed=4, must=[big]), 0]
    yk = ky[np.isin(ky[:, 1], sk)]
    rows = np.nonzero(np.isin(ky[:, 1], sk))[0]
    yrel = (yk, w["Y"][1], w["Y"][2][torch.as_tensor(rows)])
    jn = np.unique(yk[:, 0])
    xrel = (jn[:, None].astype(np.int32), w["X"][1], w["X"][2][torch.as_tensor(jn)])
    ref = oracle_ref(w["spec1"], [xrel, yrel], sample_keys=sk[:, None])
    assert_parity(T, ref, torch.bfloat16, select=np.searchsorted(kt[:, 0], sk))
    for r in (X, Y, T):
        r.destroy()
    c.close()


def test_l2_hints_do_not_change_results(monkeypatch):
    """L2 eviction hints on the TMA loads change where lines live, never the
    arithmetic: results with and without them are bit-identical."""
    w = workloads.gnn_chain(seed=5, n=30000, degree=16)
    outs = []
    for hints in ("1", "0"):
        monkeypatch.setenv("UCL_L2_HINTS", hints)
        c = Context(0)
        X, Y = gpu_rel(c, w["X"]), gpu_rel(c, w["Y"])
        T = c.einsum(w["spec1"], X, Y, out_dtype="bf16")
        outs.append(T.download())
        for r in (X, Y, T):
            r.destroy()
        c.close()
    assert np.array_equal(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1], outs[1][1])


@pytest.mark.parametrize("na,nb", [(32, 32), (33, 32), (100, 100), (256, 2), (257, 2)])
def test_small_key_stage_and_fallback(ctx, na, nb):
    """Small binary EinSums run their whole key stage in one CTA (at most
    256 tuples per input, 1024 pairs); a cross product just past 1024 pairs,
    or an input past 256 tuples, takes the general path.  Both against the
    oracle; the small path launches far fewer kernels."""
    rng = np.random.default_rng(na * 7 + nb)
    a = (np.arange(na, dtype=np.int32)[:, None], (na,), torch.from_numpy(rng.standard_normal((na, 4))).float())
    b = (np.arange(nb, dtype=np.int32)[:, None], (nb,), torch.from_numpy(rng.standard_normal((nb, 4))).float())
    out = ctx.einsum("Ii,Ki->IK", gpu_rel(ctx, a), gpu_rel(ctx, b))
    st = ctx.last_stats()
    assert_parity(out, oracle_ref("Ii,Ki->IK", [a, b]), torch.float32)
    small = na * nb <= 1024 and na <= 256 and nb <= 256
    assert (st["launches"] <= 4) == small, st
    # a join on a shared label, inputs shuffled
    pa, pb = rng.permutation(na), rng.permutation(nb)
    ka = np.stack([np.arange(na) % 7, np.arange(na)], 1).astype(np.int32)[pa]
    kb = np.stack([np.arange(nb) % 7, np.arange(nb)], 1).astype(np.int32)[pb]
    ra = (ka, (7, na), torch.from_numpy(rng.standard_normal((na, 3, 2))).float())
    rb = (kb, (7, nb), torch.from_numpy(rng.standard_normal((nb, 3))).float())
    out = ctx.einsum("JIij,JKi->IKj", gpu_rel(ctx, ra), gpu_rel(ctx, rb))
    assert_parity(out, oracle_ref("JIij,JKi->IKj", [ra, rb]), torch.float32)


def test_spgemm_small(ctx):
    """Block-sparse x block-sparse, 128 x 128 bf16 tiles, band + uniform, fp32 out."""
    w = workloads.spgemm(seed=2, n=8192, density=0.05)
    ref = oracle_ref(w["spec"], [w["A"], w["B"]])
    out = ctx.einsum(w["spec"], gpu_rel(ctx, w["A"]), gpu_rel(ctx, w["B"]))
    assert_parity(out, ref, torch.bfloat16)


def _sample_rows(n, k, seed, must=()):
    rng = np.random.default_rng(seed)
    pick = set(rng.choice(n, size=min(k, n), replace=False).tolist()) | set(int(m) for m in must)
    return np.array(sorted(pick))


def test_gnn_full_size_sampled(ctx):
    """The full message-passing workload (100000 vertices, 1.6M R-MAT edges,
    358k Y tiles): every output key checked, values checked on sampled keys
    (including the largest segment) against the oracle with all their pairs."""
    w = workloads.gnn_chain(seed=0, device="cuda")
    X, Y, Z = (gpu_rel(ctx, w[k]) for k in ("X", "Y", "Z"))
    T = ctx.einsum(w["spec1"], X, Y, out_dtype="bf16")
    keys_t, _ = T.download()
    ky = w["Y"][0]
    want_keys = np.unique(ky[:, 1])[:, None].astype(np.int32)
    assert np.array_equal(keys_t, want_keys)
    biggest = np.argmax(np.bincount(ky[:, 1]))
    sel = _sample_rows(len(keys_t), 24, 0, must=[int(np.searchsorted(want_keys[:, 0], biggest))])
    sk = keys_t[sel]
    ysel = np.isin(ky[:, 1], sk[:, 0])
    yk = ky[ysel]
    yt = workloads.adjacency_tiles_subset(w["edges"][0], w["edges"][1], w["n"], w["t"], yk)
    ref = oracle_ref(w["spec1"], [w["X"], (yk, w["Y"][1], yt)], sample_keys=sk)
    assert_parity(T, ref, torch.bfloat16, select=sel)


def test_spgemm_full_size_sampled(ctx):
    w = workloads.spgemm(seed=0)
    out = ctx.einsum(w["spec"], gpu_rel(ctx, w["A"]), gpu_rel(ctx, w["B"]))
    keys, _ = out.download()
    ka, kb = w["A"][0], w["B"][0]
    # full key set: (I, K) for every A(I, J), B(J, K)
    want = set()
    byJ = {}
    for J, K in kb:
        byJ.setdefault(int(J), []).append(int(K))
    for I, J in ka:
        for K in byJ.get(int(J), []):
            want.add((int(I), K))
    assert keys.tolist() == [list(k) for k in sorted(want)]
    sel = _sample_rows(len(keys), 32, 1)
    ref = oracle_ref(w["spec"], [w["A"], w["B"]], sample_keys=keys[sel])
    assert_parity(out, ref, torch.bfloat16, select=sel)


# ------------------------------------------------------------------ edge cases


def test_empty_relation_and_empty_join(ctx):
    e = (np.zeros((0, 1), np.int32), (4,), torch.zeros((0, 2, 3)))
    f = (np.array([[1]], np.int32), (4,), torch.ones((1, 3, 2)))
    out = ctx.einsum("Jij,Jjk->ik", gpu_rel(ctx, e), gpu_rel(ctx, f))
    assert out.n == 0 and out.shape == (2, 2)
    g = (np.array([[2]], np.int32), (4,), torch.ones((1, 2, 3)))
    out = ctx.einsum("Jij,Jjk->Jik", gpu_rel(ctx, g), gpu_rel(ctx, f))
    assert out.n == 0 and ctx.last_stats()["n_pairs"] == 0


def test_one_segment_across_all_units(ctx_even):
    """All pairs share one output key (a key-less output summed over J): the
    segment is split across every work unit and reassembled by the fixup."""
    ctx = ctx_even
    rng = np.random.default_rng(4)
    nJ = 3000
    ka = np.arange(nJ, dtype=np.int32)[:, None]
    A = (ka, (nJ,), torch.from_numpy(rng.standard_normal((nJ, 8, 5)).astype(np.float32)))
    B = (ka.copy(), (nJ,), torch.from_numpy(rng.standard_normal((nJ, 5, 6)).astype(np.float32)))
    ref = oracle_ref("Jij,Jjk->ik", [A, B])
    out = ctx.einsum("Jij,Jjk->ik", gpu_rel(ctx, A), gpu_rel(ctx, B))
    assert ctx.last_stats()["n_units"] > 1
    assert_parity(out, ref, torch.float32)


@pytest.mark.parametrize("path", ["tc", "simt"])
def test_small_lists_cut_at_segments(ctx, ctx_even, path):
    """On the tcgen05 path small pair lists are cut into work units at
    segment boundaries: no segment spans two units and the fixup moves
    nothing.  The FFMA path keeps the even split.  Both cuts match the
    oracle."""
    rng = np.random.default_rng(21)
    nI, nJ, nK = 12, 30, 5
    keys_u = [(i, j) for i in range(nI) for j in range(nJ) if rng.random() < 0.6]
    keys_v = [(j, k) for j in range(nJ) for k in range(nK) if rng.random() < 0.6]
    U = (np.array(keys_u, np.int32), (nI, nJ), torch.randn((len(keys_u), 128, 64)).to(torch.bfloat16))
    V = (np.array(keys_v, np.int32), (nJ, nK), torch.randn((len(keys_v), 64, 64)).to(torch.bfloat16))
    spec = "IiJj,JjKk->IiKk"
    ref = oracle_ref(spec, [U, V])
    for c, cut in ((ctx, True), (ctx_even, False)):
        c.fixup_bytes(reset=True)
        out = c.einsum(spec, gpu_rel(c, U), gpu_rel(c, V), path=path)
        st = c.last_stats()
        assert st["n_pairs"] == ref["n_pairs"] and st["path"] == path
        assert_parity(out, ref, torch.bfloat16)
        c.synchronize()
        moved = c.fixup_bytes(reset=True)
        if cut and path == "tc":
            assert moved == 0 and st["n_units"] <= st["n_segments"]
        else:
            assert moved > 0


def test_unary_relu_scale_bf16_out(ctx):
    """Unary EinSum (Sec. 3's ReLU as a sum over the empty set, here also
    summing an upper label), scale and relu after the sum, bf16 output."""
    rng = np.random.default_rng(5)
    k = np.array([(i, j) for i in range(6) for j in range(4) if (i + j) % 3], np.int32)
    t = torch.from_numpy(rng.standard_normal((len(k), 3, 7)).astype(np.float32))
    rel = (k, (6, 4), t)
    ref = oracle_ref("IJab->Ib", [rel], epi="relu", scale=0.5)
    out = ctx.einsum("IJab->Ib", gpu_rel(ctx, rel), epi="relu", scale=0.5, out_dtype="bf16")
    assert_parity(out, ref, torch.float32, scale=0.5)


def test_wide_keys_64_bits(ctx):
    """Three key columns of 2^20 values each pack into 60 bits."""
    rng = np.random.default_rng(6)
    n = 500
    kx = np.unique(rng.integers(0, 2**20, size=(n, 3)), axis=0).astype(np.int32)
    ky = kx[rng.permutation(len(kx))[: len(kx) // 2]][:, [1, 2]]
    ky = np.unique(ky, axis=0)
    X = (kx, (2**20,) * 3, torch.from_numpy(rng.standard_normal((len(kx), 4)).astype(np.float32)))
    Y = (ky, (2**20,) * 2, torch.from_numpy(rng.standard_normal((len(ky), 4)).astype(np.float32)))
    ref = oracle_ref("IJKa,JKa->IK", [X, Y])
    out = ctx.einsum("IJKa,JKa->IK", gpu_rel(ctx, X), gpu_rel(ctx, Y))
    assert_parity(out, ref, torch.float32)


def test_host_copy_and_download(ctx):
    w = workloads.blocksparse_matmul(seed=2)
    ka, ba, ta = w["A"]
    A = ctx.relation(torch.from_numpy(ka), ba, ta)           # host tensors -> UCL_MEM_HOST_COPY
    B = ctx.relation(torch.from_numpy(w["B"][0]), w["B"][1], w["B"][2])
    out = ctx.einsum(w["spec"], A, B)
    assert_parity(out, oracle_ref(w["spec"], [w["A"], w["B"]]), torch.float32)
    # the same result downloaded into reused pinned buffers (larger than needed)
    k0, t0 = out.download()
    kb = torch.full((out.n * out.u + 7,), -1, dtype=torch.int32).pin_memory()
    tb = torch.full((t0.numel() + 5,), float("nan"), dtype=torch.float32).pin_memory()
    for _ in range(2):
        k1, t1 = out.download(kb, tb)
        assert np.array_equal(k1, k0) and torch.equal(t1, t0)
    assert np.all(kb[out.n * out.u:].numpy() == -1) and torch.isnan(tb[t0.numel():]).all()
    # copied relations from pinned host memory and from device memory
    ta_p = ta.pin_memory()
    A2 = ctx.relation(torch.from_numpy(ka), ba, ta_p)
    A3 = ctx.relation(torch.from_numpy(ka).cuda(), ba, ta.cuda(), copy=True)
    for R in (A2, A3):
        o = ctx.einsum(w["spec"], R, B)
        k2, t2 = o.download()
        assert np.array_equal(k2, k0) and torch.equal(t2, t0)
    with pytest.raises(ValueError):
        out.download(kb[:1], tb)


def test_deterministic(ctx):
    w = workloads.gnn_chain(seed=5, n=8192, degree=16)
    X, Y = gpu_rel(ctx, w["X"]), gpu_rel(ctx, w["Y"])
    a = ctx.einsum(w["spec1"], X, Y).download()[1]
    b = ctx.einsum(w["spec1"], X, Y).download()[1]
    assert torch.equal(a, b)


# ---------------------------------------------------------------------- errors


def test_errors(ctx):
    v = (np.array([[1]], np.int32), (2,), torch.ones((1, 3)))
    with pytest.raises(UclError, match="UCL_ERR_DUP_KEY"):
        gpu_rel(ctx, (np.array([[0], [1], [0]], np.int32), (2,), torch.ones((3, 3))))
    with pytest.raises(UclError, match="UCL_ERR_KEY_RANGE"):
        gpu_rel(ctx, (np.array([[2]], np.int32), (2,), torch.ones((1, 3))))
    with pytest.raises(UclError, match="UCL_ERR_KEY_RANGE"):
        gpu_rel(ctx, (np.array([[-1]], np.int32), (2,), torch.ones((1, 3))))
    R = gpu_rel(ctx, v)
    with pytest.raises(UclError, match="UCL_ERR_SPEC"):
        ctx.einsum("Ij,jK", R, R)
    with pytest.raises(UclError, match="UCL_ERR_SPEC"):
        ctx.einsum("Ij,jK->IQ", R, R)
    with pytest.raises(UclError, match="UCL_ERR_SHAPE"):
        ctx.einsum("Iij,jK->IK", R, R)
    W = gpu_rel(ctx, (np.array([[1]], np.int32), (2,), torch.ones((1, 4))))
    with pytest.raises(UclError, match="UCL_ERR_SHAPE"):
        ctx.einsum("Ij,jK->IK", R, W)
    # the context stays usable after errors
    out = ctx.einsum("Ij,Ij->I", R, R)
    assert out.download()[1].tolist() == [3.0]
    ctx.synchronize()


def _band_crossings(ky, jext, bands, G):
    """Work-unit boundaries inside each output key's pairs for a message
    passing whose pairs are one per Y tuple (J, K) and are ordered by
    (band of J, K): per band b, G_b = min(P_b, G) units of equal pair count.
    Returns the crossing count of every K (summed over bands)."""
    jb = int(np.ceil(np.log2(jext))) if jext > 1 else 0
    bits = int(np.log2(bands))
    band = ky[:, 0].astype(np.int64) >> (jb - bits) if bits else np.zeros(len(ky), np.int64)
    nk = int(ky[:, 1].max()) + 1
    cross = np.zeros(nk, np.int64)
    base = 0
    for b in range(bands):
        kb = ky[band == b, 1]
        Pb = len(kb)
        if Pb == 0:
            continue
        cnt = np.bincount(kb, minlength=nk)
        pre = base + np.concatenate([[0], np.cumsum(cnt)])[:-1]
        Gb = min(Pb, G)
        starts = [base + Pb * u // Gb for u in range(1, Gb)]
        cross += np.where(cnt > 0, _crossings(pre, pre + cnt, starts), 0)
        base += Pb
    return cross


def test_two_layer_gnn_full_size_sampled(ctx):
    """Two-layer GNN at scale: R-MAT with 2M vertices / 40M drawn edges as
    64x64 0/1 tiles (~16.6M tiles, ~136 GB), 256-wide embeddings, chained
    T1=(XY)^T, H1=relu(T1 W1), T2=(H1 Y)^T, O=T2 W2.  Every step's key set
    is checked in full; values stage-locally on sampled output keys drawn
    over the whole size distribution, always including one whose pairs span
    at least three work units (carried across CTAs by partials and the
    fixup).  The oracle gets exactly the tiles each sampled key joins with,
    one spawned process per key."""
    w = workloads.gnn_two_layer(seed=0)
    dev = torch.device("cuda", 0)
    X, Y, W1, W2 = (gpu_rel(ctx, w[k]) for k in ("X", "Y", "W1", "W2"))
    ky = w["Y"][0]
    want_k = np.unique(ky[:, 1]).astype(np.int32)[:, None]
    src, dst = w["edges"]
    t, n = w["t"], w["n"]
    cnt = np.bincount(ky[:, 1], minlength=want_k.max() + 1)

    def y_subset(kset):
        m = torch.isin(dst // t, torch.as_tensor(kset, device=dst.device, dtype=torch.int64))
        s_, d_ = src[m].cpu().numpy(), dst[m].cpu().numpy()
        yk = ky[np.isin(ky[:, 1], kset)]
        return yk, workloads.adjacency_tiles_subset(s_, d_, n, t, yk)

    def rows(rel, keys_sel):
        k, tl = rel.device_tensors()
        kk = k[:, 0].cpu().numpy()
        idx = np.searchsorted(kk, keys_sel)
        assert np.array_equal(kk[idx], keys_sel)
        return keys_sel[:, None].astype(np.int32), tl[torch.as_tensor(idx, device=tl.device)].cpu()

    # step 1: T1 = (X Y)^T
    T1 = ctx.einsum(w["spec1"], X, Y, out_dtype="bf16")
    st = ctx.last_stats()
    kt1, _ = T1.device_tensors()
    assert np.array_equal(kt1.cpu().numpy(), want_k)
    cross = _band_crossings(ky, w["X"][1][0], st["n_bands"], st["n_units"])
    rng = np.random.default_rng(3)
    present = np.nonzero(cnt > 0)[0]
    picks = set(rng.choice(present, size=3, replace=False).tolist())
    big = np.nonzero(cross >= 2)[0]
    assert len(big) > 0
    kbig = int(big[np.argmin(cnt[big])])
    picks.add(kbig)
    sk = np.array(sorted(picks), dtype=np.int32)
    subsets = {int(k): y_subset(np.array([k])) for k in sk}
    tasks = []
    for k in sk:
        yk, yt = subsets[int(k)]
        jneed = np.unique(yk[:, 0])
        xrel = (jneed[:, None].astype(np.int32), w["X"][1], w["X"][2][torch.as_tensor(jneed, device=dev)].cpu())
        tasks.append((w["spec1"], [xrel, (yk, w["Y"][1], yt)], {"sample_keys": np.array([[k]], np.int32)}))
    kt1h = kt1[:, 0].cpu().numpy()
    for k, ref in zip(sk, oracle_parallel(tasks)):
        assert_parity(T1, ref, torch.bfloat16, select=np.searchsorted(kt1h, [k]))
    sel = np.searchsorted(kt1h, sk)
    # step 2: H1 = relu(T1 W1), stage-local
    H1 = ctx.einsum(w["spec2"], T1, W1, out_dtype="bf16", epi="relu")
    t1k, t1t = rows(T1, sk)
    ref = oracle_ref(w["spec2"], [(t1k, T1.bounds, t1t), w["W1"]], epi="relu")
    assert_parity(H1, ref, torch.bfloat16, select=sel)
    # step 3: T2 = (H1 Y)^T with H1 keyed by J; only K reached from a J that
    # H1 holds (a destination tile of some edge) appear
    T2 = ctx.einsum(w["spec3"], H1, Y, out_dtype="bf16")
    kt2 = T2.device_tensors()[0].cpu().numpy()
    want_k2 = np.unique(ky[np.isin(ky[:, 0], want_k[:, 0]), 1]).astype(np.int32)[:, None]
    assert np.array_equal(kt2, want_k2)
    sk2 = sk[np.isin(sk, kt2[:, 0])]
    assert len(sk2) > 0 and kbig in sk2
    tasks = []
    for k in sk2:
        yk, yt = subsets[int(k)]
        keep = np.isin(yk[:, 0], want_k[:, 0])
        yk2, yt2 = yk[keep], yt[keep]
        hk, ht = rows(H1, np.unique(yk2[:, 0]))
        tasks.append((w["spec3"], [(hk, H1.bounds, ht), (yk2, w["Y"][1], yt2)],
                      {"sample_keys": np.array([[k]], np.int32)}))
    for k, ref in zip(sk2, oracle_parallel(tasks)):
        assert_parity(T2, ref, torch.bfloat16, select=np.searchsorted(kt2[:, 0], [k]))
    sel2 = np.searchsorted(kt2[:, 0], sk2)
    # step 4: O = T2 W2
    O = ctx.einsum(w["spec4"], T2, W2)
    t2k, t2t = rows(T2, sk2)
    ref = oracle_ref(w["spec4"], [(t2k, T2.bounds, t2t), w["W2"]])
    assert_parity(O, ref, torch.bfloat16, select=sel2)
    for r in (X, Y, W1, W2, T1, H1, T2, O):
        r.destroy()
    del w
    torch.cuda.empty_cache()


# ------------------------------------------------------------ three inputs


@pytest.mark.parametrize("path", ["simt", "auto", "tc"])
def test_mttkrp_small(ctx, path):
    """MTTKRP over a 1000^3 Zipf(1.1) tensor with 5000 nonzeros in 16^3 tiles,
    rank 64, bf16: the whole output checked."""
    w = workloads.mttkrp(seed=0, n=1000, nnz=5000)
    ref = oracle_ref(w["spec"], [w["T"], w["B"], w["C"]])
    out = ctx.einsum(w["spec"], *(gpu_rel(ctx, w[k]) for k in ("T", "B", "C")), path=path)
    assert_parity(out, ref, torch.bfloat16)
    assert ctx.last_stats()["n_pairs"] == ref["n_pairs"] == len(w["T"][0])
    assert ctx.last_stats()["path"] == ("simt" if path == "simt" else "tc")
    # operands in another order: the join order is chosen from the keys
    out2 = ctx.einsum("Jjr,IJKijk,Kkr->Iir", *(gpu_rel(ctx, w[k]) for k in ("B", "T", "C")), path=path)
    assert_parity(out2, ref, torch.bfloat16)
    # T tiles stored [k][i][j]: the same EinSum, the same output
    wk = workloads.mttkrp(seed=0, n=1000, nnz=5000, layout="kij")
    out3 = ctx.einsum(wk["spec"], *(gpu_rel(ctx, wk[k]) for k in ("T", "B", "C")), path=path)
    assert_parity(out3, ref, torch.bfloat16)


def _crossings(seg_lo, seg_hi, starts):
    """Unit boundaries strictly inside each pair range [seg_lo, seg_hi)."""
    starts = np.asarray(starts)
    return np.searchsorted(starts, seg_hi, side="left") - np.searchsorted(starts, seg_lo, side="right")


def test_mttkrp_full_size_sampled(ctx):
    """MTTKRP at full size: a 100000^3 tensor with 1e7 Zipf(1.1) nonzeros in
    16^3 tiles (~3.9M tiles, ~32 GB bf16), rank-64 factors.  The whole output
    key set is checked; values on sampled output keys drawn over the whole
    size distribution, always including a key whose triples span at least
    three work units (its sum is carried across CTAs by the partial / fixup
    path).  The oracle gets the T tiles of those keys and the factor tiles
    they join with, one spawned process per key."""
    w = workloads.mttkrp(seed=0, device="cuda")
    dev = torch.device("cuda", 0)
    rels = [gpu_rel(ctx, w[k]) for k in ("T", "B", "C")]
    out = ctx.einsum(w["spec"], *rels)
    st = ctx.last_stats()
    kt = w["T"][0]
    got = out.device_tensors()[0].cpu().numpy()
    assert np.array_equal(got, np.unique(kt[:, 0]).astype(np.int32)[:, None])
    P, G = st["n_pairs"], st["n_units"]
    assert P == len(kt)
    cnt = np.bincount(kt[:, 0])
    # triples are ordered by output key I: key i holds [pre[i], pre[i] + cnt[i])
    pre = np.concatenate([[0], np.cumsum(cnt)])[:-1]
    units = np.array([P * u // G for u in range(1, G)])
    cross = _crossings(pre, pre + cnt, units)
    rng = np.random.default_rng(5)
    present = np.nonzero(cnt > 0)[0]
    picks = set(rng.choice(present, size=4, replace=False).tolist())
    # the smallest key spanning at least three units (oracle time ~ its triples)
    big = np.nonzero(cross >= 2)[0]
    assert len(big) > 0
    kbig = int(big[np.argmin(cnt[big])])
    picks.add(kbig)
    tasks, order = [], sorted(picks)

    def factor_rows(f, rows):
        rows = np.unique(rows)
        return (rows[:, None].astype(np.int32), f[1], f[2][torch.as_tensor(rows, device=dev)].cpu())

    for key in order:
        m = np.nonzero(kt[:, 0] == key)[0]
        tsub = (kt[m], w["T"][1], w["T"][2][torch.as_tensor(m, device=dev)].cpu())
        tasks.append((w["spec"], [tsub, factor_rows(w["B"], kt[m, 1]), factor_rows(w["C"], kt[m, 2])],
                      {"sample_keys": np.array([[key]], np.int32)}))
    refs = oracle_parallel(tasks)
    for key, ref in zip(order, refs):
        assert_parity(out, ref, torch.bfloat16, select=np.searchsorted(got[:, 0], [key]))
    assert cross[kbig] >= 2
    for r in rels + [out]:
        r.destroy()
    del w
    torch.cuda.empty_cache()


TC3_CASES = [
    # (spec, T tile permutation, factor order, E layout [j][r] or [r][j])
    ("IJKijk,Jjr,Kkr->Iir", (0, 1, 2), "BC", "jr"),   # E = B, groups of equal J
    ("IJKijk,Jjr,Kkr->rIi", (0, 1, 2), "BC", "jr"),   # transposed output tile
    ("IJKijk,Kkr,Jjr->Iir", (0, 1, 2), "CB", "jr"),   # first join on K: E changes every triple
    ("IJKikj,Kkr,Jjr->Iir", (0, 2, 1), "CB", "jr"),   # T laid out [i][k][j]: E = C, F = B
    ("IJKijk,Jrj,Kkr->Iir", (0, 1, 2), "BC", "rj"),   # E stored [r][j]
    ("IJKkij,Jjr,Kkr->Iir", (2, 0, 1), "BC", "jr"),   # T laid out [k][i][j]: MN-major T, 128-byte TMA rows
    ("IJKkij,Jjr,Kkr->rIi", (2, 0, 1), "BC", "jr"),   # ... with a transposed output tile
    ("IJKjik,Kkr,Jjr->Iir", (1, 0, 2), "CB", "jr"),   # T laid out [j][i][k]: E = C, F = B
]


@pytest.mark.parametrize("spec,perm,order,elay", TC3_CASES)
def test_tc3_layouts(ctx, spec, perm, order, elay):
    """The tcgen05 MTTKRP path for every operand arrangement it accepts, with
    bf16 / relu / scale epilogues; 2000^3 tensor, 20000 Zipf nonzeros."""
    w = workloads.mttkrp(seed=4, n=2000, nnz=20000)
    kt, bt, tt = w["T"]
    T = (kt, bt, tt.permute(0, *[1 + p for p in perm]).contiguous())
    fac = {"B": w["B"], "C": w["C"]}
    if elay == "rj":
        kb, bb, tb = fac["B"]
        fac["B"] = (kb, bb, tb.transpose(1, 2).contiguous())
    rels = [T, fac[order[0]], fac[order[1]]]
    ref = oracle_ref(spec, rels)
    out = ctx.einsum(spec, *(gpu_rel(ctx, r) for r in rels), path="tc")
    assert ctx.last_stats()["path"] == "tc"
    assert_parity(out, ref, torch.bfloat16)
    ref2 = oracle_ref(spec, rels, epi="relu", scale=0.5)
    out2 = ctx.einsum(spec, *(gpu_rel(ctx, r) for r in rels), path="tc", out_dtype="bf16", epi="relu", scale=0.5)
    assert_parity(out2, ref2, torch.bfloat16, scale=0.5)


# ------------------------------------------------------------ repartition

from oracle.repartition import repartition as oracle_repartition  # noqa: E402

REPART_CASES = [
    # (dense labels, extents, upper labels of the input, output side of the spec)
    ("ij", {"i": 5, "j": 4}, {"i"}, "iJ"),                     # rows -> columns
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"i"}, "IjK"),            # decompose only
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"i", "j"}, "iJk"),       # stack only
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"j", "k"}, "Ijk"),       # both
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"i"}, "Ikj"),            # tile dims reordered
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"j", "k"}, "KiJ"),       # promoted label between kept ones
    ("ijk", {"i": 3, "j": 4, "k": 2}, set(), "IJK"),            # one dense tuple -> scalars
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"i", "j", "k"}, "kji"),  # scalars -> one dense tuple
    ("ijkl", {"i": 70, "j": 3, "k": 40, "l": 5}, {"i", "k"}, "KjIl"),   # several tiles' worth of keys
]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("labels,ext,src,rhs", REPART_CASES)
def test_repartition_matches_oracle(ctx, labels, ext, src, rhs, dtype):
    """Every output key and value bit-exact against the oracle (values are
    copies), with the input's tuples in key order and shuffled."""
    rng = np.random.default_rng(abs(hash((labels, rhs))) % 2**31)
    dense = random_sparse(rng, [ext[c] for c in labels], density=0.4, block_axes=range(len(labels)))
    # the oracle sees exactly the values the GPU holds
    dense = _bf16_exact(dense) if dtype == torch.bfloat16 else dense.astype(np.float32).astype(np.float64)
    keys, bounds, tiles = decompose(dense, labels, src)
    lhs = "".join(c.upper() for c in labels if c in src) + "".join(c for c in labels if c not in src)
    spec = lhs + "->" + rhs
    want_k, want_b, want_t = oracle_repartition(spec, (keys, bounds, tiles))
    perm = rng.permutation(len(keys))
    for k, t in ((keys, tiles), (keys[perm], tiles[perm])):
        rel = gpu_rel(ctx, (k.astype(np.int32), tuple(int(b) for b in bounds), torch.from_numpy(t).to(dtype)))
        out = ctx.repartition(spec, rel)
        gk, gt = out.download()
        assert out.bounds == tuple(want_b)
        assert np.array_equal(gk.reshape(want_k.shape), want_k)
        np.testing.assert_array_equal(gt.to(torch.float64).numpy().reshape(want_t.shape), want_t)


def test_repartition_empty_and_errors(ctx):
    empty = gpu_rel(ctx, (np.zeros((0, 1), np.int32), (4,), torch.zeros((0, 3))))
    out = ctx.repartition("Ij->iJ", empty)
    assert out.n == 0 and out.bounds == (3,) and out.shape == (4,)
    R = gpu_rel(ctx, (np.array([[1]], np.int32), (2,), torch.ones((1, 3))))
    for bad, err in [("Ij->Ik", "UCL_ERR_SPEC"), ("IJj->IJj", "UCL_ERR_SPEC"), ("IJ->IJ", "UCL_ERR_SHAPE"),
                     ("Ij", "UCL_ERR_SPEC"), ("Ij->I|jj", "UCL_ERR_SPEC"), ("Ij->I|j|", "UCL_ERR_SPEC")]:
        with pytest.raises(UclError, match=err):
            ctx.repartition(bad, R)
    # no key labels stay upper: no sync, every promoted index gets a tuple
    out = ctx.repartition("Ij->iJ", R)
    k, t = out.download()
    assert k[:, 0].tolist() == [0, 1, 2]
    assert t.tolist() == [[0.0, 1.0]] * 3


def test_repartition_round_trip_full_size(ctx):
    """The message-passing X (128 x 100000 bf16 as 1563 tiles [f][j]) split
    into 128-row vectors keyed (F, J) and stacked back: bit-identical, and
    the split relation matches the oracle on sampled tuples."""
    w = workloads.gnn_chain(seed=0, n=100_000, device="cpu")
    kx, bx, tx = w["X"]
    X = gpu_rel(ctx, w["X"])
    V = ctx.repartition("Jfj->fJ|j", X)
    assert V.n == 128 * len(kx) and V.shape == (64,)
    back = ctx.repartition("FJj->J|Fj", V)
    bk, bt = back.download()
    assert np.array_equal(bk, kx)
    assert torch.equal(bt, tx)
    vk, vt = V.download()
    rng = np.random.default_rng(1)
    rows = np.sort(rng.choice(len(kx), size=6, replace=False))
    want_k, _, want_t = oracle_repartition("Jfj->fJ|j", (kx[rows], bx, tx[rows].to(torch.float64).numpy()))
    got = {tuple(k): t for k, t in zip(vk.tolist(), vt.to(torch.float64).numpy())}
    for k, t in zip(want_k.tolist(), want_t):
        np.testing.assert_array_equal(got[tuple(k)], t)


def test_random_graph_contraction_sampled(ctx):
    """A message-passing-shaped EinSum on a uniform random graph: 600 vertex
    blocks, ~90k random (J, K) tiles over 1000 destination blocks (one in five
    empty).  The full key set and the values of 48 sampled keys (incl. the
    largest) against the oracle; then a second run, bit-identical."""
    rng = np.random.default_rng(11)
    nJ, nK, f, t = 600, 1000, 128, 64
    live = np.nonzero(rng.random(nK) < 0.8)[0]
    codes = np.unique(rng.integers(0, nJ, 120_000) * nK + rng.choice(live, 120_000))
    ky = np.stack([codes // nK, codes % nK], 1).astype(np.int32)
    g = torch.Generator().manual_seed(5)
    Xt = torch.randn((nJ, f, t), generator=g).to(torch.bfloat16)
    Yt = (torch.rand((len(ky), t, t), generator=g) < 0.1).to(torch.bfloat16)
    X = (np.arange(nJ, dtype=np.int32)[:, None], (nJ,), Xt)
    Y = (ky, (nJ, nK), Yt)
    spec = "fJj,JjKk->Kkf"
    out = ctx.einsum(spec, gpu_rel(ctx, X), gpu_rel(ctx, Y), out_dtype="bf16")
    assert ctx.last_stats()["n_pairs"] == len(ky) >= 1 << 16
    keys, _ = out.download()
    assert np.array_equal(keys[:, 0], np.unique(ky[:, 1]))
    cnt = np.bincount(ky[:, 1], minlength=nK)
    sk = np.unique(np.concatenate([rng.choice(np.nonzero(cnt)[0], 47, replace=False), [np.argmax(cnt)]]))
    m = np.isin(ky[:, 1], sk)
    ref = oracle_ref(spec, [X, (ky[m], (nJ, nK), Yt[torch.from_numpy(np.nonzero(m)[0])])],
                     sample_keys=sk[:, None].astype(np.int32))
    sel = np.searchsorted(keys[:, 0], sk)
    assert_parity(out, ref, torch.bfloat16, select=sel)
    out2 = ctx.einsum(spec, gpu_rel(ctx, X), gpu_rel(ctx, Y), out_dtype="bf16")
    assert torch.equal(out.download()[1], out2.download()[1])
