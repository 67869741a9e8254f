"""Pins of the CPU oracle against facts fixed by the paper and by mathematics.

Nothing here compares the oracle with itself: the references are the paper's
printed worked example (tests/golden/worked_example.txt), numpy.einsum (a
library routine), a pure-Python brute force over all index tuples, the
split invariant of Sec. 4.2 (every decomposition denotes the same tensor),
closed-form cardinalities (Sec. 1), and hand-derived rounding values.
"""
import itertools
import os

import numpy as np
import pytest

import oracle
import workloads
from oracle.repartition import RepartitionError, repartition
from tests.ucl_testutil import brute_force, decompose, golden, random_sparse, recompose, ucl_operand

GOLD = golden(os.path.join(os.path.dirname(__file__), "golden", "worked_example.txt"))


# --------------------------------------------------------------- Sec. 4.1 / 4.3


def test_worked_example_scalars():
    """Sec. 4.1: U as row vectors (key i), V as column vectors (key k), cross
    product + dot product -> W = {(0,0,7),(0,2,7.55),(2,0,4.48),(2,2,3.14)},
    with 16 scalar multiplications."""
    U, V = GOLD["U"], GOLD["V"]
    rows = [i for i in range(4) if U[i].any()]
    cols = [k for k in range(4) if V[:, k].any()]
    assert rows == [0, 2] and cols == [0, 2]
    relU = (np.array(rows, np.int32)[:, None], [4], U[rows])
    relV = (np.array(cols, np.int32)[:, None], [4], V[:, cols].T)
    r = oracle.einsum("Ij,jK->IK", [relU, relV])
    want = GOLD["W_scalars"]
    assert r["keys"].tolist() == want[:, :2].astype(int).tolist()
    np.testing.assert_allclose(r["acc"], want[:, 2], rtol=0, atol=1e-12)
    assert r["n_pairs"] == 4
    assert r["n_mults"] == int(GOLD["W_scalars_mults"][0, 0])


def test_worked_example_column_vectors():
    """Sec. 4.3: W_{i,K} <- sum U_{i,J} x V_{J,K} with V fully relational
    (its six (J, K, value) tuples as listed there) gives the column vectors
    K=0: [7,0,4.48,0] and K=2: [7.55,0,3.14,0] from six joined pairs."""
    U = GOLD["U"]
    vt = GOLD["V_relational_tuples"]
    relU = (np.arange(4, dtype=np.int32)[:, None], [4], U.T)  # key J, tile over i
    relV = (vt[:, :2].astype(np.int32), [4, 4], vt[:, 2])     # keys (J, K), rank-0 tiles
    r = oracle.einsum("iJ,JK->iK", [relU, relV])
    want = GOLD["W_colvec"]
    assert r["keys"][:, 0].tolist() == want[:, 0].astype(int).tolist()
    np.testing.assert_allclose(r["acc"], want[:, 1:], rtol=0, atol=1e-12)
    assert r["n_pairs"] == 6


def test_worked_example_dense_split_agrees():
    """The same product with every label demoted (one key-less tuple each)
    equals the dense product and the two decompositions above."""
    U, V = GOLD["U"], GOLD["V"]
    r = oracle.einsum("ij,jk->ik", [(np.zeros((1, 0), np.int32), [], U[None]),
                                    (np.zeros((1, 0), np.int32), [], V[None])])
    np.testing.assert_allclose(r["acc"][0], U @ V, rtol=0, atol=1e-12)
    assert r["n_pairs"] == 1 and r["n_mults"] == 64


# ----------------------------------------------------- dense references


CASES = [
    # (dense spec, shapes)  -- extents all distinct so a transposed operand fails
    ("ij,jk->ik", {"i": 3, "j": 4, "k": 5}),
    ("ij,jk->ki", {"i": 3, "j": 4, "k": 2}),
    ("ijb,jbk->ik", {"i": 2, "j": 3, "b": 4, "k": 5}),         # Sec. 3 batch-matmul-with-sum
    ("bij,bjk->bik", {"b": 2, "i": 3, "j": 4, "k": 3}),
    ("ij,j->i", {"i": 4, "j": 5}),
    ("i,j->ij", {"i": 3, "j": 4}),                             # outer product, no shared label
    ("ij,ij->i", {"i": 3, "j": 4}),
    ("ijk,jr,kr->ir", {"i": 3, "j": 2, "k": 4, "r": 5}),       # MTTKRP, three operands
    ("ijk->ki", {"i": 3, "j": 2, "k": 4}),                     # unary with a summed label
]


def _dense_inputs(rng, spec, ext):
    ops = spec.split("->")[0].split(",")
    arrs = []
    for op in ops:
        arrs.append(random_sparse(rng, [ext[c] for c in op], density=0.6, block_axes=range(len(op))))
    return ops, arrs


def _run_split(spec, ext, arrs, promoted):
    lhs, out = spec.split("->")
    ops = lhs.split(",")
    rels = [decompose(a, op, promoted) for op, a in zip(ops, arrs)]
    uspec = ",".join(ucl_operand(op, promoted) for op in ops) + "->" + ucl_operand(out, promoted)
    r = oracle.einsum(uspec, rels)
    dense = recompose(r["keys"], r["acc"], out, promoted, ext)
    dense_abs = recompose(r["keys"], r["abs"], out, promoted, ext)
    return r, dense, dense_abs


@pytest.mark.parametrize("spec,ext", CASES)
def test_matches_numpy_einsum(spec, ext):
    rng = np.random.default_rng(7)
    ops, arrs = _dense_inputs(rng, spec, ext)
    want = np.einsum(spec, *arrs)
    want_abs = np.einsum(spec, *[np.abs(a) for a in arrs])
    labels = sorted(ext)
    for promoted in [set(), set(labels[:1]), set(labels[1:]), set(labels)]:
        _, got, got_abs = _run_split(spec, ext, arrs, promoted)
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(got_abs, want_abs, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("spec,ext", CASES[:6])
def test_matches_brute_force(spec, ext):
    """Pure-Python enumeration of the definition, independent of numpy.einsum."""
    rng = np.random.default_rng(11)
    ops, arrs = _dense_inputs(rng, spec, ext)
    want = brute_force(spec, arrs)
    labels = sorted(ext)
    _, got, _ = _run_split(spec, ext, arrs, set(labels[::2]))
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("spec,ext", [CASES[0], CASES[2], CASES[7]])
def test_split_invariant(spec, ext):
    """Sec. 4.2: all decompositions of a tensor denote the same tensor, so every
    consistent choice of promoted labels -- from all-lower (one key-less tuple,
    i.e. the dense computation) to all-upper (rank-0 tiles, i.e. purely
    relational) -- yields the same result."""
    rng = np.random.default_rng(3)
    ops, arrs = _dense_inputs(rng, spec, ext)
    labels = sorted(ext)
    ref = None
    for k in range(len(labels) + 1):
        for sub in itertools.combinations(labels, k):
            _, got, _ = _run_split(spec, ext, arrs, set(sub))
            if ref is None:
                ref = got
            np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_tiled_reshape_matches_dense():
    """A8 reading: a dense extent split into (tile index I, offset i) by
    reshape; block-sparse matmul over tiles equals the dense matmul, with the
    ragged last tile zero-padded."""
    rng = np.random.default_rng(5)
    m, n, p, t = 10, 7, 9, 4  # not multiples of t -> padded tiles
    A = rng.standard_normal((m, n)) * (rng.random((m, n)) < 0.5)
    B = rng.standard_normal((n, p))

    def tiles_of(M):
        r, c = M.shape
        R, C = -(-r // t), -(-c // t)
        P = np.zeros((R * t, C * t))
        P[:r, :c] = M
        keys, vals = [], []
        for I in range(R):
            for J in range(C):
                blk = P[I * t:(I + 1) * t, J * t:(J + 1) * t]
                if blk.any():
                    keys.append((I, J))
                    vals.append(blk)
        return np.array(keys, np.int32), [R, C], np.array(vals)

    ka, ba, va = tiles_of(A)
    kb, bb, vb = tiles_of(B)
    r = oracle.einsum("IiJj,JjKk->IiKk", [(ka, ba, va), (kb, bb, vb)])
    C = np.zeros((ba[0] * t, bb[1] * t))
    for (I, K), tile in zip(r["keys"], r["acc"]):
        C[I * t:(I + 1) * t, K * t:(K + 1) * t] = tile
    np.testing.assert_allclose(C[:m, :p], A @ B, rtol=1e-12, atol=1e-12)
    assert not C[m:, :].any() and not C[:, p:].any()  # padding comes out zero
    # closed-form pair count of the join on J
    cnt_a = np.bincount(ka[:, 1], minlength=ba[1])
    cnt_b = np.bincount(kb[:, 0], minlength=bb[0])
    assert r["n_pairs"] == int((cnt_a * cnt_b).sum())


def test_mttkrp_workload_matches_dense():
    """The sparse MTTKRP workload (Zipf coordinates in t^3 tiles, ragged last
    tile row of the factors) evaluated by the oracle equals the dense
    MTTKRP of the same values; one triple per nonempty T tile."""
    n, t, rank = 42, 4, 3
    w = workloads.mttkrp(seed=2, n=n, nnz=300, t=t, rank=rank)
    T, B, C = (workloads.to_oracle(w[k]) for k in ("T", "B", "C"))
    assert np.unique(w["coords"].numpy()).size == 300
    dense = np.zeros((len(B[2]) * t,) * 3)
    for (I, J, K), tile in zip(T[0], T[2]):
        dense[I * t:(I + 1) * t, J * t:(J + 1) * t, K * t:(K + 1) * t] = tile
    assert np.count_nonzero(dense) <= 300 and not dense[n:].any()
    Bd, Cd = B[2].reshape(-1, rank), C[2].reshape(-1, rank)
    assert not Bd[n:].any() and not Cd[n:].any()
    want = np.einsum("ijk,jr,kr->ir", dense, Bd, Cd)
    r = oracle.einsum(w["spec"], [T, B, C])
    assert r["n_pairs"] == len(T[0])
    got = np.zeros_like(want)
    for (I,), tile in zip(r["keys"], r["acc"]):
        got[I * t:(I + 1) * t] = tile
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


# ------------------------------------------------------ cardinalities (Sec. 1)


def test_gnn_cardinalities_closed_form():
    """Sec. 1's message-passing arithmetic, scaled down: with n vertices of
    out-degree d and embeddings of width e, the purely relational join of X
    and Y produces n*d*e tuples which group down to n*e; the tensor-relational
    version (X as per-vertex vectors) produces n*d tuples.  At the paper's
    sizes (n=1e8, d=1000, e=8192) these are the quoted 820 trillion, 820
    billion and 100 billion."""
    n, d, e = 12, 3, 5
    assert 10**8 * 1000 * 8192 == 819_200_000_000_000  # "820 trillion"
    assert 10**8 * 8192 == 819_200_000_000             # "820 billion"
    assert 10**8 * 1000 == 100_000_000_000             # "100 billion"
    rng = np.random.default_rng(0)
    X = rng.standard_normal((e, n)) + 3.0  # no zero entries
    edges = np.array([(j, (j + s) % n) for j in range(n) for s in range(1, d + 1)], np.int32)
    # purely relational: X(F, J) scalars, Y(J, K) scalars -> T(K, F)
    fx = np.array([(f, j) for f in range(e) for j in range(n)], np.int32)
    r = oracle.einsum("FJ,JK->KF", [(fx, [e, n], X[fx[:, 0], fx[:, 1]]),
                                    (edges, [n, n], np.ones(len(edges)))])
    assert r["n_pairs"] == n * d * e
    assert r["keys"].shape[0] == n * e
    # tensor-relational: X(J) vectors over f, Y(J, K) scalars -> T(K) vectors
    r2 = oracle.einsum("fJ,JK->Kf", [(np.arange(n, dtype=np.int32)[:, None], [n], X.T),
                                     (edges, [n, n], np.ones(len(edges)))])
    assert r2["n_pairs"] == n * d
    # both denote the same tensor
    dense = np.zeros((n, e))
    for (K, F), v in zip(r["keys"], r["acc"]):
        dense[K, F] = v
    np.testing.assert_allclose(r2["acc"], dense[r2["keys"][:, 0]], rtol=1e-12)


# -------------------------------------------------------------- epilogue, cast


def test_round_bf16_hand_values():
    """Round-to-nearest-even to bfloat16 (8 significant bits), hand-derived."""
    assert oracle.round_bf16(1.0 + 2.0**-8) == 1.0                  # tie -> even
    assert oracle.round_bf16(1.0 + 3 * 2.0**-8) == 1.0 + 2.0**-6     # tie -> even (up)
    assert oracle.round_bf16(1.0 + 2.0**-8 + 2.0**-20) == 1.0 + 2.0**-7
    assert oracle.round_bf16(-(1.0 + 2.0**-8 + 2.0**-20)) == -(1.0 + 2.0**-7)
    assert oracle.round_bf16(np.pi) == 3.140625
    assert oracle.round_bf16(2.0**-133) == 2.0**-133                 # smallest subnormal
    assert oracle.round_bf16(2.0**-135) == 0.0
    assert oracle.round_bf16((2 - 2.0**-7) * 2.0**127) == (2 - 2.0**-7) * 2.0**127
    assert np.isinf(oracle.round_bf16(2.0**128))
    assert oracle.round_bf16(0.0) == 0.0


def test_epilogue_scale_relu_cast():
    """Epilogue after the full sum (Sec. 3 MLP example: ReLU as a unary
    EinSum over the empty set): out = cast(relu(scale * sum))."""
    keys = np.array([[0], [1]], np.int32)
    a = np.array([[1.5, -2.0, 0.1], [3.0, -0.25, 2.0]])
    r = oracle.einsum("Ij->I", [(keys, [2], a)], epi="relu", scale=-2.0, out_dtype="f32")
    np.testing.assert_array_equal(r["acc"], a.sum(axis=1))
    want = [max(0.0, -2.0 * (1.5 - 2.0 + 0.1)), max(0.0, -2.0 * (3.0 - 0.25 + 2.0))]
    np.testing.assert_array_equal(r["out"], np.float32(want).astype(np.float64))
    r = oracle.einsum("Ij->Ij", [(keys, [2], a)], out_dtype="bf16")
    np.testing.assert_array_equal(r["out"], np.vectorize(oracle.round_bf16)(a))


# ----------------------------------------------------------- edge cases, errors


def test_empty_inputs_and_empty_join():
    e = (np.zeros((0, 1), np.int32), [4], np.zeros((0, 2, 3)))
    f = (np.array([[1]], np.int32), [4], np.ones((1, 3, 2)))
    r = oracle.einsum("Jij,Jjk->ik", [e, f])
    assert r["keys"].shape == (0, 0) and r["acc"].shape == (0, 2, 2)
    g = (np.array([[2]], np.int32), [4], np.ones((1, 2, 3)))
    r = oracle.einsum("Jij,Jjk->Jik", [g, f])  # keys 2 vs 1: empty join
    assert r["n_pairs"] == 0 and r["keys"].shape == (0, 1)


def test_zero_sum_keys_are_kept():
    """A2 reading: an output key produced by the join stays even if it sums to 0."""
    u = (np.array([[0]], np.int32), [1], np.array([[1.0, -1.0]]))
    v = (np.array([[0]], np.int32), [1], np.array([[1.0, 1.0]]))
    r = oracle.einsum("Ij,Ij->I", [u, v])
    assert r["keys"].tolist() == [[0]] and r["acc"].tolist() == [0.0]


def test_sampled_keys_match_full():
    rng = np.random.default_rng(9)
    spec, ext = CASES[0]
    ops, arrs = _dense_inputs(rng, spec, ext)
    promoted = {"i", "k"}
    rels = [decompose(a, op, promoted) for op, a in zip(ops, arrs)]
    full = oracle.einsum("Ij,jK->IK", rels)
    pick = full["keys"][::2]
    part = oracle.einsum("Ij,jK->IK", rels, sample_keys=pick)
    assert part["keys"].tolist() == pick.tolist()
    np.testing.assert_array_equal(part["acc"], full["acc"][::2])
    assert part["n_pairs"] == full["n_pairs"]


@pytest.mark.parametrize("spec,n_in,err", [
    ("Ij,jK", 2, "ERR_SPEC"),        # no arrow
    ("Ij,jK->IQ", 2, "ERR_SPEC"),    # output label from nowhere
    ("Iij,jK->IK", 2, "ERR_SHAPE"),  # operand arity does not match the relation
    ("IIj,jK->IK", 2, "ERR_SPEC"),   # repeated label
    ("Ij,j1->I", 2, "ERR_SPEC"),     # not a letter
    ("Ij->I", 2, "ERR_SPEC"),        # operand count
])
def test_spec_errors(spec, n_in, err):
    u = (np.array([[0]], np.int32), [2], np.ones((1, 3)))
    v = (np.array([[1]], np.int32), [2], np.ones((1, 3)))
    with pytest.raises(oracle.OracleError) as ei:
        oracle.einsum(spec, [u, v][:n_in])
    assert ei.value.name == err


def test_relation_errors():
    v = (np.array([[1]], np.int32), [2], np.ones((1, 3)))
    dup = (np.array([[0], [0]], np.int32), [2], np.ones((2, 3)))
    with pytest.raises(oracle.OracleError, match="ERR_DUP_KEY"):
        oracle.einsum("Ij,jK->IK", [dup, v])
    bad = (np.array([[2]], np.int32), [2], np.ones((1, 3)))
    with pytest.raises(oracle.OracleError, match="ERR_KEY_RANGE"):
        oracle.einsum("Ij,jK->IK", [bad, v])
    neg = (np.array([[-1]], np.int32), [2], np.ones((1, 3)))
    with pytest.raises(oracle.OracleError, match="ERR_KEY_RANGE"):
        oracle.einsum("Ij,jK->IK", [neg, v])
    w = (np.array([[1]], np.int32), [2], np.ones((1, 4)))  # extent of j disagrees
    with pytest.raises(oracle.OracleError, match="ERR_SHAPE"):
        oracle.einsum("Ij,jK->IK", [v, w])
    x = (np.array([[1]], np.int32), [3], np.ones((1, 3)))  # bound of I disagrees
    with pytest.raises(oracle.OracleError, match="ERR_SHAPE"):
        oracle.einsum("Ij,Ij->I", [v, x])


# ---------------------------------------------------- repartition (Sec. 6)



def test_repartition_row_vectors_to_column_vectors():
    """Sec. 6's example: T stored as row vectors (upper row index) becomes T
    stored as column vectors (upper column index); every column index gets a
    tuple (the decompose step ranges over the whole label)."""
    T = np.array([[1.0, 0.0, 2.0, 0.0], [0.0, 0.0, 3.0, 0.0], [4.0, 0.0, 5.0, 0.0]])
    rows = decompose(T, "ki", {"k"}, drop_zero=False)
    keys, bounds, tiles = repartition("Ki->kI", rows)
    assert bounds == (4,)
    assert keys[:, 0].tolist() == [0, 1, 2, 3]
    np.testing.assert_array_equal(tiles, T.T)


@pytest.mark.parametrize("labels,ext,src,rhs", [
    ("ij", {"i": 5, "j": 4}, {"i"}, "iJ"),             # rows -> columns
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"i"}, "IjK"),    # decompose only
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"i", "j"}, "iJk"),   # stack only
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"j", "k"}, "Ijk"),   # both
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"i"}, "Ikj"),    # tile dims reordered
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"j", "k"}, "KiJ"),   # keys reordered, i promoted
    ("ijk", {"i": 3, "j": 4, "k": 2}, set(), "IJK"),    # dense -> scalars
    ("ijk", {"i": 3, "j": 4, "k": 2}, {"i", "j", "k"}, "kji"),   # scalars -> one dense tuple, reversed
])
def test_repartition_keeps_the_tensor(labels, ext, src, rhs):
    """The repartitioned relation denotes the same dense tensor, and its key
    set is (kept key values present) x (full range of each promoted label),
    in ascending order."""
    rng = np.random.default_rng(len(labels) * 7 + len(src) + len(rhs))
    dense = random_sparse(rng, [ext[c] for c in labels], density=0.5, block_axes=range(len(labels)))
    rel = decompose(dense, labels, src)
    lhs = "".join(c.upper() for c in labels if c in src) + "".join(c for c in labels if c not in src)
    keys, bounds, tiles = repartition(lhs + "->" + rhs, rel)
    dst = {c.lower() for c in rhs if c.isupper()}
    out_order = rhs.lower()
    back = recompose(keys, tiles, out_order, dst, ext)
    np.testing.assert_array_equal(np.transpose(back, [out_order.index(c) for c in labels]), dense)
    src_up = [c for c in labels if c in src]
    out_up = [c.lower() for c in rhs if c.isupper()]
    kept = [c for c in out_up if c in src]
    prom = [c for c in out_up if c not in src]
    kept_vals = {tuple(int(k[src_up.index(c)]) for c in kept) for k in rel[0]}
    want = set()
    for kv in kept_vals:
        for pv in itertools.product(*[range(ext[c]) for c in prom]):
            d = dict(zip(kept, kv))
            d.update(zip(prom, pv))
            want.add(tuple(d[c] for c in out_up))
    assert set(map(tuple, keys.tolist())) == want
    assert keys.tolist() == sorted(keys.tolist())
    assert bounds == tuple(ext[c] for c in out_up)


def test_repartition_identity_and_errors():
    rng = np.random.default_rng(2)
    rel = decompose(random_sparse(rng, [4, 3], density=0.6, block_axes=(0, 1)), "ij", {"i"})
    k, b, t = repartition("Ij->Ij", rel)
    np.testing.assert_array_equal(k, rel[0])
    np.testing.assert_array_equal(t, rel[2])
    for bad in ["Ij->Ik", "Ij->IJj", "Ij", "IJj->Ij", "Ij->I"]:
        with pytest.raises(RepartitionError):
            repartition(bad, rel)


def test_repartition_explicit_form_with_tile_and_offset_labels():
    """A reshaped dense index keeps its tile index J and offset j as two
    labels; the explicit "<keys>|<tile dims>" form names them apart.  Here X
    stored as [f][j] tiles keyed J becomes j-vectors keyed (f, J), and back."""
    rng = np.random.default_rng(9)
    dense = random_sparse(rng, [5, 3, 4], density=0.5, block_axes=(0, 1, 2))   # axes J, f, j
    ext = {"J": 5, "f": 3, "j": 4}
    rel = decompose(dense, "Jfj", {"J"})
    keys, bounds, tiles = repartition("Jfj->fJ|j", rel)
    assert bounds == (3, 5) and tiles.shape[1:] == (4,)
    back = recompose(keys, tiles, "fJj", {"f", "J"}, ext)
    np.testing.assert_array_equal(np.transpose(back, [1, 0, 2]), dense)
    assert len(keys) == 3 * len(rel[0])    # every f for every J present
    k2, b2, t2 = repartition("FJj->J|Fj", (keys, bounds, tiles))
    np.testing.assert_array_equal(k2, rel[0])
    np.testing.assert_array_equal(t2, rel[2])
    with pytest.raises(RepartitionError):
        repartition("Jfj->fJ", rel)      # case form cannot tell J from j
    with pytest.raises(RepartitionError):
        repartition("Jfj->fj|J|", rel)


# ------------------------------------------- extended EinSum (Sec. 3, Eq. Einsum)

def _rel_from_dense(dense, labels, up):
    keys, bounds, tiles = decompose(dense, labels, set(up), drop_zero=False)
    return keys, bounds, tiles


def _ext(spec, dense_ops, op_labels, ups, out_labels, out_up, **kw):
    rels = [_rel_from_dense(d, l, u) for d, l, u in zip(dense_ops, op_labels, ups)]
    r = oracle.einsum(spec, rels, **kw)
    ext = {}
    for d, l in zip(dense_ops, op_labels):
        ext.update(zip(l, d.shape))
    return recompose(r["keys"], r["out"], out_labels, set(out_up), ext), r


@pytest.mark.parametrize("ups", [("ij", "ij", "i"), ("i", "i", "i"), ("", "", ""), ("j", "j", "")])
def test_extended_max_squared_difference(ups):
    """Sec. 3's example W_i = max_j (U_ij - V_ij)^2 under several splits."""
    rng = np.random.default_rng(21)
    U, V = rng.standard_normal((3, 5)), rng.standard_normal((3, 5))
    spec = ucl_operand("ij", set(ups[0])) + "," + ucl_operand("ij", set(ups[1])) + "->" + ucl_operand("i", set(ups[2]))
    got, r = _ext(spec, [U, V], ["ij", "ij"], ups[:2], "i", ups[2], agg="max", comb="sub", map="square")
    np.testing.assert_allclose(got, np.max((U - V) ** 2, axis=1), rtol=1e-15)
    # the magnitude bound of MAX is the largest |term|
    assert np.all(r["abs"].reshape(-1) >= np.abs(r["acc"].reshape(-1)))


@pytest.mark.parametrize("agg,np_fn", [("min", np.min), ("max", np.max), ("sum", np.sum)])
@pytest.mark.parametrize("comb,np_op", [("mul", np.multiply), ("add", np.add), ("sub", np.subtract)])
def test_extended_aggregates_and_combinations(agg, np_fn, comb, np_op):
    rng = np.random.default_rng(22)
    U, V = rng.standard_normal((4, 3)), rng.standard_normal((3, 5))
    want = np_fn(np_op(U[:, :, None], V[None, :, :]), axis=1)
    for ups in [("i", "k", "ik"), ("ij", "jk", "ik"), ("", "", ""), ("j", "j", "")]:
        spec = (ucl_operand("ij", set(ups[0])) + "," + ucl_operand("jk", set(ups[1])) + "->" +
                ucl_operand("ik", set(ups[2])))
        got, _ = _ext(spec, [U, V], ["ij", "jk"], ups[:2], "ik", ups[2], agg=agg, comb=comb)
        np.testing.assert_allclose(got, want, rtol=1e-13, atol=1e-15)


def test_extended_unary_maps_and_division():
    rng = np.random.default_rng(23)
    U = rng.standard_normal((3, 4))
    for m, fn in [("relu", lambda x: np.maximum(x, 0)), ("exp", np.exp), ("square", np.square), ("ident", lambda x: x)]:
        got, _ = _ext("Ij->Ij", [U], ["ij"], ["i"], "ij", "i", map=m)
        np.testing.assert_allclose(got, fn(U), rtol=1e-15)
    D = rng.uniform(1, 2, 3)
    got, _ = _ext("Ij,I->Ij", [U, D], ["ij", "i"], ["i", "i"], "ij", "i", comb="div")
    np.testing.assert_allclose(got, U / D[:, None], rtol=1e-15)


def test_softmax_as_extended_einsums():
    """Row softmax as four EinSums (max; exp of the difference; sum;
    quotient) against the textbook formula."""
    rng = np.random.default_rng(24)
    C = rng.standard_normal((5, 7)) * 3
    rc = _rel_from_dense(C, "ij", {"i"})
    M = oracle.einsum("Ij->I", [rc], agg="max")
    rm = (M["keys"], M["bounds"], M["out"])
    S = oracle.einsum("Ij,I->Ij", [rc, rm], comb="sub", map="exp")
    rs = (S["keys"], S["bounds"], S["out"])
    D = oracle.einsum("Ij->I", [rs])
    E = oracle.einsum("Ij,I->Ij", [rs, (D["keys"], D["bounds"], D["out"])], comb="div")
    ref = np.exp(C) / np.exp(C).sum(axis=1, keepdims=True)
    np.testing.assert_allclose(E["out"], ref, rtol=1e-13)


def test_extended_aggregate_ranges_over_present_tuples():
    """MAX over a relation with absent tuples: the absent ones contribute
    nothing (brute force over the tuples present)."""
    rng = np.random.default_rng(25)
    keys = np.array([[0, 1], [0, 3], [2, 0], [2, 2], [2, 3]], np.int32)
    vals = -rng.uniform(1, 2, len(keys))               # all negative: an absent zero would win a dense max
    r = oracle.einsum("IJ->I", [(keys, (3, 4), vals)], agg="max")
    want = {}
    for (i, j), v in zip(keys.tolist(), vals):
        want[i] = max(want.get(i, -np.inf), v)
    assert r["keys"][:, 0].tolist() == sorted(want)
    np.testing.assert_array_equal(r["out"], [want[i] for i in sorted(want)])


def test_extended_three_inputs_unsupported():
    rel = (np.zeros((1, 0), np.int32), (), np.ones((1, 2)))
    with pytest.raises(oracle.OracleError, match="UNSUPPORTED"):
        oracle.einsum("i,i,i->i", [rel, rel, rel], agg="max")
