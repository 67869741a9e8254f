"""Seeded synthetic inputs shaped like the paper's workloads.

This module only draws random tensors and cuts them into tensor-relations
(keys + tiles); it holds none of the EinSum arithmetic.  Both the GPU tests
and the oracle tests consume what it returns, so neither side depends on the
other.  The paper's datasets (ogbn-*, friendster, Planetoid, QASMBench) are
not available; these inputs stand in for them.

A relation is returned as ``(keys, bounds, tiles)``: keys int32 [n, u] (numpy),
bounds a tuple, tiles a torch tensor [n, *shape] (CPU unless built on the GPU).
Keys are emitted in ascending lexicographic order.
"""
from __future__ import annotations

import math

import numpy as np
import torch

# ------------------------------------------------------------------ helpers


def _tiles_of_dense(dense: torch.Tensor, tr: int, tc: int):
    """Cut a dense [R, C] matrix into [tr x tc] tiles keyed (I, J), zero-padding
    the ragged edge; every tile is kept (dense operand)."""
    R, C = dense.shape
    nr, nc = -(-R // tr), -(-C // tc)
    pad = torch.zeros((nr * tr, nc * tc), dtype=dense.dtype, device=dense.device)
    pad[:R, :C] = dense
    tiles = pad.reshape(nr, tr, nc, tc).permute(0, 2, 1, 3).reshape(nr * nc, tr, tc).contiguous()
    I, J = np.meshgrid(np.arange(nr), np.arange(nc), indexing="ij")
    keys = np.stack([I.ravel(), J.ravel()], axis=1).astype(np.int32)
    return keys, (nr, nc), tiles


def rmat_edges(n: int, n_edges: int, a=0.57, b=0.19, c=0.19, seed=0, batch=1 << 22):
    """R-MAT edge list (Chakrabarti et al.) on 2^ceil(log2 n) vertices; edges
    with an endpoint >= n are rejected and redrawn until n_edges remain, then
    duplicates are removed (self-loops kept).  Returns (src, dst) int64
    sorted by (src, dst)."""
    rng = np.random.default_rng(seed)
    levels = max(1, math.ceil(math.log2(n)))
    srcs, dsts, have = [], [], 0
    while have < n_edges:
        m = min(batch, 2 * (n_edges - have) + 1024)
        s = np.zeros(m, dtype=np.int64)
        d = np.zeros(m, dtype=np.int64)
        for _ in range(levels):
            r = rng.random(m)
            sb = r >= a + b                       # quadrants c, d: lower half of the rows
            db = ((r >= a) & (r < a + b)) | (r >= a + b + c)  # quadrants b, d: right half
            s = (s << 1) | sb
            d = (d << 1) | db
        ok = (s < n) & (d < n)
        s, d = s[ok], d[ok]
        take = min(len(s), n_edges - have)
        srcs.append(s[:take])
        dsts.append(d[:take])
        have += take
    s = np.concatenate(srcs)
    d = np.concatenate(dsts)
    code = np.unique(s * n + d)
    return code // n, code % n


def adjacency_tiles(src, dst, n: int, t: int, device="cpu", dtype=torch.bfloat16):
    """0/1 adjacency Y[src, dst] = 1 stored as only-nonempty [t x t] tiles
    keyed (J = src // t, K = dst // t), ascending."""
    nt = -(-n // t)
    tcode = (src // t) * nt + (dst // t)
    ukeys, inv = np.unique(tcode, return_inverse=True)
    keys = np.stack([ukeys // nt, ukeys % nt], axis=1).astype(np.int32)
    tiles = torch.zeros((len(ukeys), t, t), dtype=dtype, device=device)
    idx = torch.as_tensor(inv, device=device)
    r = torch.as_tensor(src % t, device=device)
    q = torch.as_tensor(dst % t, device=device)
    tiles[idx, r, q] = 1
    return keys, (nt, nt), tiles


def adjacency_tiles_subset(src, dst, n: int, t: int, keys_wanted: np.ndarray):
    """The same tiles as adjacency_tiles, only for the (J, K) keys given, as a
    float64 CPU array (for the oracle on sampled output keys)."""
    nt = -(-n // t)
    want = keys_wanted[:, 0].astype(np.int64) * nt + keys_wanted[:, 1]
    tcode = (src // t) * nt + (dst // t)
    pos = {int(c): i for i, c in enumerate(want)}
    tiles = np.zeros((len(want), t, t))
    sel = np.isin(tcode, want)
    for s, d, c in zip(src[sel], dst[sel], tcode[sel]):
        tiles[pos[int(c)], s % t, d % t] = 1.0
    return tiles


# ----------------------------------------------------------------- workloads


def blocksparse_matmul(seed=0, n=1024, m=256, t=32, density=0.10):
    """Block-sparse C[I,K] = sum_J A[I,J] B[J,K] over t x t fp32 tiles: A
    n x n with round(density * (n/t)^2) tiles drawn uniformly without
    replacement, B dense n x m, values U[-1, 1].  Spec IiJj,JjKk->IiKk."""
    rng = np.random.default_rng(seed)
    g = n // t
    nnz = round(density * g * g)
    pick = np.sort(rng.choice(g * g, size=nnz, replace=False))
    ka = np.stack([pick // g, pick % g], axis=1).astype(np.int32)
    ta = torch.from_numpy(rng.uniform(-1, 1, size=(nnz, t, t)).astype(np.float32))
    B = torch.from_numpy(rng.uniform(-1, 1, size=(n, m)).astype(np.float32))
    kb, bb, tb = _tiles_of_dense(B, t, t)
    return {
        "spec": "IiJj,JjKk->IiKk",
        "A": (ka, (g, g), ta),
        "B": (kb, bb, tb),
    }


def gnn_chain(seed=0, n=100_000, feat=128, out_feat=128, degree=16, t=64, device="cpu", z_std=0.1):
    """Message passing (X x Y)^T x Z: X feat x n bf16 N(0,1) stored per vertex
    tile J as [f x j] tiles; Y an R-MAT adjacency (a,b,c = .57,.19,.19, n*degree
    edges) as only-nonempty t x t 0/1 tiles keyed (J, K); Z feat x out_feat
    bf16 N(0, z_std^2) as one key-less tuple.
    Specs: fJj,JjKk->Kkf (T = (X Y)^T), then Kkf,fg->Kkg (T Z)."""
    g = torch.Generator().manual_seed(seed)
    X = torch.randn((feat, n), generator=g).to(torch.bfloat16)
    nt = -(-n // t)
    Xp = torch.zeros((feat, nt * t), dtype=torch.bfloat16)
    Xp[:, :n] = X
    xt = Xp.reshape(feat, nt, t).permute(1, 0, 2).contiguous()   # [J][f][j]
    kx = np.arange(nt, dtype=np.int32)[:, None]
    src, dst = rmat_edges(n, n * degree, seed=seed + 1)
    ky, by, ty = adjacency_tiles(src, dst, n, t, device=device)
    Z = (torch.randn((feat, out_feat), generator=g) * z_std).to(torch.bfloat16)
    return {
        "spec1": "fJj,JjKk->Kkf",
        "spec2": "Kkf,fg->Kkg",
        "X": (kx, (nt,), xt.to(device)),
        "Y": (ky, by, ty),
        "Z": (np.zeros((1, 0), np.int32), (), Z[None].to(device)),
        "edges": (src, dst),
        "n": n,
        "t": t,
    }


def spgemm(seed=0, n=65536, t=128, density=0.005, band=(-1, 0, 1, 2)):
    """Block-sparse x block-sparse: A and B n x n with t x t bf16 N(0,1) tiles
    at the given tile density, half of the tiles on the band J - I in `band`,
    half uniform among the off-band tiles; drawn independently for A and B.
    Spec IiJj,JjKk->IiKk (fp32 output)."""
    rng = np.random.default_rng(seed)
    g = n // t
    nnz = round(density * g * g)
    n_band = nnz // 2

    def draw():
        I = np.arange(g)
        bi = np.concatenate([I for _ in band])
        bj = np.concatenate([I + d for d in band])
        ok = (bj >= 0) & (bj < g)
        bcodes = (bi * g + bj)[ok]
        bsel = rng.choice(bcodes, size=n_band, replace=False)
        rest = nnz - n_band
        chosen = set(bsel.tolist())
        bandset = set(bcodes.tolist())
        out = []
        while len(out) < rest:
            c = int(rng.integers(0, g * g))
            if c in bandset or c in chosen:
                continue
            chosen.add(c)
            out.append(c)
        codes = np.sort(np.concatenate([bsel, np.array(out, dtype=np.int64)]))
        keys = np.stack([codes // g, codes % g], axis=1).astype(np.int32)
        tiles = torch.from_numpy(rng.standard_normal((len(codes), t, t)).astype(np.float32)).to(torch.bfloat16)
        return keys, (g, g), tiles

    return {"spec": "IiJj,JjKk->IiKk", "A": draw(), "B": draw()}


def rmat_edges_device(n: int, n_edges: int, a=0.57, b=0.19, c=0.19, seed=0, device="cuda", batch=1 << 25):
    """rmat_edges drawn with torch on the GPU (for graphs too large for host
    numpy): same model and rejection rule; returns (src, dst) int64 device
    tensors, de-duplicated and sorted by (src, dst)."""
    g = torch.Generator(device=device).manual_seed(seed)
    levels = max(1, math.ceil(math.log2(n)))
    parts, have = [], 0
    while have < n_edges:
        m = min(batch, int((n_edges - have) * 1.15) + 1024)
        s = torch.zeros(m, dtype=torch.int64, device=device)
        d = torch.zeros(m, dtype=torch.int64, device=device)
        for _ in range(levels):
            r = torch.rand(m, generator=g, device=device)
            sb = (r >= a + b).long()
            db = (((r >= a) & (r < a + b)) | (r >= a + b + c)).long()
            s = s * 2 + sb
            d = d * 2 + db
        ok = (s < n) & (d < n)
        code = (s * n + d)[ok][: n_edges - have]
        parts.append(code)
        have += code.numel()
    code = torch.unique(torch.cat(parts))
    return code // n, code % n


def adjacency_tiles_device(src, dst, n: int, t: int, dtype=torch.bfloat16):
    """adjacency_tiles for device edge tensors: only-nonempty [t x t] 0/1
    tiles keyed (J = src // t, K = dst // t), ascending; keys returned as a
    host int32 array, tiles on the device."""
    nt = -(-n // t)
    tcode = (src // t) * nt + (dst // t)
    ukeys, inv = torch.unique(tcode, return_inverse=True)
    tiles = torch.zeros((ukeys.numel(), t, t), dtype=dtype, device=src.device)
    tiles[inv, src % t, dst % t] = 1
    keys = torch.stack([ukeys // nt, ukeys % nt], dim=1).to(torch.int32).cpu().numpy()
    return keys, (nt, nt), tiles


def gnn_two_layer(seed=0, n=2_000_000, n_edges=40_000_000, feat=256, t=64, device="cuda", w_std=None):
    """Two-layer GNN at scale: an R-MAT graph (a,b,c = .57,.19,.19) with
    n_edges drawn edges as only-nonempty t x t 0/1 bf16 tiles Y keyed (J, K);
    X feat x n bf16 N(0,1) as per-J tiles [f x j]; W1, W2 feat x feat bf16
    N(0, 1/feat) (the config leaves their distribution open).  Chain:
    T1 = (X Y)^T, H1 = relu(T1 W1), T2 = (H1 Y)^T, O = T2 W2."""
    g = torch.Generator(device=device).manual_seed(seed)
    nt = -(-n // t)
    X = torch.randn((nt, feat, t), generator=g, device=device).to(torch.bfloat16)
    if n % t:
        X[-1, :, n % t:] = 0
    std = w_std if w_std is not None else feat ** -0.5
    W1 = (torch.randn((feat, feat), generator=g, device=device) * std).to(torch.bfloat16)
    W2 = (torch.randn((feat, feat), generator=g, device=device) * std).to(torch.bfloat16)
    src, dst = rmat_edges_device(n, n_edges, seed=seed + 1, device=device)
    ky, by, ty = adjacency_tiles_device(src, dst, n, t)
    nokey = np.zeros((1, 0), np.int32)
    return {
        "spec1": "fJj,JjKk->Kkf",
        "spec2": "Kkf,fg->Kkg",
        "spec3": "Jjg,JjKk->Kkg",
        "spec4": "Kkg,gh->Kkh",
        "X": (np.arange(nt, dtype=np.int32)[:, None], (nt,), X),
        "Y": (ky, by, ty),
        "W1": (nokey, (), W1[None]),
        "W2": (nokey, (), W2[None]),
        "edges": (src, dst),
        "n": n,
        "t": t,
    }


def zipf_coords(n: int, nnz: int, order=3, s=1.1, seed=0, device="cpu", batch=1 << 23):
    """nnz distinct order-`order` coordinates over [0, n)^order, each mode
    drawn independently from a Zipf law over ranks 1..n (P(rank) ~ rank^-s,
    index = rank - 1); draws continue until nnz distinct coordinates have
    appeared and the first nnz in draw order are kept.  Returns the sorted
    row-major codes (int64 tensor on `device`)."""
    g = torch.Generator(device=device).manual_seed(seed)
    w = torch.arange(1, n + 1, dtype=torch.float64, device=device) ** -s
    cdf = torch.cumsum(w, 0)
    cdf = cdf / cdf[-1]
    draws = []
    while True:
        m = batch if draws else max(1024, min(batch, int(nnz * 1.3)))
        code = torch.zeros(m, dtype=torch.int64, device=device)
        for _ in range(order):
            u = torch.rand(m, generator=g, device=device, dtype=torch.float64)
            code = code * n + torch.searchsorted(cdf, u, right=True).clamp_(max=n - 1)
        draws.append(code)
        if torch.unique(torch.cat(draws)).numel() >= nnz:
            break
    allc = torch.cat(draws)
    uniq, inv = torch.unique(allc, return_inverse=True)
    pos = torch.arange(allc.numel(), device=device)
    first = torch.full((uniq.numel(),), allc.numel(), dtype=torch.int64, device=device)
    first.scatter_reduce_(0, inv, pos, reduce="amin")
    keep = torch.argsort(first)[:nnz]
    return torch.sort(uniq[keep]).values


def mttkrp(seed=0, n=100_000, nnz=10_000_000, t=16, rank=64, s=1.1, device="cpu", layout="ijk"):
    """MTTKRP M[i,r] = sum_{j,k} T[i,j,k] B[j,r] C[k,r]: T sparse n^3 with nnz
    Zipf(s) coordinates (zipf_coords), values U[-1,1), grouped into only-
    nonempty t^3 bf16 tiles keyed (I, J, K); B and C dense n x rank bf16
    U[-1,1) as per-tile-row relations keyed J (resp. K) with [t x rank] tiles
    (rows past n zero).  Spec "IJKijk,Jjr,Kkr->Iir"; layout="kij" stores each
    T tile as [k][i][j] instead (spec "IJKkij,Jjr,Kkr->Iir", the same EinSum
    and the same values)."""
    if layout not in ("ijk", "kij"):
        raise ValueError("layout must be 'ijk' or 'kij'")
    codes = zipf_coords(n, nnz, 3, s, seed, device)
    g = torch.Generator(device=device).manual_seed(seed + 1)
    vals = torch.rand(codes.numel(), generator=g, device=device) * 2 - 1
    i, j, k = codes // (n * n), (codes // n) % n, codes % n
    nt = -(-n // t)
    tcode = ((i // t) * nt + j // t) * nt + k // t
    ukeys, inv = torch.unique(tcode, return_inverse=True)
    tiles = torch.zeros((ukeys.numel(), t, t, t), dtype=torch.bfloat16, device=device)
    tiles[inv, i % t, j % t, k % t] = vals.to(torch.bfloat16)
    keys = torch.stack([ukeys // (nt * nt), (ukeys // nt) % nt, ukeys % nt], 1).to(torch.int32).cpu().numpy()

    def factor():
        f = torch.zeros((nt * t, rank), device=device)
        f[:n] = torch.rand((n, rank), generator=g, device=device) * 2 - 1
        return (np.arange(nt, dtype=np.int32)[:, None], (nt,), f.view(nt, t, rank).to(torch.bfloat16))

    if layout == "kij":
        tiles = tiles.permute(0, 3, 1, 2).contiguous()
    return {
        "spec": "IJKijk,Jjr,Kkr->Iir" if layout == "ijk" else "IJKkij,Jjr,Kkr->Iir",
        "T": (keys, (nt, nt, nt), tiles),
        "B": factor(),
        "C": factor(),
        "coords": codes,
        "n": n,
        "t": t,
    }


def graph_attention(seed=0, n=3327, feat=3703, feat_nnz=32, edges=9104, dk=1024, device="cpu"):
    """Sparse attention of a graph transformer, shaped like the paper's
    Planetoid.CiteSeer experiment (3327 nodes, 3703 bag-of-words features,
    9104 directed edge entries, 1024-wide projections).

    X: 0/1 bag-of-words, ``feat_nnz`` distinct features per node drawn
    uniformly, as scalar tuples keyed (node, feature); WQ, WK: feat x dk bf16
    N(0, 1/feat), one dk-vector per feature; A: ``edges`` / 2 distinct
    undirected node pairs (no self-loops) drawn uniformly, both directions,
    value 1, keyed (node, node).

    The chain (the schema of the paper's table of UCL EinSums, then row
    softmax over the neighbours present as four extended EinSums):
      T0 = IM,Mk->Ik   T1 = JN,Nk->Jk   T2 = Ik,IJ->IJk   T3 = IJk,Jk->IJ
      Attn = IJ->IJ scaled by 1/sqrt(dk)
      M = max_J Attn; S = exp(Attn - M); D = sum_J S; P = S / D."""
    rng = np.random.default_rng(seed)
    rows = np.repeat(np.arange(n), feat_nnz)
    cols = np.concatenate([rng.choice(feat, size=feat_nnz, replace=False) for _ in range(n)])
    xk = np.stack([rows, cols], axis=1).astype(np.int32)
    xk = xk[np.lexsort((xk[:, 1], xk[:, 0]))]
    X = (xk, (n, feat), torch.ones(len(xk), dtype=torch.bfloat16, device=device))
    g = torch.Generator().manual_seed(seed)

    def proj():
        w = (torch.randn((feat, dk), generator=g) / math.sqrt(feat)).to(torch.bfloat16)
        return (np.arange(feat, dtype=np.int32)[:, None], (feat,), w.to(device))

    want = edges // 2
    pairs = set()
    while len(pairs) < want:
        a, b = rng.integers(0, n, size=2 * (want - len(pairs)) + 16).reshape(-1, 2).T
        for x, y in zip(a.tolist(), b.tolist()):
            if x != y and len(pairs) < want:
                pairs.add((min(x, y), max(x, y)))
    e = np.array(sorted(pairs), dtype=np.int64)
    ak = np.concatenate([e, e[:, ::-1]]).astype(np.int32)
    ak = ak[np.lexsort((ak[:, 1], ak[:, 0]))]
    A = (ak, (n, n), torch.ones(len(ak), dtype=torch.bfloat16, device=device))
    chain = [
        ("T0", "IM,Mk->Ik", ["XQ", "WQ"], {"out_dtype": "bf16"}),
        ("T1", "JN,Nk->Jk", ["XK", "WK"], {"out_dtype": "bf16"}),
        ("T2", "Ik,IJ->IJk", ["T0", "A"], {"out_dtype": "bf16"}),
        ("T3", "IJk,Jk->IJ", ["T2", "T1"], {"out_dtype": "f32"}),
        ("Attn", "IJ->IJ", ["T3"], {"out_dtype": "f32", "scale": 1.0 / math.sqrt(dk)}),
        ("M", "IJ->I", ["Attn"], {"out_dtype": "f32", "agg": "max"}),
        ("S", "IJ,I->IJ", ["Attn", "M"], {"out_dtype": "f32", "comb": "sub", "map": "exp"}),
        ("D", "IJ->I", ["S"], {"out_dtype": "f32"}),
        ("P", "IJ,I->IJ", ["S", "D"], {"out_dtype": "f32", "comb": "div"}),
    ]
    return {"X": X, "XQ": X, "XK": X, "WQ": proj(), "WK": proj(), "A": A, "chain": chain, "n": n, "dk": dk}


def to_oracle(rel):
    """(keys, bounds, tiles) with tiles converted exactly to float64 numpy."""
    keys, bounds, tiles = rel
    return keys, bounds, tiles.detach().to("cpu", torch.float64).numpy()
