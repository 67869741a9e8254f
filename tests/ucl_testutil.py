"""Test helpers: build tensor-relations from dense arrays and back.

A dense tensor with axes named by lower-case letters is decomposed into a
tensor-relation by promoting a chosen set of labels (Sec. 4.2): one tuple per
combination of promoted indices, whose tile is the sub-tensor over the
remaining labels; all-zero tiles are dropped (zero-tuple elimination, Sec. 4.2).
"""
from __future__ import annotations

import itertools
import string

import numpy as np


def golden(path):
    """Parse tests/golden/*.txt: '[name]' sections of whitespace-separated numbers."""
    sec, out = None, {}
    for line in open(path):
        line = line.split("#", 1)[0].strip()
        if not line:
            continue
        if line.startswith("["):
            sec = line.strip("[]").strip()
            out[sec] = []
            continue
        out[sec].append([float(x) for x in line.split()])
    return {k: np.array(v) for k, v in out.items()}


def ucl_operand(dense_labels: str, promoted: set) -> str:
    return "".join(c.upper() if c in promoted else c for c in dense_labels)


def decompose(dense: np.ndarray, labels: str, promoted: set, drop_zero=True):
    """Dense array with axes `labels` -> (keys int32[n,u], bounds, tiles[n,...])."""
    up_axes = [a for a, c in enumerate(labels) if c in promoted]
    low_axes = [a for a, c in enumerate(labels) if c not in promoted]
    perm = up_axes + low_axes
    t = np.transpose(dense, perm)
    up_shape = [dense.shape[a] for a in up_axes]
    low_shape = [dense.shape[a] for a in low_axes]
    keys, tiles = [], []
    for idx in itertools.product(*[range(b) for b in up_shape]):
        tile = t[idx] if idx else t
        if drop_zero and not np.any(tile):
            continue
        keys.append(idx)
        tiles.append(np.array(tile, dtype=np.float64).reshape(low_shape))
    n = len(tiles)
    keys = np.array(keys, dtype=np.int32).reshape(n, len(up_axes))
    tiles = np.array(tiles, dtype=np.float64).reshape([n] + low_shape)
    return keys, np.array(up_shape, dtype=np.int64), tiles


def recompose(keys, tiles, out_labels: str, promoted: set, extents: dict):
    """Inverse of decompose for the output relation (missing tuples read as 0)."""
    up = [c for c in out_labels if c in promoted]
    low = [c for c in out_labels if c not in promoted]
    full = np.zeros([extents[c] for c in up + low], dtype=np.float64)
    for k, tile in zip(keys, tiles):
        full[tuple(int(x) for x in k)] = tile
    # axes are (up..., low...): move them back to out_labels order
    order = up + low
    return np.transpose(full, [order.index(c) for c in out_labels])


def brute_force(spec: str, arrays):
    """The EinSum definition (Sec. 3, Eq. Einsum) by enumeration of every label
    assignment in pure Python: W[l_W] += prod_k U_k[l_k].  Tiny inputs only."""
    lhs, out = spec.split("->")
    ops = lhs.split(",")
    ext = {}
    for op, a in zip(ops, arrays):
        for c, e in zip(op, a.shape):
            ext[c] = e
    labels = sorted(ext)
    W = np.zeros([ext[c] for c in out], dtype=np.float64)
    for vals in itertools.product(*[range(ext[c]) for c in labels]):
        env = dict(zip(labels, vals))
        p = 1.0
        for op, a in zip(ops, arrays):
            p *= float(a[tuple(env[c] for c in op)])
        W[tuple(env[c] for c in out)] += p
    return W


def random_sparse(rng, shape, density=0.5, block_axes=()):
    """Random dense array with whole slices zeroed along `block_axes`, so that
    tile elimination is exercised."""
    a = rng.standard_normal(shape)
    mask = rng.random(shape) < density
    a = a * mask
    for ax in block_axes:
        kill = rng.random(shape[ax]) < 0.3
        idx = [slice(None)] * len(shape)
        idx[ax] = kill
        a[tuple(idx)] = 0.0
    return a


LETTERS = string.ascii_lowercase
