"""Oracle for repartitioning a tensor-relation (test infrastructure only).

Changing the upper/lower split of a relation between two EinSums (paper
Sec. 5, the third step of compiling an EinSum DAG) happens in two steps:

  1. decompose: every tuple is split along each label that turns from lower
     to upper, one sub-tuple per index value of that label over its whole
     range (the ALLINTS table function), carrying the sub-tensor at that
     index;
  2. aggregate: the sub-tuples are grouped by the output's upper labels and
     the labels that turn from upper to lower are stacked into new tile
     dimensions at the positions given by their key values (the STACK
     aggregate); positions no sub-tuple fills are zero.

This module follows those two steps tuple at a time, in fp64, with no
blocking or fusion.  Only the tests, ``__graft_entry__.smoke`` and the CPU leg
of ``bench.py`` may use it; it shares nothing with the GPU executor.

Spec: ``"<input labels>-><output labels>"``, one letter per label, the case
of a letter giving its class on that side (upper = key column, lower = tile
dimension, in the order the letters appear).  A label is the same letter on
both sides, compared without case, so one side may not hold two letters that
differ only in case.
"""
from __future__ import annotations

import itertools

import numpy as np


class RepartitionError(ValueError):
    pass


def _parse(spec, u, r):
    if "->" not in spec:
        raise RepartitionError("spec has no '->'")
    lhs, rhs = spec.split("->", 1)
    for side in (lhs, rhs):
        if not side.isalpha() and side != "":
            raise RepartitionError("labels must be letters")
        low = side.lower()
        if len(set(low)) != len(low):
            raise RepartitionError("a label appears twice on one side")
    if sorted(lhs.lower()) != sorted(rhs.lower()):
        raise RepartitionError("both sides must hold the same labels")
    in_up = [c.lower() for c in lhs if c.isupper()]
    in_low = [c for c in lhs if c.islower()]
    if len(in_up) != u or len(in_low) != r:
        raise RepartitionError("input side does not match the relation's key/tile arity")
    out_up = [c.lower() for c in rhs if c.isupper()]
    out_low = [c for c in rhs if c.islower()]
    return in_up, in_low, out_up, out_low


def repartition(spec, rel):
    """Repartition ``rel = (keys int32 [n, u], bounds, tiles [n, ...])``
    (tiles as a float64 numpy array) as ``spec`` says.  Returns
    ``(keys, bounds, tiles)`` with keys in ascending lexicographic order."""
    keys, bounds, tiles = rel
    keys = np.asarray(keys, dtype=np.int64).reshape(len(tiles), -1) if len(tiles) else np.zeros((0, len(bounds)), np.int64)
    tiles = np.asarray(tiles, dtype=np.float64)
    n = tiles.shape[0]
    in_up, in_low, out_up, out_low = _parse(spec, len(bounds), tiles.ndim - 1)
    ext = {}
    for c, b in zip(in_up, bounds):
        ext[c] = int(b)
    for c, e in zip(in_low, tiles.shape[1:]):
        ext[c] = int(e)

    # step 1 -- decompose along the labels that become upper (ALLINTS)
    promoted = [c for c in in_low if c in out_up]
    kept_low = [c for c in in_low if c not in out_up]
    sub = []   # (label -> key value, sub-tensor over kept_low in input order)
    for t in range(n):
        for vals in itertools.product(*[range(ext[c]) for c in promoted]):
            key = {c: int(keys[t, q]) for q, c in enumerate(in_up)}
            key.update(zip(promoted, vals))
            index = tuple(key[c] if c in promoted else slice(None) for c in in_low)
            sub.append((key, tiles[t][index] if in_low else tiles[t]))

    # step 2 -- group by the output's upper labels and stack the labels that
    # become lower (STACK); unfilled positions stay zero
    out_shape = [ext[c] for c in out_low]
    groups = {}
    for key, s in sub:
        g = tuple(key[c] for c in out_up)
        tile = groups.get(g)
        if tile is None:
            tile = groups[g] = np.zeros(out_shape)
        # s's axes are kept_low in input order; place them in output order
        s = np.transpose(s, [kept_low.index(c) for c in out_low if c in kept_low]) if kept_low else s
        index = tuple(key[c] if c not in kept_low else slice(None) for c in out_low)
        tile[index] = s
    order = sorted(groups)
    out_keys = np.array(order, dtype=np.int32).reshape(len(order), len(out_up))
    out_tiles = np.array([groups[g] for g in order]).reshape([len(order)] + out_shape)
    return out_keys, tuple(ext[c] for c in out_up), out_tiles
