"""Oracle for repartitioning a tensor-relation (test infrastructure only).

Changing the upper/lower split of a relation between two EinSums (paper
Sec. 6, the third step of compiling an EinSum DAG) happens in two steps:

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

Spec: ``"<input labels>-><output>"``.  The input side lists the relation's
labels, one letter each, upper case for key columns and lower case for tile
dimensions, in order.  The output side is either ``"<keys>|<tile dims>"``,
the input's letters as written, or the same letters with their case changed
to give the new class (letters then compare without case, so that form needs
no two input letters that differ only in case).
"""
from __future__ import annotations

import itertools

import numpy as np


class RepartitionError(ValueError):
    pass


def _parse(spec, u, r):
    """Labels are named by their input-side letter.  Returns the input's
    upper and lower labels and the output's, each in order."""
    if "->" not in spec:
        raise RepartitionError("spec has no '->'")
    lhs, rhs = spec.split("->", 1)
    if not lhs.isalpha() and lhs != "":
        raise RepartitionError("labels must be letters")
    if len(set(lhs)) != len(lhs):
        raise RepartitionError("a label appears twice on the input side")
    in_up = [c for c in lhs if c.isupper()]
    in_low = [c for c in lhs if c.islower()]
    if len(in_up) != u or len(in_low) != r:
        raise RepartitionError("input side does not match the relation's key/tile arity")
    if "|" in rhs:
        # explicit form: output keys | output tile dims, input letters as written
        up, low = rhs.split("|", 1)
        out = up + low
        if (out and not out.isalpha()) or sorted(out) != sorted(lhs):
            raise RepartitionError("both sides must hold the same labels")
        return in_up, in_low, list(up), list(low)
    # case form: the letter's case gives its output class; letters compare without case
    if not rhs.isalpha() and rhs != "":
        raise RepartitionError("labels must be letters")
    if len(set(lhs.lower())) != len(lhs) or len(set(rhs.lower())) != len(rhs):
        raise RepartitionError("a label appears twice on one side (letters compare without case)")
    if sorted(lhs.lower()) != sorted(rhs.lower()):
        raise RepartitionError("both sides must hold the same labels")
    name = {c.lower(): c for c in lhs}
    return in_up, in_low, [name[c.lower()] for c in rhs if c.isupper()], [name[c.lower()] for c in rhs if c.islower()]


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
