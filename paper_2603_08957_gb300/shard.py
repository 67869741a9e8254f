"""Multi-GPU execution of UCL EinSum chains by output-key range.

One process per GPU.  Sec. 5 evaluates a UCL EinSum as SUM ... GROUP BY the
output's upper labels, so output tuples with different keys never combine:
cutting the output-key space into contiguous ranges, one per rank, splits an
EinSum into independent EinSums whose results are disjoint and need no
reduction.  For each EinSum of a chain:

  * the partition label L is the output's leading upper label (the most
    significant field of the packed output key, so a contiguous range of L
    is a contiguous range of output keys and the ranks' results concatenate
    in rank order into the single-GPU result);
  * an operand that holds L is co-partitioned: each rank keeps its tuples
    whose L lies in the rank's range (a local row selection, no transfer);
  * an operand that does not hold L is replicated on every rank; a
    replicated operand that is itself a partitioned result of an earlier
    EinSum is all-gathered first -- the only exchange step of the path
    (the layer boundary of a GNN: H1 keyed by destination block is read,
    keyed by source block, by the next message passing);
  * ranges are balanced by joined-pair count: each partitioned tuple weighs
    the number of tuples it joins with in the replicated operands, and the
    cut points are prefix-sum quantiles over the values of L.

Sec. 7.2 charges a repartition C_xfer per byte moved; here the moved bytes
are the all-gathered operands only.  The relations handled here are plain
tuples (keys int32 [n, u], bounds, tiles [n, ...]) of torch tensors on any
device; the EinSum itself is a callable (the GPU executor on a GPU rank), so
that this host logic is the same on every backend torch.distributed offers.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch


@dataclass
class Part:
    """How a relation is spread over the ranks: `col` is the key column whose
    value ranges split it (None: every rank holds all of it), `cuts` the
    range boundaries over that column's values (rank r holds
    [cuts[r], cuts[r + 1]))."""
    col: int | None = None
    cuts: tuple | None = None


def _parse(spec):
    lhs, out = spec.split("->")
    return lhs.split(","), out


def leading_upper(out):
    for c in out:
        if c.isupper():
            return c
    return None


def balanced_cuts(weights, world):
    """Boundaries 0 = c_0 <= ... <= c_world = len(weights) over the values of
    the partition label: rank r takes values [c_r, c_{r+1}) and about
    sum(weights) / world of the weight."""
    w = np.asarray(weights, dtype=np.float64)
    n = len(w)
    pre = np.concatenate([[0.0], np.cumsum(w)])
    total = pre[-1]
    cuts = [0]
    for r in range(1, world):
        cuts.append(int(np.searchsorted(pre, total * r / world, side="left")))
    cuts.append(n)
    for r in range(1, len(cuts)):   # monotone even when weights are zero
        cuts[r] = max(cuts[r], cuts[r - 1])
    return tuple(cuts)


def _codes(keys, cols, bounds):
    """Mixed-radix code of the given key columns (lexicographic order)."""
    keys = np.asarray(keys, dtype=np.int64)
    code = np.zeros(keys.shape[0], dtype=np.int64)
    for c in cols:
        code = code * int(bounds[c]) + keys[:, c]
    return code


def pair_weights(spec, keys, bounds, part_op):
    """Joined-tuple count of each tuple of operand `part_op`: the product,
    over the other operands, of the number of their tuples that agree with it
    on the labels they share (exact for binary EinSums and star joins)."""
    ops, _ = _parse(spec)
    mine = [c for c in ops[part_op] if c.isupper()]
    km = np.asarray(keys[part_op]).reshape(-1, len(mine))
    w = np.ones(km.shape[0], dtype=np.float64)
    for k, op in enumerate(ops):
        if k == part_op:
            continue
        ups = [c for c in op if c.isupper()]
        kk = np.asarray(keys[k]).reshape(-1, len(ups))
        shared = [c for c in ups if c in mine]
        if not shared:
            w *= kk.shape[0]
            continue
        other = _codes(kk, [ups.index(c) for c in shared], bounds[k])
        me = _codes(km, [mine.index(c) for c in shared], bounds[part_op])
        u, cnt = np.unique(other, return_counts=True)
        if len(u) == 0:
            w *= 0.0
            continue
        pos = np.minimum(np.searchsorted(u, me), len(u) - 1)
        w *= np.where(u[pos] == me, cnt[pos], 0)
    return w


def rows_in_range(keys, col, lo, hi):
    k = keys[:, col]
    return (k >= lo) & (k < hi)


def select(rel, mask):
    keys, bounds, tiles = rel
    m = torch.as_tensor(np.asarray(mask), device=keys.device)
    return keys[m].contiguous(), bounds, tiles[m.to(tiles.device)].contiguous()


class ShardedChain:
    """Runs a chain of UCL EinSums over `world` ranks by output-key range.

    einsum(spec, rels, **opts) -> (keys, bounds, tiles) evaluates one EinSum
    on this rank's device; group is the torch.distributed process group (None:
    the default one).  Relations stay on the device of their tensors."""

    def __init__(self, rank, world, einsum, group=None):
        self.rank, self.world, self.einsum = rank, world, einsum
        self.group = group
        self.gathered_bytes = 0   # bytes this rank received by all-gathers

    # ----------------------------------------------------------- exchange
    def allgather(self, rel):
        """Concatenate every rank's part of a partitioned relation, in rank
        order (ascending keys when the parts are contiguous key ranges)."""
        import torch.distributed as dist
        keys, bounds, tiles = rel
        n = torch.tensor([keys.shape[0]], dtype=torch.int64, device=keys.device)
        ns = [torch.zeros_like(n) for _ in range(self.world)]
        dist.all_gather(ns, n, group=self.group)
        ns = [int(x.item()) for x in ns]
        m = max(ns)

        def gather(t):
            pad = torch.zeros((m,) + tuple(t.shape[1:]), dtype=t.dtype, device=t.device)
            pad[: t.shape[0]] = t
            if pad.dtype == torch.bfloat16 and pad.device.type == "cpu":
                # gloo has no bf16: move the bit patterns as bytes
                raw = pad.view(torch.uint8)
                outs = [torch.empty_like(raw) for _ in range(self.world)]
                dist.all_gather(outs, raw, group=self.group)
                outs = [o.view(torch.bfloat16) for o in outs]
            else:
                outs = [torch.empty_like(pad) for _ in range(self.world)]
                dist.all_gather(outs, pad, group=self.group)
            return torch.cat([o[:c] for o, c in zip(outs, ns)])

        k, t = gather(keys), gather(tiles)
        per_tuple = keys.shape[1] * 4 + int(np.prod(tiles.shape[1:])) * tiles.element_size()
        self.gathered_bytes += sum(ns[r] for r in range(self.world) if r != self.rank) * per_tuple
        return k.contiguous(), bounds, t.contiguous()

    # -------------------------------------------------------------- chain
    def cuts_for(self, spec, rels, part_op, col):
        keys = [r[0].cpu().numpy() for r in rels]
        bounds = [tuple(int(b) for b in r[1]) for r in rels]
        w = pair_weights(spec, keys, bounds, part_op)
        L = int(bounds[part_op][col])
        per_value = np.bincount(keys[part_op][:, col], weights=w, minlength=L) if len(w) else np.zeros(L)
        return balanced_cuts(per_value, self.world)

    def run(self, chain, inputs):
        """chain: [(name, spec, input names, opts)]; inputs: name -> full
        relation (every rank passes the same inputs).  Returns name ->
        (relation part held by this rank, Part)."""
        env = {k: (v, Part()) for k, v in inputs.items()}
        for name, spec, ins, opts in chain:
            ops, out = _parse(spec)
            L = leading_upper(out)
            rels = []
            holders = [k for k, op in enumerate(ops) if L is not None and L in op]
            # the partition of this EinSum: reuse the cuts of a holder that is
            # already partitioned on L's column, else balance a new cut
            cuts, col_of = None, {}
            for k in holders:
                col_of[k] = [c for c in ops[k] if c.isupper()].index(L)
            for k in holders:
                rel, part = env[ins[k]]
                if part.col is not None and part.col == col_of[k]:
                    cuts = part.cuts
                    break
            full = []
            for k, op in enumerate(ops):
                rel, part = env[ins[k]]
                if part.col is not None and (k not in holders or part.col != col_of[k] or part.cuts != cuts):
                    rel = self.allgather(rel)      # exchange: every rank needs all of it
                    part = Part()
                full.append((rel, part))
            if L is None or self.world == 1:
                res = self.einsum(spec, [r for r, _ in full], **opts)
                env[name] = (res, Part())
                continue
            if cuts is None:
                k0 = holders[0]
                cuts = self.cuts_for(spec, [r for r, _ in full], k0, col_of[k0])
            lo, hi = cuts[self.rank], cuts[self.rank + 1]
            for k, (rel, part) in enumerate(full):
                if k in holders and part.col is None:
                    rel = select(rel, rows_in_range(rel[0].cpu().numpy(), col_of[k], lo, hi))
                rels.append(rel)
            res = self.einsum(spec, rels, **opts)
            env[name] = (res, Part(col=0, cuts=cuts))
        return env

    def gather_result(self, entry):
        """The whole relation of a run() result, on every rank."""
        rel, part = entry
        return rel if part.col is None else self.allgather(rel)
