"""Run a tree of binary EinSums under a plan chosen by ``plan`` (ucl_plan),
or a DAG under a plan chosen by ``plan_dag`` (ucl_plan_dag).

The program is the one handed to the planner: vertices in topological order, each
an input tensor or W = Σ U × V, every label one lower-case letter.  A plan
gives every tensor's split (its promoted labels).  In the executor's spec
grammar a promoted label is written upper case, so the plan alone fixes every
spec string (paper Sec. 6, steps 1 and 2 of compiling an EinSum DAG):

* an input is brought into the split its consumer reads: ucl_repartition
  from the split it is stored in, then ucl_drop_zero_tiles;
* every EinSum is one ucl_einsum, its operands' and output's letters cased by
  the plan;
* a tensor whose producer and consumer split it differently is repartitioned
  between the two (step 3), and its all-zero tuples dropped.

A relation of a tensor with labels ``l`` and split ``up`` holds its key
columns in the order the promoted labels appear in ``l`` and its tile
dimensions in the order of the others.  Every step runs in the library; this
module only writes the spec strings.
"""
from __future__ import annotations


def cased(labels: str, up: str) -> str:
    """Spec letters of a tensor under a split: promoted labels upper case."""
    return "".join(c.upper() if c in up else c for c in labels)


def repartition_spec(labels: str, up_from: str, up_to: str) -> str:
    """ucl_repartition spec (explicit form) from one split to another."""
    src = cased(labels, up_from)
    keys = "".join(x for c, x in zip(labels, src) if c in up_to)
    tiles = "".join(x for c, x in zip(labels, src) if c not in up_to)
    return f"{src}->{keys}|{tiles}"


def einsum_spec(lU: str, upU: str, lV: str, upV: str, lW: str, upW: str) -> str:
    return f"{cased(lU, upU)},{cased(lV, upV)}->{cased(lW, upW)}"


def _same(a: str, b: str) -> bool:
    return set(a) == set(b)


def resplit(ctx, rel, labels: str, up_from: str, up_to: str, drop_zero: bool = True):
    """``rel`` (split ``up_from``) in split ``up_to``; ``rel`` itself when the
    two promote the same labels."""
    if _same(up_from, up_to):
        return rel
    out = ctx.repartition(repartition_spec(labels, up_from, up_to), rel)
    if drop_zero:
        dense = out
        out = ctx.drop_zero_tiles(dense)
        dense.destroy()
    return out


def prepare_inputs(ctx, vertices, ups, stored):
    """Each input vertex i, stored as (relation, split), in the split the plan
    reads it in (``ups[i]``).  Returns {i: relation}."""
    out = {}
    for i, v in enumerate(vertices):
        if v.get("left") is None:
            rel, up = stored[i]
            out[i] = resplit(ctx, rel, v["labels"], up, ups[i])
    return out


def execute_dag(ctx, vertices, ups, inputs, *, path="auto", keep=False):
    """Evaluate a program whose tensors may be consumed more than once under
    one plan (``ups`` as ``plan`` or ``plan_dag`` return it; ``inputs`` maps
    each input vertex to its relation in ``ups[i]``).  Every consuming edge
    reads its tensor in the split its consumer wants, repartitioning a copy
    when the tensor has another split.  An intermediate is destroyed after
    its last consumer ran, unless ``keep``.  Returns {vertex: relation} for
    every EinSum vertex no EinSum consumes (the program's outputs)."""
    uses = [0] * len(vertices)
    for v in vertices:
        if v.get("left") is not None:
            uses[v["left"]] += 1
            uses[v["right"]] += 1
    pending = list(uses)
    rel = dict(inputs)
    for i, v in enumerate(vertices):
        if v.get("left") is None:
            continue
        upW, upU, upV = ups[i]
        operands, copies = [], []
        for child, up_read in ((v["left"], upU), (v["right"], upV)):
            cv = vertices[child]
            up_have = ups[child] if cv.get("left") is None else ups[child][0]
            r = resplit(ctx, rel[child], cv["labels"], up_have, up_read)
            if r is not rel[child]:
                copies.append(r)
            operands.append(r)
        spec = einsum_spec(vertices[v["left"]]["labels"], upU, vertices[v["right"]]["labels"], upV, v["labels"], upW)
        out_dtype = "bf16" if v.get("dtype_bytes", 2) == 2 else "f32"
        rel[i] = ctx.einsum(spec, *operands, out_dtype=out_dtype, path=path)
        for r in copies:
            r.destroy()
        for child in (v["left"], v["right"]):
            pending[child] -= 1
            if pending[child] == 0 and not keep and vertices[child].get("left") is not None:
                rel.pop(child).destroy()
    return {i: rel[i] for i, v in enumerate(vertices) if v.get("left") is not None and uses[i] == 0}


def execute(ctx, vertices, ups, inputs, *, path="auto", keep=False):
    """Evaluate the tree under one plan.  ``ups`` is a plan as ``plan``
    returns it; ``inputs`` maps each input vertex to its relation in the
    plan's split.  Returns the root's relation (and every intermediate
    relation is destroyed once consumed, unless ``keep``)."""
    rel = dict(inputs)
    for i, v in enumerate(vertices):
        if v.get("left") is None:
            continue
        upW, upU, upV = ups[i]
        operands = []
        for child, up_read in ((v["left"], upU), (v["right"], upV)):
            cv = vertices[child]
            up_have = ups[child] if cv.get("left") is None else ups[child][0]
            r = resplit(ctx, rel[child], cv["labels"], up_have, up_read)
            if r is not rel[child] and cv.get("left") is not None and not keep:
                rel[child].destroy()
            operands.append(r)
        spec = einsum_spec(vertices[v["left"]]["labels"], upU, vertices[v["right"]]["labels"], upV, v["labels"], upW)
        out_dtype = "bf16" if v.get("dtype_bytes", 2) == 2 else "f32"
        rel[i] = ctx.einsum(spec, *operands, out_dtype=out_dtype, path=path)
        if not keep:
            for child, r in zip((v["left"], v["right"]), operands):
                if vertices[child].get("left") is not None:
                    r.destroy()
    return rel[len(vertices) - 1]
