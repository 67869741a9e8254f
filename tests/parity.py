"""Parity helpers: compare an output relation of the GPU executor with the
oracle's result for the same inputs.

The bar (per output entry, Sigma|a*b| = the oracle's magnitude sum):
  keys: bit-exact, same order;
  values: |gpu - oracle| <= tol * |scale| * Sigma|a*b|, tol = 1e-2 for bf16
  inputs (fp32 accumulate) and 1e-5 for fp32 inputs, plus the output cast
  when the output is bf16; entries with Sigma|a*b| = 0 are exactly 0;
  non-finite oracle entries (the extended EinSum's division by zero) must be
  matched exactly: NaN where the oracle has NaN, the same infinity where it
  has one, and a finite GPU value wherever the oracle's is finite.

The cast term.  One round-to-nearest-even cast to bf16 (8 significant bits)
errs by at most the unit roundoff 2^-8 times the magnitude of the value cast:
1 + 2^-8 lies halfway between the neighbours 1 and 1 + 2^-7 and rounds to 1,
an error of 2^-8 / (1 + 2^-8) of the value.  The value cast is the fp32 sum,
which lies within the accumulation bound of the oracle's, so the cast term
is 2^-8 * (|oracle| + accumulation bound).
"""
from __future__ import annotations

import numpy as np
import torch

import oracle

TOL = {torch.bfloat16: 1e-2, torch.float32: 1e-5}
BF16_CAST = 2.0**-8


def gpu_rel(ctx, rel, copy=False):
    keys, bounds, tiles = rel
    dev = torch.device("cuda", ctx.device)
    return ctx.relation(torch.as_tensor(keys).to(dev), bounds, tiles.to(dev), copy=copy)


def oracle_ref(spec, rels, *, epi="none", scale=1.0, sample_keys=None, **ext):
    """Oracle result with the epilogue applied in fp64 (no output cast);
    ``ext`` passes the extended EinSum's agg / comb / map."""
    ins = [(k, b, t.detach().to("cpu", torch.float64).numpy() if torch.is_tensor(t) else t) for k, b, t in rels]
    return oracle.einsum(spec, ins, epi=epi, scale=scale, out_dtype="f64", sample_keys=sample_keys, **ext)


def _widen(t):
    """Tile array as sent to a worker: bf16 travels as its raw 16-bit
    patterns (half the bytes) and is widened exactly here."""
    if isinstance(t, tuple) and t[0] == "bf16":
        return (t[1].astype(np.uint16).astype(np.uint32) << 16).view(np.float32)
    return t


def _oracle_task(task):
    spec, rels, kw = task
    return oracle.einsum(spec, [(k, b, _widen(t)) for k, b, t in rels], out_dtype="f64", **kw)


def _to_worker(t):
    if torch.is_tensor(t) and t.dtype == torch.bfloat16:
        return ("bf16", t.detach().contiguous().view(torch.int16).cpu().numpy())
    return t.detach().to("cpu", torch.float32).numpy() if torch.is_tensor(t) else np.asarray(t, np.float32)


def oracle_parallel(tasks):
    """oracle_ref for several independent (spec, rels, kwargs) tasks at once,
    one spawned process each (never a fork of a process holding a CUDA
    context).  Tiles reach the oracle as float32 (bf16 and fp32 inputs are
    exact in float32); results come back in task order."""
    import multiprocessing as mpc
    import os
    conv = []
    for spec, rels, kw in tasks:
        ins = [(np.asarray(k), tuple(int(x) for x in b), _to_worker(t)) for k, b, t in rels]
        conv.append((spec, ins, kw))
    n = max(1, min(len(conv), os.cpu_count() or 1))
    with mpc.get_context("spawn").Pool(n) as pool:
        return pool.map(_oracle_task, conv, chunksize=1)


def check_values(g, want, mag, in_dtype, out_bf16, scale=1.0):
    """Element-wise value bar on arrays: g (GPU, float64), want and mag (the
    oracle's value and Sigma|a*b|).  Raises AssertionError on the first
    violation; returns the largest error relative to |scale| * Sigma|a*b|."""
    g = np.asarray(g, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    mag = np.asarray(mag, dtype=np.float64)
    assert g.shape == want.shape == mag.shape, (g.shape, want.shape, mag.shape)
    fin_w, fin_g = np.isfinite(want), np.isfinite(g)
    if not np.array_equal(fin_w, fin_g):
        i = tuple(np.argwhere(fin_w != fin_g)[0])
        raise AssertionError(f"finite / non-finite pattern differs; first at {i}: gpu={g[i]!r} oracle={want[i]!r}")
    nf = ~fin_w
    if nf.any():
        same = (np.isnan(g[nf]) & np.isnan(want[nf])) | (g[nf] == want[nf])
        if not same.all():
            i = tuple(np.argwhere(nf)[np.argmin(same)])
            raise AssertionError(f"non-finite entry differs at {i}: gpu={g[i]!r} oracle={want[i]!r}")
    gf, wf, mf = g[fin_w], want[fin_w], mag[fin_w]
    acc = TOL[in_dtype] * abs(scale) * mf
    bound = acc + BF16_CAST * (np.abs(wf) + acc) if out_bf16 else acc
    zero = mf == 0
    if not np.all(gf[zero] == 0):
        raise AssertionError("entries with no contribution must be exactly zero")
    err = np.abs(gf - wf)
    bad = ~(err <= bound)
    if bad.any():
        j = int(np.argmax(bad))
        i = tuple(np.argwhere(fin_w)[j])
        raise AssertionError(f"{int(bad.sum())} entries out of tolerance; first at {i}: gpu={g[i]!r} "
                             f"oracle={want[i]!r} sum|ab|={mag[i]!r} bound={bound[j]!r}")
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(mf > 0, err / (abs(scale) * mf), 0.0)
    return float(r.max()) if r.size else 0.0


def assert_parity(out_rel, ref, in_dtype, *, scale=1.0, select=None):
    """Check a GPU output relation against an oracle result.  `select`
    (indices into the GPU output) restricts the value check to sampled keys,
    whose oracle result `ref` then holds exactly those keys in that order."""
    keys, tiles = out_rel.download()
    g = tiles.to(torch.float64).numpy()
    if select is None:
        assert keys.shape == ref["keys"].shape, (keys.shape, ref["keys"].shape)
        assert np.array_equal(keys, ref["keys"]), "output key set differs"
    else:
        keys, g = keys[select], g[select]
        assert np.array_equal(keys, ref["keys"]), "sampled keys differ"
    return check_values(g, ref["out"], ref["abs"], in_dtype, out_rel.dtype == torch.bfloat16, scale)
