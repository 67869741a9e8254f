"""Parity helpers: compare an output relation of the GPU executor with the
oracle's result for the same inputs.

The bar (per output entry, Sigma|a*b| = the oracle's magnitude sum):
  keys: bit-exact, same order;
  values: |gpu - oracle| <= tol * |scale| * Sigma|a*b|, tol = 1e-2 for bf16
  inputs (fp32 accumulate) and 1e-5 for fp32 inputs, plus the output cast
  (2^-8 |value| when the output is bf16); entries with Sigma|a*b| = 0 are
  exactly 0.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle

TOL = {torch.bfloat16: 1e-2, torch.float32: 1e-5}


def gpu_rel(ctx, rel, copy=False):
    keys, bounds, tiles = rel
    dev = torch.device("cuda", ctx.device)
    return ctx.relation(torch.as_tensor(keys).to(dev), bounds, tiles.to(dev), copy=copy)


def oracle_ref(spec, rels, *, epi="none", scale=1.0, sample_keys=None, **ext):
    """Oracle result with the epilogue applied in fp64 (no output cast);
    ``ext`` passes the extended EinSum's agg / comb / map."""
    ins = [(k, b, t.detach().to("cpu", torch.float64).numpy() if torch.is_tensor(t) else t) for k, b, t in rels]
    return oracle.einsum(spec, ins, epi=epi, scale=scale, out_dtype="f64", sample_keys=sample_keys, **ext)


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
    want, mag = ref["out"], ref["abs"]
    assert g.shape == want.shape, (g.shape, want.shape)
    bound = TOL[in_dtype] * abs(scale) * mag
    if out_rel.dtype == torch.bfloat16:
        bound = bound + 2.0**-8 * np.abs(want)
    err = np.abs(g - want)
    zero = mag == 0
    assert np.all(g[zero] == 0), "entries with no contribution must be exactly zero"
    bad = err > bound
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{bad.sum()} entries out of tolerance; first at {tuple(i)}: gpu={g[tuple(i)]!r} "
                             f"oracle={want[tuple(i)]!r} sum|ab|={mag[tuple(i)]!r}")
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(mag > 0, err / (abs(scale) * mag), 0.0)
    return float(r.max()) if r.size else 0.0
