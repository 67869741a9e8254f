"""CPU oracle for upper-case-lower-case EinSum over tensor-relations.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference leg of ``bench.py`` may import this package.  The
product (``paper_2603_08957_gb300``) never imports it, and this package never
imports the product: the two share no code.

The arithmetic lives in ``ucl_oracle.c`` (plain C, fp64, tuple at a time; paper
Sec. 5, Eq. eqn-TRA and its TR-SQL template).  This module only marshals numpy
arrays into it and compiles it with gcc on first use.

Pins (tests/test_oracle.py): the worked example of Sec. 4.1 and its second
decomposition in Sec. 4.3 (tests/golden/), numpy.einsum on tiny dense inputs,
a pure-Python brute force over all index tuples, the split invariant (every
upper/lower split of one EinSum gives the same tensor, Sec. 4.2), closed-form
join/group cardinalities (Sec. 1), and hand-checked rounding values.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ucl_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")

STATUS = {
    0: "OK",
    1: "ERR_ARG",
    2: "ERR_SPEC",
    3: "ERR_SHAPE",
    4: "ERR_DUP_KEY",
    5: "ERR_KEY_RANGE",
    6: "ERR_OOM",
    8: "ERR_UNSUPPORTED",
}
EPI = {"none": 0, "relu": 1}
OUT = {"bf16": 0, "f32": 1, "f64": 2}
AGG = {"sum": 0, "max": 1, "min": 2}
COMB = {"mul": 0, "add": 1, "sub": 2, "div": 3}
MAP = {"ident": 0, "relu": 1, "exp": 2, "square": 3}

_MAXOPLEN = 16


class OracleError(RuntimeError):
    def __init__(self, code: int):
        self.code = code
        self.name = STATUS.get(code, f"status {code}")
        super().__init__(self.name)


class _Rel(ctypes.Structure):
    _fields_ = [
        ("n", ctypes.c_int64),
        ("u", ctypes.c_int),
        ("keys", ctypes.POINTER(ctypes.c_int32)),
        ("bounds", ctypes.POINTER(ctypes.c_int64)),
        ("r", ctypes.c_int),
        ("shape", ctypes.POINTER(ctypes.c_int64)),
        ("vals", ctypes.POINTER(ctypes.c_double)),
    ]


class _Opts(ctypes.Structure):
    _fields_ = [
        ("epi", ctypes.c_int),
        ("scale", ctypes.c_double),
        ("out_dtype", ctypes.c_int),
        ("sample_keys", ctypes.POINTER(ctypes.c_int32)),
        ("n_sample", ctypes.c_int64),
        ("agg", ctypes.c_int),
        ("comb", ctypes.c_int),
        ("map", ctypes.c_int),
    ]


class _Result(ctypes.Structure):
    _fields_ = [
        ("m", ctypes.c_int64),
        ("uw", ctypes.c_int),
        ("rw", ctypes.c_int),
        ("bounds", ctypes.c_int64 * _MAXOPLEN),
        ("shape", ctypes.c_int64 * _MAXOPLEN),
        ("tile", ctypes.c_int64),
        ("keys", ctypes.POINTER(ctypes.c_int32)),
        ("acc", ctypes.POINTER(ctypes.c_double)),
        ("absacc", ctypes.POINTER(ctypes.c_double)),
        ("out", ctypes.POINTER(ctypes.c_double)),
        ("n_pairs", ctypes.c_int64),
        ("n_mults", ctypes.c_int64),
    ]


_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ucl_oracle.c into a shared library (gcc, -O2); returns its path."""
    os.makedirs(_BUILD, exist_ok=True)
    stale = not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _SO + f".{os.getpid()}.tmp"
        subprocess.run(
            ["gcc", "-O2", "-std=c11", "-Wall", "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"],
            check=True,
        )
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.uo_einsum.restype = ctypes.c_int
            lib.uo_einsum.argtypes = [
                ctypes.c_char_p,
                ctypes.c_int,
                ctypes.POINTER(_Rel),
                ctypes.POINTER(_Opts),
                ctypes.POINTER(_Result),
            ]
            lib.uo_free.restype = None
            lib.uo_free.argtypes = [ctypes.POINTER(_Result)]
            lib.uo_round_bf16.restype = ctypes.c_double
            lib.uo_round_bf16.argtypes = [ctypes.c_double]
            _lib = lib
    return _lib


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def einsum(spec, rels, *, epi="none", scale=1.0, out_dtype="f64", sample_keys=None, agg="sum", comb="mul",
           map="ident"):
    """Evaluate one UCL EinSum.

    ``rels`` is a list of ``(keys, bounds, tiles)``: keys int32 [n, u], bounds
    int [u], tiles float [n, *shape] (converted exactly to float64 here).
    ``sample_keys`` (int32 [s, uw]) restricts evaluation to those output keys.
    ``agg`` / ``comb`` / ``map`` select the extended EinSum of Sec. 3: the
    aggregate (sum, max, min) over the joined values of comb (mul, add, sub,
    div) followed by map (ident, relu, exp, square).

    Returns a dict: keys [m, uw] int32, acc / abs / out [m, *shape] float64,
    bounds, shape, n_pairs, n_mults.
    """
    lib = _load()
    arrs = []
    crels = (_Rel * len(rels))()
    for i, (keys, bounds, tiles) in enumerate(rels):
        tiles = np.ascontiguousarray(np.asarray(tiles, dtype=np.float64))
        n = tiles.shape[0]
        bounds = np.ascontiguousarray(np.asarray(bounds, dtype=np.int64).reshape(-1))
        keys = np.ascontiguousarray(np.asarray(keys, dtype=np.int32).reshape(n, bounds.shape[0]))
        shape = np.ascontiguousarray(np.asarray(tiles.shape[1:], dtype=np.int64))
        if keys.shape[1] != bounds.shape[0] and n > 0:
            raise ValueError("keys and bounds disagree on the number of key columns")
        if n == 0:
            keys = np.zeros((0, bounds.shape[0]), dtype=np.int32)
        arrs += [tiles, keys, bounds, shape]
        crels[i].n = n
        crels[i].u = int(bounds.shape[0])
        crels[i].keys = _ptr(keys, ctypes.c_int32)
        crels[i].bounds = _ptr(bounds, ctypes.c_int64)
        crels[i].r = int(shape.shape[0])
        crels[i].shape = _ptr(shape, ctypes.c_int64)
        crels[i].vals = _ptr(tiles, ctypes.c_double)
    opts = _Opts()
    opts.epi = EPI[epi]
    opts.scale = float(scale)
    opts.out_dtype = OUT[out_dtype]
    opts.agg = AGG[agg]
    opts.comb = COMB[comb]
    opts.map = MAP[map]
    if sample_keys is not None:
        sk = np.ascontiguousarray(np.asarray(sample_keys, dtype=np.int32))
        arrs.append(sk)
        opts.sample_keys = _ptr(sk, ctypes.c_int32)
        opts.n_sample = sk.shape[0]
    else:
        opts.sample_keys = None
        opts.n_sample = -1
    res = _Result()
    st = lib.uo_einsum(spec.encode(), len(rels), crels, ctypes.byref(opts), ctypes.byref(res))
    if st != 0:
        raise OracleError(st)
    try:
        m, uw, rw = res.m, res.uw, res.rw
        shape = tuple(int(res.shape[q]) for q in range(rw))
        tile = int(res.tile)

        def grab(p, count, dtype):
            if count == 0:
                return np.zeros(0, dtype=dtype)
            return np.ctypeslib.as_array(p, shape=(count,)).astype(dtype, copy=True)

        out = {
            "keys": grab(res.keys, m * uw, np.int32).reshape(m, uw),
            "acc": grab(res.acc, m * tile, np.float64).reshape((m,) + shape),
            "abs": grab(res.absacc, m * tile, np.float64).reshape((m,) + shape),
            "out": grab(res.out, m * tile, np.float64).reshape((m,) + shape),
            "bounds": tuple(int(res.bounds[q]) for q in range(uw)),
            "shape": shape,
            "n_pairs": int(res.n_pairs),
            "n_mults": int(res.n_mults),
        }
    finally:
        lib.uo_free(ctypes.byref(res))
    return out


def round_bf16(x: float) -> float:
    """Round-to-nearest-even of a double to bfloat16, as the oracle's cast does."""
    return float(_load().uo_round_bf16(float(x)))


def to_dense(spec_operand: str, bounds, shape, keys, tiles):
    """Recompose the dense tensor of a tensor-relation (the point lookup of
    Sec. 4.2 with LEFT OUTER JOIN ZERO: a missing tuple reads as zeros).

    ``spec_operand`` is the operand's letter string; the dense tensor's axes
    follow its letters in order.  Used by the oracle's own pins only.
    """
    ups = [c for c in spec_operand if c.isupper()]
    lows = [c for c in spec_operand if c.islower()]
    ext = {}
    for c, b in zip(ups, bounds):
        ext[c] = int(b)
    for c, e in zip(lows, shape):
        ext[c] = int(e)
    dense = np.zeros([ext[c] for c in spec_operand], dtype=np.float64)
    tiles = np.asarray(tiles, dtype=np.float64)
    keys = np.asarray(keys).reshape(tiles.shape[0], len(ups))
    for t in range(tiles.shape[0]):
        idx = []
        for c in spec_operand:
            if c.isupper():
                idx.append(int(keys[t, ups.index(c)]))
            else:
                idx.append(slice(None))
        # axes of the tile follow the lower letters in operand order, which is
        # the order the remaining slice axes appear in the dense index
        dense[tuple(idx)] = tiles[t]
    return dense
