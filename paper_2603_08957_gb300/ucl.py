"""Python binding of the UCL EinSum executor: argument marshalling only.

Every step of an EinSum runs inside libucl.so on the GPU; this module turns
torch tensors into pointers and sizes, calls the C ABI (include/ucl.h) and
wraps the returned handles.  PyTorch provides device memory (its caching
allocator backs the executor's workspace and outputs) and the stream.
"""
from __future__ import annotations

import ctypes

import numpy as np
import torch

from . import _lib

BF16, F32 = 0, 1
_DTYPES = {torch.bfloat16: BF16, torch.float32: F32}
_TORCH = {BF16: torch.bfloat16, F32: torch.float32}
EPI = {"none": 0, "relu": 1}
PATH = {"auto": 0, "simt": 1, "tc": 2}
AGG = {"sum": 0, "max": 1, "min": 2}
COMB = {"mul": 0, "add": 1, "sub": 2, "div": 3}
MAP = {"ident": 0, "relu": 1, "exp": 2, "square": 3}
OUT = {"bf16": BF16, "f32": F32, torch.bfloat16: BF16, torch.float32: F32}
MEM_BORROW, MEM_DEVICE_COPY, MEM_HOST_COPY = 0, 1, 2


class UclError(RuntimeError):
    def __init__(self, status: int, detail: str = ""):
        self.status = status
        self.name = _lib.STATUS_NAMES.get(status, f"status {status}")
        self.detail = detail
        super().__init__(f"{self.name}: {detail}" if detail else self.name)


class _DevArray:
    """Minimal __cuda_array_interface__ holder for a zero-copy torch view."""

    def __init__(self, ptr, shape, typestr, owner):
        self.__cuda_array_interface__ = {
            "shape": tuple(int(s) for s in shape),
            "typestr": typestr,
            "data": (int(ptr), False),
            "version": 3,
            "strides": None,
        }
        self._owner = owner


class Context:
    """An executor context bound to one device and one CUDA stream."""

    def __init__(self, device: int = 0, stream: torch.cuda.Stream | None = None, torch_allocator: bool = True):
        self.lib = _lib.load()
        self.device = int(device)
        self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        h = ctypes.c_void_p()
        if torch_allocator:
            dev, s = self.device, self.stream.cuda_stream

            def _alloc(nbytes, user):
                try:
                    return torch.cuda.caching_allocator_alloc(int(nbytes), dev, s)
                except Exception:  # noqa: BLE001 -- reported to C as NULL -> UCL_ERR_OOM
                    return None

            def _free(ptr, nbytes, user):
                torch.cuda.caching_allocator_delete(int(ptr))

            self._alloc_cb = _lib.ALLOC_FN(_alloc)
            self._free_cb = _lib.FREE_FN(_free)
        else:
            self._alloc_cb = ctypes.cast(None, _lib.ALLOC_FN)
            self._free_cb = ctypes.cast(None, _lib.FREE_FN)
        self._check(self.lib.ucl_ctx_create(self.device, ctypes.c_void_p(self.stream.cuda_stream), self._alloc_cb,
                                            self._free_cb, None, ctypes.byref(h)), ctx=None)
        self.handle = h
        self._rels = set()

    # ------------------------------------------------------------ helpers
    def _check(self, st, ctx="self"):
        if st != 0:
            detail = ""
            if ctx == "self" and getattr(self, "handle", None):
                detail = (self.lib.ucl_last_error(self.handle) or b"").decode()
            raise UclError(st, detail)

    def close(self):
        if getattr(self, "handle", None):
            for r in list(self._rels):
                r.destroy()
            self.lib.ucl_ctx_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:  # noqa: BLE001
            pass

    def synchronize(self):
        self._check(self.lib.ucl_ctx_synchronize(self.handle))

    def set_timing(self, on: bool):
        self._check(self.lib.ucl_ctx_set_timing(self.handle, 1 if on else 0))

    def timings(self, reset: bool = True, max_calls: int = 4096):
        """Per-call stage times [calls, 4] (ms) of timed einsums since the last reset."""
        buf = (ctypes.c_float * (max_calls * _lib.UCL_NSTAGES))()
        n = ctypes.c_int()
        self._check(self.lib.ucl_ctx_timings(self.handle, buf, max_calls, ctypes.byref(n), 1 if reset else 0))
        k = min(n.value, max_calls)
        return np.frombuffer(buf, dtype=np.float32, count=k * _lib.UCL_NSTAGES).reshape(k, _lib.UCL_NSTAGES).copy()

    def last_stats(self) -> dict:
        st = _lib.Stats()
        self._check(self.lib.ucl_get_last_stats(self.handle, ctypes.byref(st)))
        return {
            "n_pairs": st.n_pairs,
            "n_segments": st.n_segments,
            "flops": st.flops,
            "bytes_contract": st.bytes_contract,
            "path": {1: "simt", 2: "tc"}.get(st.path, "none"),
            "launches": st.launches,
            "n_units": st.n_units,
            "n_bands": st.n_bands,
            "n_band_segments": st.n_band_segments,
            "stage_ms": list(st.stage_ms) if st.timed else None,
        }

    def set_wait_limit(self, cycles: int = 0):
        """SM cycles a tcgen05 role waits on one barrier phase before it
        aborts (0: the default, about a second)."""
        self._check(self.lib.ucl_ctx_set_wait_limit(self.handle, int(cycles)))

    def withhold_stage(self, fill: int):
        """Failure-detection test hook: the next binary tcgen05 contraction
        skips this pipeline stage fill (-1 cancels)."""
        self._check(self.lib.ucl_ctx_withhold_stage(self.handle, int(fill)))

    def fixup_bytes(self, reset: bool = True) -> int:
        """Bytes the fixup kernels moved since the last reset (device counter)."""
        v = ctypes.c_int64()
        self._check(self.lib.ucl_ctx_fixup_bytes(self.handle, ctypes.byref(v), 1 if reset else 0))
        return v.value

    # ---------------------------------------------------------- relations
    def relation(self, keys, bounds, tiles, *, copy: bool = False) -> "Relation":
        """Tensor-relation from device tensors: keys int32 [n, u], tiles
        [n, *shape] bf16/fp32.  Borrowed (zero copy) unless copy=True."""
        keys = torch.as_tensor(keys)
        if keys.dtype != torch.int32:
            raise TypeError("keys must be int32")
        if tiles.dtype not in _DTYPES:
            raise TypeError("tiles must be bfloat16 or float32")
        n = tiles.shape[0]
        bounds = [int(b) for b in bounds]
        keys = keys.reshape(n, len(bounds))
        host = keys.device.type == "cpu"
        if host != (tiles.device.type == "cpu"):
            raise ValueError("keys and tiles must both be on the host or both on the device")
        if not host and (keys.device.index != self.device or tiles.device.index != self.device):
            raise ValueError("tensors live on another device than the context")
        keys = keys.contiguous()
        tiles = tiles.contiguous()
        mem = MEM_HOST_COPY if host else (MEM_DEVICE_COPY if copy else MEM_BORROW)
        shape = list(tiles.shape[1:])
        b_arr = (ctypes.c_int64 * max(1, len(bounds)))(*bounds)
        s_arr = (ctypes.c_int64 * max(1, len(shape)))(*shape)
        h = ctypes.c_void_p()
        self._check(self.lib.ucl_relation_create(
            self.handle, n, len(bounds), ctypes.c_void_p(keys.data_ptr() if keys.numel() else 0), b_arr,
            len(shape), s_arr, _DTYPES[tiles.dtype], ctypes.c_void_p(tiles.data_ptr() if tiles.numel() else 0),
            mem, ctypes.byref(h)))
        rel = Relation(self, h, borrowed=(keys, tiles) if mem == MEM_BORROW else None)
        return rel

    def einsum(self, spec: str, *rels: "Relation", out_dtype="f32", epi="none", scale: float = 1.0,
               path="auto", agg="sum", comb="mul", map="ident") -> "Relation":
        """Evaluate one UCL EinSum (see include/ucl.h for the grammar); agg /
        comb / map select the extended EinSum (sum|max|min, mul|add|sub|div,
        ident|relu|exp|square)."""
        opts = _lib.EinsumOpts(OUT[out_dtype], EPI[epi], float(scale), PATH[path], AGG[agg], COMB[comb], MAP[map])
        arr = (ctypes.c_void_p * len(rels))(*[r.handle for r in rels])
        h = ctypes.c_void_p()
        self._check(self.lib.ucl_einsum(self.handle, spec.encode(), len(rels), arr, ctypes.byref(opts),
                                        ctypes.byref(h)))
        return Relation(self, h)

    def repartition(self, spec: str, rel: "Relation") -> "Relation":
        """Change a relation's upper/lower split (see include/ucl.h)."""
        h = ctypes.c_void_p()
        self._check(self.lib.ucl_repartition(self.handle, spec.encode(), rel.handle, ctypes.byref(h)))
        return Relation(self, h)

    def stats(self, rel: "Relation"):
        """(T, V): non-zero elements of the tensor a relation stores, and for
        each key column then each tile dim the number of its values or indices
        that carry a non-zero (paper Sec. 7.1)."""
        nnz = ctypes.c_int64()
        d = (ctypes.c_int64 * max(1, rel.u + rel.r))()
        self._check(self.lib.ucl_relation_stats(self.handle, rel.handle, ctypes.byref(nnz), d))
        return nnz.value, [d[i] for i in range(rel.u + rel.r)]

    def drop_zero_tiles(self, rel: "Relation") -> "Relation":
        """A relation holding the tuples of ``rel`` whose tile has a non-zero."""
        h = ctypes.c_void_p()
        self._check(self.lib.ucl_drop_zero_tiles(self.handle, rel.handle, ctypes.byref(h)))
        return Relation(self, h)


class Relation:
    """Handle of a tensor-relation living on the GPU."""

    def __init__(self, ctx: Context, handle: ctypes.c_void_p, borrowed=None):
        self.ctx = ctx
        self.handle = handle
        self._borrowed = borrowed
        n, u, r, dt = ctypes.c_int64(), ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
        kb = (ctypes.c_int64 * 16)()
        ts = (ctypes.c_int64 * 16)()
        ctx._check(ctx.lib.ucl_relation_info(handle, ctypes.byref(n), ctypes.byref(u), ctypes.byref(r), kb, ts,
                                             ctypes.byref(dt)))
        self.n, self.u, self.r = n.value, u.value, r.value
        self.bounds = tuple(kb[i] for i in range(self.u))
        self.shape = tuple(ts[i] for i in range(self.r))
        self.dtype = _TORCH[dt.value]
        ctx._rels.add(self)

    def destroy(self):
        if self.handle:
            self.ctx.lib.ucl_relation_destroy(self.handle)
            self.ctx._rels.discard(self)
            self.handle = None
            self._borrowed = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:  # noqa: BLE001
            pass

    def _ptrs(self):
        k, t = ctypes.c_void_p(), ctypes.c_void_p()
        self.ctx._check(self.ctx.lib.ucl_relation_data(self.handle, ctypes.byref(k), ctypes.byref(t)))
        return k.value or 0, t.value or 0

    def device_tensors(self):
        """Zero-copy torch views (keys int32 [n, u], tiles [n, *shape]) of the
        relation's device buffers; valid while the relation lives."""
        kp, tp = self._ptrs()
        dev = torch.device("cuda", self.ctx.device)
        if self.n == 0:
            return (torch.zeros((0, self.u), dtype=torch.int32, device=dev),
                    torch.zeros((0,) + self.shape, dtype=self.dtype, device=dev))
        keys = torch.as_tensor(_DevArray(kp, (self.n, self.u), "<i4", self), device=dev) if self.u else \
            torch.zeros((self.n, 0), dtype=torch.int32, device=dev)
        ts = "<i2" if self.dtype == torch.bfloat16 else "<f4"
        tiles = torch.as_tensor(_DevArray(tp, (self.n,) + self.shape, ts, self), device=dev)
        if self.dtype == torch.bfloat16:
            tiles = tiles.view(torch.bfloat16)
        return keys, tiles

    def download(self, keys_out=None, tiles_out=None):
        """Copy to the host through the C ABI: (keys np.int32 [n, u], tiles torch CPU [n, *shape]).

        keys_out / tiles_out: optional host buffers to copy into (e.g. pinned
        torch tensors reused across calls); they must hold at least n * u
        int32 and n * prod(shape) elements of the relation's dtype, and the
        returned arrays are views of their leading elements."""
        if keys_out is None:
            keys = np.zeros((self.n, self.u), dtype=np.int32)
        else:
            kt = torch.as_tensor(keys_out)
            if kt.device.type != "cpu" or kt.dtype != torch.int32 or not kt.is_contiguous() \
                    or kt.numel() < self.n * self.u:
                raise ValueError("keys_out must be a contiguous host int32 buffer of at least n * u elements")
            keys = kt.reshape(-1)[: self.n * self.u].numpy().reshape(self.n, self.u)
        if tiles_out is None:
            tiles = torch.empty((self.n,) + self.shape, dtype=self.dtype)
        else:
            per = int(np.prod(self.shape)) if self.shape else 1
            if tiles_out.device.type != "cpu" or tiles_out.dtype != self.dtype or not tiles_out.is_contiguous() \
                    or tiles_out.numel() < self.n * per:
                raise ValueError("tiles_out must be a contiguous host buffer of the relation's dtype, "
                                 "at least n * prod(shape) elements")
            tiles = tiles_out.reshape(-1)[: self.n * per].view((self.n,) + self.shape)
        self.ctx._check(self.ctx.lib.ucl_relation_download(
            self.handle, ctypes.c_void_p(keys.ctypes.data if keys.size else 0),
            ctypes.c_void_p(tiles.data_ptr() if tiles.numel() else 0)))
        return keys, tiles


def _plan_args(vertices, bounds, cost_model):
    """ctypes arguments of ucl_plan / ucl_plan_dag (plus buffers to keep alive)."""
    n = len(vertices)
    arr = (_lib.PlanVertex * n)()
    keep = []
    for i, v in enumerate(vertices):
        lab = v["labels"].encode()
        keep.append(lab)
        leaf = "left" not in v or v["left"] is None
        arr[i].left = -1 if leaf else int(v["left"])
        arr[i].right = -1 if leaf else int(v["right"])
        arr[i].labels = lab
        arr[i].dtype_bytes = int(v.get("dtype_bytes", 2))
        if v.get("V") is not None:
            dv = (ctypes.c_double * len(v["labels"]))(*[float(v["V"][c]) for c in v["labels"]])
            keep.append(dv)
            arr[i].distinct = dv
            arr[i].nnz = float(v["T"])
        else:
            arr[i].distinct = None
            arr[i].nnz = -1.0
    names = "".join(bounds).encode()
    bnd = (ctypes.c_int64 * len(bounds))(*[int(bounds[c]) for c in bounds])
    cm = _lib.CostModel(float(cost_model.get("xfer", 0.0)), float(cost_model.get("flop", 0.0)),
                        float(cost_model.get("add", 0.0)), float(cost_model.get("fixed", 0.0)),
                        int(cost_model.get("key_bytes", 4)), float(cost_model.get("max_call_bytes", 0.0)))
    return n, arr, names, bnd, cm, keep


def _ups(labels, mask):
    return "".join(c for q, c in enumerate(labels) if mask >> q & 1)


def _per_vertex(vertices, pc):
    per = []
    for i, v in enumerate(vertices):
        if "left" not in v or v["left"] is None:
            per.append(_ups(v["labels"], pc.up[i]))
        else:
            per.append((_ups(v["labels"], pc.up[i]), _ups(vertices[v["left"]]["labels"], pc.in_up[i][0]),
                        _ups(vertices[v["right"]]["labels"], pc.in_up[i][1])))
    return per


def plan(vertices, bounds: dict, cost_model: dict, k: int = 1):
    """The k cheapest decompositions of an EinSum tree (include/ucl.h, ucl_plan).

    ``vertices``: list of dicts in topological order, the last the root, each
    with ``labels`` (str, one character per label) and either ``T`` and ``V``
    (input tensor: non-zero count and distinct count per label) or ``left``
    and ``right`` (producer indices; ``T``/``V`` optional measured statistics);
    ``dtype_bytes`` defaults to 2.  ``bounds`` maps label -> extent;
    ``cost_model`` has ``xfer``, ``flop``, ``add``, ``fixed`` (and optional
    ``key_bytes`` and ``max_call_bytes``).  Returns [(cost, ups)], cheapest first, where ups[i] is
    ``(up_W, up_U, up_V)`` for an EinSum vertex and ``up`` for an input, each a
    string of the promoted labels in the tensor's label order."""
    lib = _lib.load()
    n, arr, names, bnd, cm, keep = _plan_args(vertices, bounds, cost_model)
    out = (_lib.PlanChoice * k)()
    n_out = ctypes.c_int()
    st = lib.ucl_plan(n, arr, names, bnd, len(bounds), ctypes.byref(cm), k, out, ctypes.byref(n_out))
    if st != 0:
        raise UclError(st, "ucl_plan")
    return [(out[b].cost, _per_vertex(vertices, out[b])) for b in range(n_out.value)]


def plan_dag(vertices, bounds: dict, cost_model: dict):
    """One decomposition of an EinSum DAG whose tensors may be consumed more
    than once, by Sec. 8.2's tree-by-tree heuristic (include/ucl.h,
    ucl_plan_dag).  Arguments as for ``plan``.  Returns (cost, ups, tree_root):
    ups[i] as for ``plan`` (an input's entry is the split its first consumer
    reads) and tree_root[i] the root of the tree EinSum vertex i was optimised
    in (-1 for inputs)."""
    lib = _lib.load()
    n, arr, names, bnd, cm, keep = _plan_args(vertices, bounds, cost_model)
    out = _lib.PlanChoice()
    roots = (ctypes.c_int * n)()
    st = lib.ucl_plan_dag(n, arr, names, bnd, len(bounds), ctypes.byref(cm), ctypes.byref(out), roots)
    if st != 0:
        raise UclError(st, "ucl_plan_dag")
    return out.cost, _per_vertex(vertices, out), list(roots)
