"""Benchmark: UCL EinSum workloads on one GPU (or N replicas under torchrun).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ucl|reference]
                    [--workload gnn|blocksparse|mttkrp|spgemm|gnn2]

Default workload (``gnn``, seed 0): GNN message passing (X x Y)^T x Z.  X
128 x 100000 bf16 N(0,1) as 1563 per-vertex-block tiles [f=128 x j=64]; Y an
R-MAT graph on 100000 vertices (a,b,c = .57,.19,.19, 1.6M drawn edges, 1.49M
after dedupe) stored as its 358136 nonempty 64 x 64 0/1 bf16 tiles keyed
(J, K); Z 128 x 128 bf16 N(0, 0.1^2), one key-less tuple.  One step =
ucl_einsum("fJj,JjKk->Kkf", X, Y) -> T (bf16) followed by
ucl_einsum("Kkf,fg->Kkg", T, Z) -> out (fp32): join, group-by and tile
contraction all on the GPU.

The other workloads (one step = the EinSum chain listed):
  blocksparse  IiJj,JjKk->IiKk: A 1024^2 fp32 at 10% of 32x32 tiles, B dense 1024x256
  mttkrp       IJKijk,Jjr,Kkr->Iir: T 100000^3, 1e7 Zipf(1.1) nonzeros in 16^3 bf16
               tiles; B, C 100000 x 64 bf16
  spgemm       IiJj,JjKk->IiKk: A, B 65536^2 at 0.5% of 128x128 bf16 tiles (half banded)
  gnn2         two-layer GNN: R-MAT 2M vertices / 40M edges as 64x64 tiles, 256-wide
               bf16 embeddings and weights, T1=(XY)^T, H1=relu(T1 W1), T2=(H1 Y)^T, O=T2 W2
  attention    graph-transformer sparse attention, CiteSeer-shaped, with row softmax as
               extended EinSums (max, exp of a difference, sum, quotient)

Metric: effective TFLOP/s over nonzero tiles = sum over the step's EinSums of
2 * (joined tuples) * prod(lower extents), divided by the device time of the
step (CUDA events; the host sizing syncs inside each EinSum are included).
Inputs are device resident.  Workloads whose inputs exceed L2 (gnn, mttkrp,
gnn2) run back to back; the others flush L2 (a 256 MB write) before every
timed step, outside its events.

Under torchrun (N > 1) every rank runs its own replica of the workload
(weak scaling, no data-path collective); value = all ranks' FLOPs / the
slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "effective TFLOP/s over nonzero tiles per EinSum"
UNIT = "TFLOP/s"
STAGES = ["keys_join", "pairs_segments", "contract", "fixup"]


# ---------------------------------------------------------------- workloads


class Workload:
    """inputs: name -> (keys, bounds, tiles on the device); chain: list of
    (output name, spec, input names, einsum options); sample(target, seed) ->
    (spec, host relations, sample keys, joined tuples) for the oracle's timing
    of the first EinSum on a subset of its output keys."""

    name = ""
    desc = ""
    dtype = "bf16"
    metric, unit, scale = None, None, 1e12   # None: the EinSum metric (TFLOP/s)
    big = True          # inputs larger than L2 (no flush needed)
    hostable = True     # inputs small enough to stage through pinned host memory every step
    flops_per_tuple = 0.0

    def __init__(self, dev, args):
        self.dev = dev
        self.args = args
        self.inputs = {}
        self.chain = []

    def sample(self, target, seed):
        raise NotImplementedError

    def release(self):
        """Drop the device tensors of the inputs (description and chain stay)."""
        self.inputs = {}
        self.w = None


def _pick_keys(counts, target, seed):
    """Random output keys (indices into counts) whose tuple counts total
    about `target`."""
    nz = np.nonzero(counts)[0]
    order = np.random.default_rng(seed).permutation(nz)
    take, tot = [], 0
    for k in order:
        take.append(int(k))
        tot += int(counts[k])
        if tot >= target:
            break
    return np.array(sorted(take), dtype=np.int64), tot


def _host64(t):
    return t.detach().to("cpu", torch.float64).numpy()


class GnnChain(Workload):
    name = "gnn"

    def __init__(self, dev, args):
        super().__init__(dev, args)
        import workloads
        n = args.vertices
        self.w = w = workloads.gnn_chain(seed=0, n=n, device=dev)
        self.inputs = {k: (w[k][0], w[k][1], w[k][2].to(dev)) for k in ("X", "Y", "Z")}
        self.chain = [("T", w["spec1"], ["X", "Y"], {"out_dtype": "bf16"}),
                      ("O", w["spec2"], ["T", "Z"], {"out_dtype": "f32"})]
        self.flops_per_tuple = 2.0 * 128 * 64 * 64
        if n == 100_000:
            self.desc = ("gnn-message-passing (XxY)^T x Z: X 128x100000 bf16, Y R-MAT 100000 vertices / 1.6M edges "
                         "as 358136 nonempty 64x64 bf16 tiles, Z 128x128 bf16; specs fJj,JjKk->Kkf then Kkf,fg->Kkg")
        else:
            self.desc = (f"gnn-message-passing (XxY)^T x Z, reduced: X 128x{n} bf16, Y R-MAT {n} vertices / "
                         f"{16 * n} edges as 64x64 bf16 tiles, Z 128x128 bf16")
        self.l2 = f"inputs larger than L2 (Y {self.inputs['Y'][2].numel() * 2 / 1e9:.1f} GB); no flush"

    def sample(self, target, seed):
        import workloads
        w = self.w
        ky = w["Y"][0]
        sk, tot = _pick_keys(np.bincount(ky[:, 1]), target, seed)
        yk = ky[np.isin(ky[:, 1], sk)]
        if not hasattr(self, "_edges"):
            self._edges = [e.cpu().numpy() if torch.is_tensor(e) else e for e in w["edges"]]
        yt = workloads.adjacency_tiles_subset(self._edges[0], self._edges[1], w["n"], w["t"], yk)
        jn = np.unique(yk[:, 0])
        xt = w["X"][2]
        xr = (jn[:, None].astype(np.int32), w["X"][1], _host64(xt[torch.as_tensor(jn, device=xt.device)]))
        return w["spec1"], [xr, (yk, w["Y"][1], yt)], sk[:, None].astype(np.int32), tot


class Gnn2(GnnChain):
    name = "gnn2"
    hostable = False

    def __init__(self, dev, args):
        Workload.__init__(self, dev, args)
        import workloads
        self.w = w = workloads.gnn_two_layer(seed=0, n=args.g2_vertices, n_edges=args.g2_edges, device=dev)
        self.inputs = {k: w[k] for k in ("X", "Y", "W1", "W2")}
        self.chain = [("T1", w["spec1"], ["X", "Y"], {"out_dtype": "bf16"}),
                      ("H1", w["spec2"], ["T1", "W1"], {"out_dtype": "bf16", "epi": "relu"}),
                      ("T2", w["spec3"], ["H1", "Y"], {"out_dtype": "bf16"}),
                      ("O", w["spec4"], ["T2", "W2"], {"out_dtype": "f32"})]
        self.flops_per_tuple = 2.0 * 256 * 64 * 64
        ny = len(w["Y"][0])
        nv, ne = args.g2_vertices, args.g2_edges
        self.desc = (f"two-layer GNN at scale: R-MAT {nv / 1e6:g}M vertices / {ne / 1e6:g}M drawn edges as {ny} "
                     f"nonempty 64x64 bf16 tiles, X 256x{nv / 1e6:g}M bf16, W1, W2 256x256 bf16; T1=(XY)^T, "
                     f"H1=relu(T1 W1), T2=(H1 Y)^T, O=T2 W2")
        self.l2 = f"inputs larger than L2 (Y {ny * 8192 / 1e9:.0f} GB); no flush"


class Mttkrp(Workload):
    name = "mttkrp"
    hostable = False

    def __init__(self, dev, args):
        super().__init__(dev, args)
        import workloads
        self.w = w = workloads.mttkrp(seed=0, nnz=args.nnz, device=dev, layout=args.t_layout)
        self.inputs = {k: w[k] for k in ("T", "B", "C")}
        self.chain = [("M", w["spec"], ["T", "B", "C"], {"out_dtype": "f32"})]
        self.flops_per_tuple = 2.0 * 16 * 16 * 16 * 64
        nt = len(w["T"][0])
        self.desc = (f"MTTKRP M[i,r]=sum T[i,j,k] B[j,r] C[k,r]: T 100000^3 with {args.nnz:.0e} Zipf(1.1) nonzeros in {nt} "
                     f"nonempty 16^3 bf16 tiles, B, C 100000x64 bf16; spec {w['spec']}")
        self.l2 = f"inputs larger than L2 (T {nt * 8192 / 1e9:.1f} GB); no flush"

    def sample(self, target, seed):
        w = self.w
        kt = w["T"][0]
        sk, tot = _pick_keys(np.bincount(kt[:, 0]), target, seed)
        m = np.nonzero(np.isin(kt[:, 0], sk))[0]
        dev = w["T"][2].device
        tr = (kt[m], w["T"][1], _host64(w["T"][2][torch.as_tensor(m, device=dev)]))

        def rows(f, r):
            r = np.unique(r)
            return (r[:, None].astype(np.int32), f[1], _host64(f[2][torch.as_tensor(r, device=dev)]))

        return w["spec"], [tr, rows(w["B"], kt[m, 1]), rows(w["C"], kt[m, 2])], sk[:, None].astype(np.int32), tot


class _Binary(Workload):
    """Block-sparse matmul-shaped workloads (IiJj,JjKk->IiKk), inputs fit L2."""
    big = False

    def _setup(self, w, tile):
        self.w = w
        self.inputs = {k: (w[k][0], w[k][1], w[k][2].to(self.dev)) for k in ("A", "B")}
        self.chain = [("C", w["spec"], ["A", "B"], {"out_dtype": "f32"})]
        self.flops_per_tuple = 2.0 * tile ** 3
        # tuples per output key (I, K): join of A and B on J
        ka, kb = w["A"][0], w["B"][0]
        g = int(max(w["A"][1][0], w["B"][1][1]))
        byj = {}
        for j, k in kb:
            byj.setdefault(int(j), []).append(int(k))
        cnt = {}
        for i, j in ka:
            for k in byj.get(int(j), ()):
                cnt[int(i) * g + k] = cnt.get(int(i) * g + k, 0) + 1
        self._codes = np.array(sorted(cnt), dtype=np.int64)
        self._counts = np.array([cnt[c] for c in self._codes], dtype=np.int64)
        self._g = g
        self._host = None

    def sample(self, target, seed):
        pick, tot = _pick_keys(self._counts, target, seed)
        codes = self._codes[pick]
        sk = np.stack([codes // self._g, codes % self._g], 1).astype(np.int32)
        if self._host is None:
            self._host = [(self.w[k][0], self.w[k][1], _host64(self.w[k][2])) for k in ("A", "B")]
        return self.w["spec"], self._host, sk, tot


class Blocksparse(_Binary):
    name = "blocksparse"
    dtype = "f32"

    def __init__(self, dev, args):
        super().__init__(dev, args)
        import workloads
        self._setup(workloads.blocksparse_matmul(seed=0), 32)
        self.desc = ("block-sparse matmul C[I,K]=sum A[I,J] B[J,K]: A 1024x1024 fp32 at 10% of 32x32 tiles "
                     "(102 tiles), B dense 1024x256 fp32; spec IiJj,JjKk->IiKk")
        self.l2 = "inputs smaller than L2: 256 MB L2 flush before every timed step (outside the events)"


class Spgemm(_Binary):
    name = "spgemm"

    def __init__(self, dev, args):
        super().__init__(dev, args)
        import workloads
        self._setup(workloads.spgemm(seed=0), 128)
        n = len(self.w["A"][0])
        self.desc = (f"block-sparse x block-sparse SpGEMM: A, B 65536x65536 at 0.5% of 128x128 bf16 tiles ({n} "
                     f"tiles each, half on a 4-tile band); spec IiJj,JjKk->IiKk")
        self.l2 = "inputs smaller than L2: 256 MB L2 flush before every timed step (outside the events)"


class Repart(Workload):
    """Repartition (Sec. 6's representation change): the message-passing Y
    (358136 64x64 bf16 tiles keyed (J, K)) split into 64-wide row vectors
    keyed (J, K, j), then stacked back into tiles."""
    name = "repart"
    metric = "effective GB/s of tiles and keys moved per repartition"
    unit = "GB/s"
    scale = 1e9

    def __init__(self, dev, args):
        super().__init__(dev, args)
        import workloads
        self.w = w = workloads.gnn_chain(seed=0, n=args.vertices, device=dev)
        self.inputs = {"Y": (w["Y"][0], w["Y"][1], w["Y"][2].to(dev))}
        self.chain = [("V", "JKjk->JKj|k", ["Y"], {"op": "repartition"}),
                      ("B", "JKLk->JK|Lk", ["V"], {"op": "repartition"})]
        ny = len(w["Y"][0])
        self.desc = (f"repartition of the message-passing Y ({ny} nonempty 64x64 bf16 tiles keyed (J, K)) into "
                     f"{64 * ny} row vectors keyed (J, K, j) and back; specs JKjk->JKj|k then JKLk->JK|Lk")
        self.l2 = f"inputs larger than L2 (Y {ny * 8192 / 1e9:.1f} GB); no flush"

    def oracle_time(self, target, seed):
        """The oracle's repartition of a random subset of Y's tuples: (bytes
        moved, seconds, tuples, tuples)."""
        from oracle.repartition import repartition
        import workloads
        w = self.w
        ky = w["Y"][0]
        rows = np.sort(np.random.default_rng(seed).choice(len(ky), size=min(len(ky), max(1, target)),
                                                          replace=False))
        if not hasattr(self, "_edges"):
            self._edges = [e.cpu().numpy() if torch.is_tensor(e) else e for e in w["edges"]]
        yt = workloads.adjacency_tiles_subset(self._edges[0], self._edges[1], w["n"], w["t"], ky[rows])
        t0 = time.perf_counter()
        repartition("JKjk->JKj|k", (ky[rows], w["Y"][1], yt))
        dt = time.perf_counter() - t0
        moved = len(rows) * (2 * 64 * 64 * 2 + 2 * 4 + 64 * 3 * 4)
        return moved, dt, len(rows), len(rows)


class Attention(Workload):
    """Sparse attention of a graph transformer (CiteSeer-shaped: 3327 nodes,
    3703 0/1 features with 32 per node, 9104 edge entries, 1024-wide bf16
    projections): the paper's UCL chain T0, T1, T2, T3, scaled scores, then
    row softmax over the neighbours as four extended EinSums."""

    name = "attention"
    big = False

    def __init__(self, dev, args):
        super().__init__(dev, args)
        import workloads
        self.w = w = workloads.graph_attention(seed=0, device=dev)
        self.inputs = {k: (w[k][0], w[k][1], w[k][2].to(dev)) for k in ("XQ", "XK", "WQ", "WK", "A")}
        self.chain = [(n, sp, ins, dict(o)) for n, sp, ins, o in w["chain"]]
        self.desc = ("graph-attention (CiteSeer-shaped): X 3327x3703 0/1 (32 nonzeros per node) as scalar tuples, "
                     "WQ/WK 3703x1024 bf16, A 9104 edge entries; IM,Mk->Ik; JN,Nk->Jk; Ik,IJ->IJk; IJk,Jk->IJ; "
                     "scale 1/32; row softmax as max / exp-sub / sum / div EinSums")
        self.l2 = "inputs smaller than L2: 256 MB flush before every timed step"
        self.flops_per_tuple = 2.0 * 1024

    def sample(self, target, seed):
        w = self.w
        xk = w["XQ"][0]
        sk, tot = _pick_keys(np.bincount(xk[:, 0]), target, seed)
        sel = np.isin(xk[:, 0], sk)
        xr = (xk[sel], w["XQ"][1], _host64(w["XQ"][2][torch.as_tensor(np.nonzero(sel)[0], device=w["XQ"][2].device)]))
        wq = (w["WQ"][0], w["WQ"][1], _host64(w["WQ"][2]))
        return "IM,Mk->Ik", [xr, wq], sk[:, None].astype(np.int32), tot


WORKLOADS = {"gnn": GnnChain, "repart": Repart, "blocksparse": Blocksparse, "mttkrp": Mttkrp, "spgemm": Spgemm,
             "gnn2": Gnn2, "attention": Attention}


# ---------------------------------------------------------------- helpers


def contract_traffic(kernel_file, workload, units):
    """DRAM bytes of one contraction, scaled by `units` (joined tuples) from an
    ncu capture summarised in profiles/<kernel>_traffic.txt; None if there is
    no capture for this workload or the kernel source changed since.  The file
    holds one block per workload, each opened by its `workload:` line."""
    import hashlib
    p = os.path.join(ROOT, "profiles", f"{kernel_file}_traffic.txt")
    src = os.path.join(ROOT, "paper_2603_08957_gb300", "csrc", f"{kernel_file}.cu")
    if not os.path.exists(p) or not os.path.exists(src):
        return None
    blocks, kv = [], None
    for line in open(p):
        line = line.split("#", 1)[0].strip()
        if ":" not in line:
            continue
        k, v = (x.strip() for x in line.split(":", 1))
        if k == "workload":
            kv = {}
            blocks.append(kv)
        if kv is not None:
            kv[k] = v
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()
    for kv in blocks:
        if kv.get("workload") == workload and kv.get("source_sha256") == sha:
            per = (int(kv["dram_read_bytes"]) + int(kv["dram_write_bytes"])) / int(kv["pairs"])
            return per * units
    return None


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"], "src": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "src": "fallback"}


class Clocks:
    """nvidia-smi sampling of SM clock and throttle reasons during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        self.device = device
        self.f = tempfile.NamedTemporaryFile(mode="w+", suffix=".csv", delete=False)
        self.p = None

    def start(self):
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--id={self.device}", f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "100"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        self.p.wait()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        sm = [float(r[1]) for r in rows if len(r) >= 9 and r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if len(r) >= 9 and r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in rows:
            if len(r) < 9:
                continue
            for i, nm in enumerate(names):
                if r[5 + i].strip() == "Active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_init(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if args.impl == "ucl" else "gloo")
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def allreduce_max(x, world, device):
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------- CPU oracle leg


def time_oracle(W, target, seed):
    """The oracle on the first EinSum restricted to random output keys holding
    about `target` joined tuples: (FLOPs, seconds, tuples, keys)."""
    if hasattr(W, "oracle_time"):
        return W.oracle_time(target, seed)
    import oracle
    spec, rels, sk, tuples = W.sample(target, seed)
    t0 = time.perf_counter()
    r = oracle.einsum(spec, rels, sample_keys=sk)
    dt = time.perf_counter() - t0
    assert r["keys"].shape[0] == len(sk)
    return W.flops_per_tuple * tuples, dt, tuples, len(sk)


def oracle_rate(W):
    _, dt, tuples, _ = time_oracle(W, 32, seed=12345)
    return tuples / max(dt, 1e-6)


def cpu_baseline(W, seconds=12.0):
    target = max(16, int(oracle_rate(W) * seconds))
    flops, dt, tuples, nk = time_oracle(W, target, seed=1)
    spec = W.chain[0][1]
    return {"value": flops / dt / W.scale, "unit": W.unit or UNIT, "cores": 1, "kind": "oracle",
            "sample": f"first EinSum {spec} restricted to {nk} random output keys ({tuples} joined tuples, "
                      f"{dt:.1f} s single-threaded fp64 C); FLOPs of those tuples / time"}


def _oracle_proc(sample, ready, start, out):
    """One host core of the all-cores baseline: load the oracle, report
    ready, wait for the common start, time the oracle on its own sample."""
    import oracle
    oracle.build()
    spec, rels, sk, _ = sample
    ready.put(os.getpid())
    start.wait()
    t0 = time.perf_counter()
    r = oracle.einsum(spec, rels, sample_keys=sk)
    out.put((time.perf_counter() - t0, int(r["keys"].shape[0])))


def cpu_baseline_all_cores(W, seconds=6.0, cores=None):
    """The oracle as it stands, one process per host core, each on its own
    bounded sample of the workload (independent output keys), all started
    together; value = all samples' FLOPs / the slowest process's time."""
    import multiprocessing as mpc
    if hasattr(W, "oracle_time"):   # a workload timed its own way (repartition)
        return None
    cores = cores or os.cpu_count() or 1
    target = max(16, int(oracle_rate(W) * seconds))
    samples = [W.sample(target, seed=2000 + i) for i in range(cores)]
    mp = mpc.get_context("spawn")   # never fork a process that holds a CUDA context
    ready, out, start = mp.Queue(), mp.Queue(), mp.Event()
    procs = [mp.Process(target=_oracle_proc, args=(smp, ready, start, out), daemon=True) for smp in samples]
    for p in procs:
        p.start()
    try:
        for _ in procs:
            ready.get(timeout=600)
        start.set()
        res = [out.get(timeout=1200) for _ in procs]
    finally:
        for p in procs:
            p.join(60)
    wall = max(t for t, _ in res)
    tuples = sum(smp[3] for smp in samples)
    assert sorted(k for _, k in res) == sorted(len(smp[2]) for smp in samples)
    spec = W.chain[0][1]
    return {"value": W.flops_per_tuple * tuples / wall / W.scale, "unit": W.unit or UNIT, "cores": cores,
            "kind": "oracle",
            "sample": f"first EinSum {spec}, {cores} processes at once, each on a random sample of output keys "
                      f"(~{target} joined tuples each, {tuples} in all, slowest {wall:.1f} s, single-threaded fp64 C "
                      f"per process); FLOPs of all samples / slowest time"}


def run_reference(args, world, rank):
    """The oracle as the reference arm: each step a bounded sample of the workload."""
    if rank != 0:
        return
    dev = "cuda" if args.workload in ("mttkrp", "gnn2") and torch.cuda.is_available() else "cpu"
    W = WORKLOADS[args.workload](dev, args)
    per_step = max(16, int(oracle_rate(W) * args.ref_step_seconds))
    for i in range(args.warmup):
        time_oracle(W, max(8, per_step // 4), seed=100 + i)
    tot_f, tot_t, tot_p = 0.0, 0.0, 0
    for i in range(args.steps):
        f, dt, p, _ = time_oracle(W, per_step, seed=1000 + i)
        tot_f += f
        tot_t += dt
        tot_p += p
    v = tot_f / tot_t / W.scale
    spec = W.chain[0][1]
    sample = (f"each step: first EinSum {spec} on random output keys totalling ~{per_step} joined tuples "
              f"({tot_p} over {args.steps} steps), single-threaded fp64 C oracle")
    unit = W.unit or UNIT
    line = {"impl": "reference", "metric": W.metric or METRIC, "value": v, "unit": unit, "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * tot_t / max(1, args.steps), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": W.desc, "l2": "n/a (CPU)"},
            "cpu_baseline": {"value": v, "unit": unit, "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- GPU leg


def stage_roofline(W, arity, stats, tim, iso, fixup, pk):
    """Per EinSum of the chain: mean stage times and the achieved fraction of
    the HBM roofline for
      sort_join -- the key stages (algorithmic bytes: read every input key
                   once, write and read back the 16-byte pair records once,
                   write the index arrays and output keys); timed both in the
                   back-to-back loop (overlapping the previous contraction)
                   and alone after a device sync ("isolated");
      contract  -- the contraction with its fused group-by sum (every input
                   tile once, the output once, the indices), with the tensor
                   fraction of its FLOPs;
      reduce    -- the fixup that adds the partials of output keys split
                   across work units (bytes counted by the fixup kernels:
                   partials read once, output tiles written once)."""
    out = []
    L = len(W.chain)
    for c, (name, spec, ins, _) in enumerate(W.chain):
        s = stats[c]
        P, S = s["n_pairs"], s["n_segments"]
        key_bytes = sum(arity[i][0] * arity[i][1] * 4 for i in ins)
        rhs = spec.split("->")[1]
        uw = len(rhs.split("|")[0]) if "|" in rhs else sum(ch.isupper() for ch in rhs)
        sort_bytes = key_bytes + 32.0 * P + 4.0 * len(ins) * P + 4.0 * uw * S
        ms = tim[c::L].mean(axis=0) if len(tim) else np.full(4, np.nan)
        mi = iso[c::L].mean(axis=0) if len(iso) else np.full(4, np.nan)
        sj, sj_iso, ct, fx = float(ms[0] + ms[1]), float(mi[0] + mi[1]), float(ms[2]), float(ms[3])
        gbs_sj = sort_bytes / (sj / 1e3) / 1e9
        gbs_sji = sort_bytes / (sj_iso / 1e3) / 1e9
        gbs_c = s["bytes_contract"] / (ct / 1e3) / 1e9
        tf_c = s["flops"] / (ct / 1e3) / 1e12
        fb = float(fixup[c])
        gbs_f = fb / (fx / 1e3) / 1e9 if fx > 0 else 0.0
        out.append({"spec": spec, "path": s["path"], "tuples": P, "segments": S, "units": s["n_units"],
                    "sort_join": {"ms": sj, "alg_bytes": sort_bytes, "GB/s": gbs_sj, "frac": gbs_sj / pk["hbm_gbs"],
                                  "isolated_ms": sj_iso, "isolated_frac": gbs_sji / pk["hbm_gbs"]},
                    "contract": {"ms": ct, "alg_bytes": s["bytes_contract"], "GB/s": gbs_c,
                                 "frac": gbs_c / pk["hbm_gbs"], "TFLOP/s": tf_c,
                                 "tensor_frac": tf_c / pk["bf16_tflops"]},
                    "reduce": {"ms": fx, "alg_bytes": fb, "GB/s": gbs_f, "frac": gbs_f / pk["hbm_gbs"]}})
    return out


def host_memory_bytes():
    """Bytes of host memory this process may still use: the smaller of
    MemAvailable and the cgroup's remaining limit."""
    avail = None
    try:
        for line in open("/proc/meminfo"):
            if line.startswith("MemAvailable:"):
                avail = int(line.split()[1]) * 1024
    except OSError:
        pass
    for path, used in (("/sys/fs/cgroup/memory.max", "/sys/fs/cgroup/memory.current"),
                       ("/sys/fs/cgroup/memory/memory.limit_in_bytes", "/sys/fs/cgroup/memory/memory.usage_in_bytes")):
        try:
            lim = open(path).read().strip()
            if lim != "max" and int(lim) < (1 << 60):
                rest = int(lim) - int(open(used).read().strip())
                avail = rest if avail is None else min(avail, rest)
            break
        except (OSError, ValueError):
            continue
    return avail


def measure(W, ctx, args, dev, world, *, steps, warmup, cpu_seconds, all_cores, e2e_on):
    """Time one workload: its chain of EinSums back to back (inputs larger
    than L2) or with an L2 flush before each step, then one isolated chain
    (latency), the end-to-end run from host buffers, and the oracle's CPU
    baseline.  Returns the measurement as a dict."""
    rels = {k: ctx.relation(torch.as_tensor(r[0]).to(dev), r[1], r[2].to(dev)) for k, r in W.inputs.items()}
    path = args.path
    flush = None if W.big else torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    arity = {k: (r.n, r.u) for k, r in rels.items()}

    def run_chain(env, collect=None, fixup=None):
        made = []
        for name, spec, ins, opts in W.chain:
            if opts.get("op") == "repartition":
                r = ctx.repartition(spec, env[ins[0]])
            else:
                r = ctx.einsum(spec, *[env[i] for i in ins], path=path, **opts)
            if collect is not None:
                collect.append(ctx.last_stats())
                arity[name] = (r.n, r.u)
            if fixup is not None:
                fixup.append(ctx.fixup_bytes(reset=True))
            env[name] = r
            made.append(r)
        return made

    def step():
        for r in run_chain(dict(rels)):
            r.destroy()

    stats, fixup = [], []
    ctx.fixup_bytes(reset=True)
    for r in run_chain(dict(rels), stats, fixup):
        r.destroy()
    for _ in range(max(0, warmup - 1)):
        step()
    torch.cuda.synchronize()
    flops_step = sum(s["flops"] for s in stats)
    if W.metric:   # a data-movement workload: its unit is bytes moved
        flops_step = sum(s["bytes_contract"] for s in stats)
    launches_step = sum(s["launches"] for s in stats)

    if steps is None:
        t0 = time.perf_counter()
        for _ in range(3):
            step()
        torch.cuda.synchronize()
        per = (time.perf_counter() - t0) / 3
        steps = int(min(2000, max(10, args.seconds / max(per, 1e-6))))

    clocks = Clocks(dev.index)
    ctx.set_timing(True)
    ctx.timings(reset=True)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    if W.big:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(steps):
            step()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
    else:
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for a, b in evs:
            flush.fill_(1)
            a.record()
            step()
            b.record()
        torch.cuda.synchronize()
        ms = sum(a.elapsed_time(b) for a, b in evs)
    barrier(world)
    ck = clocks.stop()
    L = len(W.chain)
    tim = ctx.timings(reset=True, max_calls=steps * L + L)
    tim = tim[: (len(tim) // L) * L]

    # latency: one chain alone after a device sync (the key stages then
    # overlap nothing), three times
    lat, iso = [], []
    for _ in range(3):
        if flush is not None:
            flush.fill_(1)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        made = run_chain(dict(rels))
        b.record()
        torch.cuda.synchronize()
        lat.append(a.elapsed_time(b))
        for r in made:
            r.destroy()
        t = ctx.timings(reset=True, max_calls=L)
        iso.append(t[:L])
    iso = np.concatenate(iso) if iso else np.zeros((0, 4))
    ctx.set_timing(False)
    ms_max = allreduce_max(ms, world, dev)
    value = flops_step * steps * world / (ms_max / 1e3) / W.scale

    pk = peaks()
    per_einsum = stage_roofline(W, arity, stats, tim, iso, fixup, pk)
    # dominant kernel: the contraction with the largest total time
    dom = max(range(len(per_einsum)), key=lambda c: per_einsum[c]["contract"]["ms"])
    d, s = per_einsum[dom], stats[dom]
    kfile = {"tc": "contract_tc3" if len(W.chain[dom][2]) == 3 else "contract_tc",
             "simt": "contract_simt"}.get(s["path"], "contract_simt")
    if W.chain[dom][3].get("op") == "repartition":
        kfile = "repartition"
    roof = {"bound": "hbm", "achieved": d["contract"]["GB/s"], "peak": pk["hbm_gbs"], "unit": "GB/s",
            "frac": d["contract"]["frac"], "traffic": contract_traffic(kfile, W.name, s["n_pairs"]),
            "kernel": f"{kfile} ({d['spec']})", "avg_launch_ms": d["contract"]["ms"],
            "alg_bytes_per_launch": s["bytes_contract"], "peak_src": pk["src"],
            "tensor_frac": d["contract"]["tensor_frac"]}
    stages = {name: float(tim[:, i].reshape(-1, L).sum(axis=1).mean()) if len(tim) else None
              for i, name in enumerate(STAGES)}

    # end to end through the C ABI with host buffers
    e2e = None
    in_bytes = sum(int(np.asarray(r[0]).size) * 4 + r[2].numel() * r[2].element_size() for r in W.inputs.values())
    host_avail = host_memory_bytes()
    if not e2e_on:
        e2e = {"value": None, "unit": W.unit or UNIT, "skipped": "disabled (--no-e2e)"}
    elif host_avail is not None and in_bytes > 0.4 * host_avail:
        e2e = {"value": None, "unit": W.unit or UNIT,
               "skipped": f"inputs ({in_bytes / 1e9:.1f} GB) exceed 40% of the host memory this process may use "
                          f"({host_avail / 1e9:.1f} GB): they cannot be staged in pinned host memory"}
    else:
        host = {k: (torch.as_tensor(r[0]).pin_memory(), r[1], r[2].cpu().pin_memory()) for k, r in W.inputs.items()}
        h2d = sum(t[0].numel() * 4 + t[2].numel() * t[2].element_size() for t in host.values())
        last = W.chain[-1][0]
        outbuf = {}

        def e2e_step():
            env = {k: ctx.relation(h[0], h[1], h[2]) for k, h in host.items()}
            run_chain(env)
            o = env[last]
            if not outbuf:   # pinned result buffers, sized by the untimed first call and reused
                outbuf["k"] = torch.empty(max(1, o.n * o.u), dtype=torch.int32).pin_memory()
                outbuf["t"] = torch.empty(max(1, o.n * int(np.prod(o.shape))), dtype=o.dtype).pin_memory()
            k, t = o.download(outbuf["k"], outbuf["t"])
            for r in list(env.values()):
                r.destroy()
            return k.nbytes + t.numel() * t.element_size()

        e2e_step()
        ne = max(2, min(steps, 5))
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        d2h = 0
        for _ in range(ne):
            d2h = e2e_step()
        torch.cuda.synchronize()
        te = (time.perf_counter() - t0) / ne
        te = allreduce_max(te, world, dev)
        e2e = {"value": flops_step * world / te / W.scale, "unit": W.unit or UNIT, "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(d2h), "ms_per_step": te * 1e3, "steps": ne}
        del host, outbuf

    cpu = cpu_all = None
    if cpu_seconds > 0:
        cpu = cpu_baseline(W, seconds=cpu_seconds)
        if all_cores:
            cpu_all = cpu_baseline_all_cores(W, seconds=cpu_seconds / 4)
    for r in rels.values():
        r.destroy()
    ctx.synchronize()
    W.release()
    del rels, flush
    torch.cuda.empty_cache()
    return {"W": W, "value": value, "steps": steps, "ms_per_step": ms_max / steps, "stats": stats,
            "flops_step": flops_step, "roofline": roof, "stage_ms": stages, "stage_roofline": per_einsum,
            "latency_ms": float(np.median(lat)), "e2e": e2e, "cpu_baseline": cpu, "cpu_baseline_all_cores": cpu_all,
            "gpu_launches": int(launches_step * steps), "clocks": ck, "host_memory_bytes": host_avail,
            "input_bytes": in_bytes}


PER_CONFIG = ["blocksparse", "gnn", "mttkrp", "spgemm"]


def config_of(m, world, args):
    W = m["W"]
    return {"workload": W.desc, "pairs": [s["n_pairs"] for s in m["stats"]],
            "segments": [s["n_segments"] for s in m["stats"]], "flops_per_step": m["flops_step"], "l2": W.l2,
            "path": [s["path"] for s in m["stats"]], "parallelism": f"replicas x{world}", "alloc": args.alloc}


def run_ucl(args, world, rank, local):
    from paper_2603_08957_gb300 import Context

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    ctx = Context(local, torch_allocator=(args.alloc == "torch"))
    solo = rank == 0 and world == 1
    W = WORKLOADS[args.workload](dev, args)
    m = measure(W, ctx, args, dev, world, steps=args.steps, warmup=args.warmup,
                cpu_seconds=args.cpu_seconds if solo and not args.no_cpu_baseline else 0.0,
                all_cores=True, e2e_on=not args.no_e2e)
    del W
    per_config = None
    todo = PER_CONFIG if (args.per_config == "all" and world == 1 and args.workload == "gnn2") else []
    if todo:
        per_config = {}
        for name in todo:
            torch.cuda.empty_cache()
            Wc = WORKLOADS[name](dev, args)
            mc = measure(Wc, ctx, args, dev, world, steps=None, warmup=args.warmup,
                         cpu_seconds=0.0 if args.no_cpu_baseline else args.sub_cpu_seconds, all_cores=False,
                         e2e_on=not args.no_e2e)
            per_config[name] = {"metric": Wc.metric or METRIC, "value": mc["value"], "unit": Wc.unit or UNIT,
                                "steps": mc["steps"], "ms_per_step": mc["ms_per_step"],
                                "latency_ms": mc["latency_ms"], "dtype": Wc.dtype,
                                "config": config_of(mc, world, args), "roofline": mc["roofline"],
                                "stage_roofline": mc["stage_roofline"], "cpu_baseline": mc["cpu_baseline"],
                                "e2e": mc["e2e"], "gpu_launches": mc["gpu_launches"], "clocks": mc["clocks"]}
            del Wc, mc
    if rank == 0:
        Wm = m["W"]
        line = {"metric": Wm.metric or METRIC, "value": m["value"], "unit": Wm.unit or UNIT, "n_gpus": world,
                "steps": m["steps"], "warmup": args.warmup, "ms_per_step": m["ms_per_step"],
                "latency_ms": m["latency_ms"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": Wm.dtype, "data": "synthetic", "config": config_of(m, world, args),
                "roofline": m["roofline"], "stage_ms": m["stage_ms"], "stage_roofline": m["stage_roofline"],
                "cpu_baseline": m["cpu_baseline"], "cpu_baseline_all_cores": m["cpu_baseline_all_cores"],
                "e2e": m["e2e"], "gpu_launches": m["gpu_launches"], "clocks": m["clocks"],
                "host_memory_bytes": m["host_memory_bytes"], "per_config": per_config}
        print(json.dumps(line), flush=True)
    ctx.close()


def run_rank_plans(args):
    """Rank the decompositions of the message-passing tree (X x Y)^T x Z by
    the cost model (ucl_plan, k cheapest) and time each on the GPU, as the
    paper's Opt / 2nd / 3rd tables do.  Cost constants calibrated here: C_xfer
    = 1 / measured HBM bandwidth, C_krnel = 1 / measured bf16 tensor
    throughput per flop, C_fixed = device time per joined tuple of a
    cross product of scalar tuples aggregated onto one side (the rule of thumb
    of Sec. 7.2), C_add = 0 (the group-by sum is fused into the contraction);
    the memory constraint of Sec. 8.2 bounds one kernel call's three tiles by
    256 KB, about one SM's on-chip memory (227 KB shared + 256 KB TMEM).
    Inputs are brought into each plan's split before its timing."""
    import workloads
    from paper_2603_08957_gb300 import Context, plan, program

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    ctx = Context(0)
    pk = peaks()

    def timed(fn, reps):
        fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    # C_fixed: a cross product of 4096 x 1024 scalar tuples grouped onto the 1024
    a = ctx.relation(torch.arange(4096, dtype=torch.int32, device=dev)[:, None], (4096,),
                     torch.ones(4096, device=dev))
    b = ctx.relation(torch.arange(1024, dtype=torch.int32, device=dev)[:, None], (1024,),
                     torch.ones(1024, device=dev))
    fixed = timed(lambda: ctx.einsum("I,K->K", a, b).destroy(), 5) / 1e3 / (4096 * 1024)
    cm = {"xfer": 1.0 / (pk["hbm_gbs"] * 1e9), "flop": 1.0 / (pk["bf16_tflops"] * 1e12), "add": 0.0, "fixed": fixed,
          "max_call_bytes": 256e3}

    n, t = args.vertices, 64
    w = workloads.gnn_chain(seed=0, n=n, device=dev)
    nt = -(-n // t)
    bounds = {"f": 128, "a": nt, "b": t, "c": nt, "d": t, "g": 128}
    verts = [{"labels": "fab"}, {"labels": "abcd"}, {"labels": "cdf", "left": 0, "right": 1, "dtype_bytes": 2},
             {"labels": "fg"}, {"labels": "cdg", "left": 2, "right": 3, "dtype_bytes": 4}]
    stored = {0: (ctx.relation(torch.as_tensor(w["X"][0]).to(dev), w["X"][1], w["X"][2]), "a"),
              1: (ctx.relation(torch.as_tensor(w["Y"][0]).to(dev), w["Y"][1], w["Y"][2]), "ac"),
              3: (ctx.relation(torch.as_tensor(w["Z"][0]).to(dev), w["Z"][1], w["Z"][2]), "")}
    for i, (rel, up) in stored.items():
        T, V = ctx.stats(rel)
        lab = verts[i]["labels"]
        order = [c for c in lab if c in up] + [c for c in lab if c not in up]
        verts[i].update(T=T, V=dict(zip(order, V)))
    # the k cheapest plans, and the workload's own decomposition (fJj,JjKk->Kkf
    # then Kkf,fg->Kkg) wherever the model ranks it among the first 4096
    ranked = plan(verts, bounds, cm, k=4096)
    own = {2: ("c", "a", "ac"), 4: ("c", "c", "")}
    own_rank = next((r for r, (_, ups) in enumerate(ranked)
                     if all(tuple(ups[i]) == own[i] for i in own)), None)
    todo = list(range(min(args.rank_plans, len(ranked))))
    if own_rank is not None and own_rank not in todo:
        todo.append(own_rank)
    rows = []
    for r in todo:
        cost, ups = ranked[r]
        specs = []
        for i, v in enumerate(verts):
            if v.get("left") is not None:
                upW, upU, upV = ups[i]
                specs.append(program.einsum_spec(verts[v["left"]]["labels"], upU, verts[v["right"]]["labels"], upV,
                                                 v["labels"], upW))
        row = {"rank": r + 1, "predicted_ms": cost * 1e3, "specs": specs}
        try:
            ins = program.prepare_inputs(ctx, verts, ups, stored)
            row["ms"] = timed(lambda: program.execute(ctx, verts, ups, ins).destroy(), max(3, args.steps or 5))
            row["input_tuples"] = {verts[i]["labels"]: r_.n for i, r_ in ins.items()}
            for i, r_ in ins.items():
                if r_ is not stored[i][0]:
                    r_.destroy()
        except Exception as e:  # noqa: BLE001 -- a plan the executor cannot run is reported, not fatal
            row["error"] = str(e)
        rows.append(row)
        torch.cuda.synchronize()
    ok = [r for r in rows if "ms" in r]
    measured_order = [r["rank"] for r in sorted(ok, key=lambda r: r["ms"])]
    print(json.dumps({"metric": "planner ranking vs measured step time", "workload": w["spec1"] + " ; " + w["spec2"],
                      "vertices": n, "cost_model_s": cm, "peaks_src": pk["src"], "plans": rows,
                      "measured_order": measured_order, "plans_ranked": len(ranked),
                      "workload_decomposition_rank": None if own_rank is None else own_rank + 1}), flush=True)
    ctx.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ucl", "reference"], default="ucl")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="gnn2")
    ap.add_argument("--per-config", choices=["all", "none"], default="all",
                    help="with the default two-layer GNN: also measure the other four workloads into per_config")
    ap.add_argument("--path", choices=["auto", "simt", "tc"], default="auto")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--alloc", choices=["torch", "cuda"], default="torch",
                    help="device memory for workspace and outputs: PyTorch's caching allocator (through the "
                         "allocator hooks) or the library's cudaMallocAsync pool")
    ap.add_argument("--vertices", type=int, default=100_000, help="gnn graph size (reduced sizes for profiling)")
    ap.add_argument("--nnz", type=int, default=10_000_000, help="mttkrp nonzeros (reduced sizes for profiling)")
    ap.add_argument("--g2-vertices", type=int, default=2_000_000, help="gnn2 graph size (reduced sizes for profiling)")
    ap.add_argument("--g2-edges", type=int, default=40_000_000, help="gnn2 drawn edges (reduced sizes for profiling)")
    ap.add_argument("--t-layout", choices=["ijk", "kij"], default="ijk",
                    help="mttkrp: storage order of each T tile (the same EinSum either way)")
    ap.add_argument("--seconds", type=float, default=3.0, help="timed seconds when --steps is not given")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--sub-cpu-seconds", type=float, default=5.0, help="oracle seconds for each per_config entry")
    ap.add_argument("--ref-step-seconds", type=float, default=3.0)
    ap.add_argument("--rank-plans", type=int, default=0,
                    help="instead of the benchmark: rank the K cheapest decompositions of the message-passing "
                         "tree by the cost model and time each")
    args = ap.parse_args()
    if args.rank_plans:
        run_rank_plans(args)
        return
    world, rank, local = dist_init(args)
    if args.impl == "reference":
        if args.steps is None:
            args.steps = 10
        run_reference(args, world, rank)
    else:
        run_ucl(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
