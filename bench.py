"""Benchmark: GNN message passing (X x Y)^T x Z as two chained UCL EinSums.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ucl|reference]

Workload (seed 0): X 128 x 100000 bf16 N(0,1) as 1563 per-vertex-block tiles
[f=128 x j=64]; Y an R-MAT graph on 100000 vertices (a,b,c = .57,.19,.19,
1.6M drawn edges, 1.49M after dedupe) stored as its 358136 nonempty 64 x 64
0/1 bf16 tiles keyed (J, K); Z 128 x 128 bf16 N(0, 0.1^2), one key-less tuple.
One step = ucl_einsum("fJj,JjKk->Kkf", X, Y) -> T (bf16) followed by
ucl_einsum("Kkf,fg->Kkg", T, Z) -> out (fp32): join, group-by and tile
contraction all on the GPU.

Metric: effective TFLOP/s over nonzero tiles = sum over the two EinSums of
2 * (joined pairs) * prod(lower extents), divided by the wall time of the
step (CUDA events, host sizing syncs included).  Inputs are device resident
and larger than L2 (Y alone is 2.9 GB), so no L2 flush is needed.

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
WORKLOAD = ("gnn-message-passing (XxY)^T x Z: X 128x100000 bf16, Y R-MAT 100000 vertices / 1.6M edges "
            "as 358136 nonempty 64x64 bf16 tiles, Z 128x128 bf16; specs fJj,JjKk->Kkf then Kkf,fg->Kkg")


def workload_name(vertices):
    if vertices == 100_000:
        return WORKLOAD
    return (f"gnn-message-passing (XxY)^T x Z, reduced: X 128x{vertices} bf16, Y R-MAT {vertices} vertices / "
            f"{16 * vertices} edges as 64x64 bf16 tiles, Z 128x128 bf16")


def contract_traffic(pairs):
    """DRAM bytes of one contraction launch, scaled by pairs from the ncu capture in
    profiles/contract_tc_traffic.txt; None once the kernel source changed since."""
    import hashlib
    p = os.path.join(ROOT, "profiles", "contract_tc_traffic.txt")
    src = os.path.join(ROOT, "paper_2603_08957_gb300", "csrc", "contract_tc.cu")
    if not os.path.exists(p):
        return None
    kv = {}
    for line in open(p):
        line = line.split("#", 1)[0].strip()
        if ":" in line:
            k, v = line.split(":", 1)
            kv[k.strip()] = v.strip()
    if hashlib.sha256(open(src, "rb").read()).hexdigest() != kv.get("source_sha256"):
        return None
    per_pair = (int(kv["dram_read_bytes"]) + int(kv["dram_write_bytes"])) / int(kv["pairs"])
    return per_pair * pairs


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


def oracle_sample(w, target_pairs, seed=0):
    """Output keys K whose pairs total about target_pairs, with the oracle's
    inputs for them (X whole, only the Y tiles of those K)."""
    import workloads
    ky = w["Y"][0]
    cnt = np.bincount(ky[:, 1])
    ks = np.nonzero(cnt)[0]
    rng = np.random.default_rng(seed)
    order = rng.permutation(ks)
    take, tot = [], 0
    for k in order:
        take.append(k)
        tot += cnt[k]
        if tot >= target_pairs:
            break
    sk = np.array(sorted(take), dtype=np.int32)[:, None]
    ysel = np.isin(ky[:, 1], sk[:, 0])
    yk = ky[ysel]
    yt = workloads.adjacency_tiles_subset(w["edges"][0], w["edges"][1], w["n"], w["t"], yk)
    xk, xb, xt = w["X"]
    return sk, (xk, xb, xt.to("cpu", torch.float64).numpy()), (yk, w["Y"][1], yt), int(tot)


def time_oracle(w, target_pairs, seed):
    import oracle
    sk, xr, yr, pairs = oracle_sample(w, target_pairs, seed)
    t0 = time.perf_counter()
    r = oracle.einsum("fJj,JjKk->Kkf", [xr, yr], sample_keys=sk)
    dt = time.perf_counter() - t0
    assert r["n_pairs"] >= pairs
    flops = 2.0 * pairs * 128 * 64 * 64
    return flops, dt, pairs, len(sk)


def calibrate_oracle(w):
    flops, dt, pairs, _ = time_oracle(w, 64, seed=12345)
    return pairs / dt  # pairs per second


def cpu_baseline(w, seconds=12.0):
    rate = calibrate_oracle(w)
    target = max(64, int(rate * seconds))
    flops, dt, pairs, nk = time_oracle(w, target, seed=1)
    return {"value": flops / dt / 1e12, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"first EinSum fJj,JjKk->Kkf restricted to {nk} random output keys K ({pairs} joined pairs, "
                      f"{dt:.1f} s single-threaded fp64 C); FLOPs of those pairs / time"}


def run_reference(args, world, rank):
    """The oracle as the reference arm: each step a bounded sample of the workload."""
    if rank != 0:
        return
    import workloads
    w = workloads.gnn_chain(seed=0, device="cpu")
    rate = calibrate_oracle(w)
    per_step = max(16, int(rate * args.ref_step_seconds))
    for i in range(args.warmup):
        time_oracle(w, max(16, per_step // 4), seed=100 + i)
    tot_f, tot_t, tot_p = 0.0, 0.0, 0
    for i in range(args.steps):
        f, dt, p, _ = time_oracle(w, per_step, seed=1000 + i)
        tot_f += f
        tot_t += dt
        tot_p += p
    v = tot_f / tot_t / 1e12
    sample = (f"each step: first EinSum fJj,JjKk->Kkf on random output keys K totalling ~{per_step} joined pairs "
              f"({tot_p} pairs over {args.steps} steps), single-threaded fp64 C oracle")
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * tot_t / max(1, args.steps), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "l2": "n/a (CPU)"},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- GPU leg


def run_ucl(args, world, rank, local):
    import workloads
    from paper_2603_08957_gb300 import Context

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = workloads.gnn_chain(seed=0, n=args.vertices, device=dev)
    ctx = Context(local, torch_allocator=(args.alloc == "torch"))

    def rel(r):
        return ctx.relation(torch.as_tensor(r[0]).to(dev), r[1], r[2].to(dev))

    X, Y, Z = rel(w["X"]), rel(w["Y"]), rel(w["Z"])
    path = args.path

    def step():
        T = ctx.einsum(w["spec1"], X, Y, out_dtype="bf16", path=path)
        O = ctx.einsum(w["spec2"], T, Z, out_dtype="f32", path=path)
        T.destroy()
        return O

    # warm-up and per-step counters (deterministic)
    T = ctx.einsum(w["spec1"], X, Y, out_dtype="bf16", path=path)
    s1 = ctx.last_stats()
    O = ctx.einsum(w["spec2"], T, Z, out_dtype="f32", path=path)
    s2 = ctx.last_stats()
    T.destroy()
    O.destroy()
    for _ in range(max(0, args.warmup - 1)):
        step().destroy()
    torch.cuda.synchronize()
    flops_step = s1["flops"] + s2["flops"]
    launches_step = s1["launches"] + s2["launches"]

    steps = args.steps
    if steps is None:
        t0 = time.perf_counter()
        for _ in range(3):
            step().destroy()
        torch.cuda.synchronize()
        per = (time.perf_counter() - t0) / 3
        steps = int(min(2000, max(10, 3.0 / max(per, 1e-6))))

    clocks = Clocks(local)
    ctx.set_timing(True)
    ctx.timings(reset=True)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        step().destroy()
    e1.record()
    torch.cuda.synchronize()
    barrier(world)
    ck = clocks.stop()
    ms = e0.elapsed_time(e1)
    tim = ctx.timings(reset=True)
    ctx.set_timing(False)
    ms_max = allreduce_max(ms, world, dev)
    value = flops_step * steps * world / (ms_max / 1e3) / 1e12

    # dominant kernel: the contraction of the first EinSum (stage 2 of every other call)
    contract_ms = tim[0::2, 2]
    avg_contract = float(contract_ms.mean()) if len(contract_ms) else float("nan")
    pk = peaks()
    achieved = s1["bytes_contract"] / (avg_contract / 1e3) / 1e9
    roof = {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
            "frac": achieved / pk["hbm_gbs"], "traffic": contract_traffic(s1["n_pairs"]),
            "kernel": f"contract_{s1['path']} (fJj,JjKk->Kkf)", "avg_launch_ms": avg_contract,
            "alg_bytes_per_launch": s1["bytes_contract"], "peak_src": pk["src"],
            "tensor_frac": (s1["flops"] / (avg_contract / 1e3) / 1e12) / pk["bf16_tflops"]}
    stages = {name: float(tim[0::2, i].mean()) for i, name in enumerate(["keys_join", "pairs_segments",
                                                                           "contract", "fixup"])}

    # end to end through the C ABI with host buffers
    e2e = None
    if not args.no_e2e:
        hx = [torch.as_tensor(w["X"][0]).pin_memory(), w["X"][2].cpu().pin_memory()]
        hy = [torch.as_tensor(w["Y"][0]).pin_memory(), w["Y"][2].cpu().pin_memory()]
        hz = [torch.as_tensor(w["Z"][0]).pin_memory(), w["Z"][2].cpu().pin_memory()]
        h2d = sum(t.numel() * t.element_size() for t in hx + hy + hz)

        def e2e_step():
            Xh = ctx.relation(hx[0], w["X"][1], hx[1])
            Yh = ctx.relation(hy[0], w["Y"][1], hy[1])
            Zh = ctx.relation(hz[0], w["Z"][1], hz[1])
            T = ctx.einsum(w["spec1"], Xh, Yh, out_dtype="bf16", path=path)
            O = ctx.einsum(w["spec2"], T, Zh, out_dtype="f32", path=path)
            k, t = O.download()
            for r in (Xh, Yh, Zh, T, O):
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
        e2e = {"value": flops_step * world / te / 1e12, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(d2h), "ms_per_step": te * 1e3}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, seconds=args.cpu_seconds)

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": steps,
                "warmup": args.warmup, "ms_per_step": ms_max / steps, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": workload_name(args.vertices), "pairs": [s1["n_pairs"], s2["n_pairs"]],
                           "segments": [s1["n_segments"], s2["n_segments"]], "flops_per_step": flops_step,
                           "l2": "inputs larger than L2 (Y 2.9 GB); no flush", "path": s1["path"],
                           "parallelism": f"replicas x{world}", "alloc": args.alloc},
                "roofline": roof, "stage_ms": stages, "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": int(launches_step * steps), "clocks": ck}
        print(json.dumps(line), flush=True)
    for r in (X, Y, Z):
        r.destroy()
    ctx.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ucl", "reference"], default="ucl")
    ap.add_argument("--path", choices=["auto", "simt", "tc"], default="auto")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--alloc", choices=["torch", "cuda"], default="torch",
                    help="device memory for workspace and outputs: PyTorch's caching allocator (through the "
                         "allocator hooks) or the library's cudaMallocAsync pool")
    ap.add_argument("--vertices", type=int, default=100_000, help="graph size (reduced sizes for profiling)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--ref-step-seconds", type=float, default=3.0)
    args = ap.parse_args()
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
