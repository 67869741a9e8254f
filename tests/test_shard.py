"""Output-key-range sharding of EinSum chains (paper_2603_08957_gb300/shard.py)
on two gloo CPU ranks.  Each rank evaluates its EinSums with the oracle (so
these tests need no GPU); the ranks' results, concatenated in rank order, must
equal the single-process chain: the same key set, bit-identical values (every
output key is summed over the same pairs in the same order on either side)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
import workloads
from paper_2603_08957_gb300 import shard


def oracle_einsum(spec, rels, out_dtype="f32", epi="none", scale=1.0):
    ins = [(k.numpy(), tuple(b), t.to(torch.float64).numpy()) for k, b, t in rels]
    r = oracle.einsum(spec, ins, epi=epi, scale=scale, out_dtype=out_dtype)
    dt = torch.bfloat16 if out_dtype == "bf16" else torch.float32
    return torch.from_numpy(r["keys"].copy()), tuple(r["bounds"]), torch.from_numpy(r["out"]).to(dt)


def _gnn2_small():
    w = workloads.gnn_two_layer(seed=3, n=3000, n_edges=40_000, feat=32, t=16, device="cpu")
    ins = {k: (torch.as_tensor(w[k][0]), tuple(w[k][1]), w[k][2]) for k in ("X", "Y", "W1", "W2")}
    chain = [("T1", w["spec1"], ["X", "Y"], {"out_dtype": "bf16"}),
             ("H1", w["spec2"], ["T1", "W1"], {"out_dtype": "bf16", "epi": "relu"}),
             ("T2", w["spec3"], ["H1", "Y"], {"out_dtype": "bf16"}),
             ("O", w["spec4"], ["T2", "W2"], {"out_dtype": "f32"})]
    return chain, ins


def _spgemm_small():
    rng = np.random.default_rng(5)
    g, t = 24, 8

    def rel():
        codes = np.sort(rng.choice(g * g, size=90, replace=False))
        keys = np.stack([codes // g, codes % g], 1).astype(np.int32)
        return torch.from_numpy(keys), (g, g), torch.from_numpy(rng.standard_normal((90, t, t))).to(torch.bfloat16)

    return [("C", "IiJj,JjKk->IiKk", ["A", "B"], {"out_dtype": "f32"})], {"A": rel(), "B": rel()}


CASES = {"gnn2": _gnn2_small, "spgemm": _spgemm_small}


def _worker(rank, world, port, case, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        _work(rank, world, case, q)
    except Exception as e:  # noqa: BLE001 -- reported to the parent, which fails the test
        q.put((rank, repr(e), -1))
        raise
    finally:
        dist.destroy_process_group()


def _work(rank, world, case, q):
    chain, ins = CASES[case]()
    sc = shard.ShardedChain(rank, world, oracle_einsum)
    env = sc.run(chain, ins)
    out = {}
    for name, *_ in chain:
        rel, part = env[name]
        full = sc.gather_result(env[name])
        out[name] = (rel[0].shape[0], part.col, part.cuts, full[0].numpy(), full[2].to(torch.float64).numpy())
    q.put((rank, out, sc.gathered_bytes))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _run(case, world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, case, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=180) for _ in procs]
    for r, o, _ in res:
        assert not isinstance(o, str), f"rank {r}: {o}"
    for p in procs:
        p.join(60)
        assert p.exitcode == 0
    return {r: (o, b) for r, o, b in res}


@pytest.mark.parametrize("case", ["gnn2", "spgemm"])
def test_two_ranks_equal_one(case):
    chain, ins = CASES[case]()
    ref = {}
    env = {k: v for k, v in ins.items()}
    for name, spec, names, opts in chain:
        env[name] = oracle_einsum(spec, [env[n] for n in names], **opts)
        ref[name] = env[name]
    res = _run(case, 2)
    for name, *_ in chain:
        for r in (0, 1):
            n_local, col, cuts, keys, tiles = res[r][0][name]
            assert np.array_equal(keys, ref[name][0].numpy()), (name, r)
            assert np.array_equal(tiles, ref[name][2].to(torch.float64).numpy()), (name, r)
            assert col == 0 and cuts is not None
        # the two parts split the output: disjoint, every key once
        n0, n1 = res[0][0][name][0], res[1][0][name][0]
        assert n0 + n1 == ref[name][0].shape[0]
        assert n0 > 0 and n1 > 0
    if case == "gnn2":
        # the exchange: H1 all-gathered once for the second message passing,
        # plus the final gathers of the test itself
        assert res[0][1] > 0 and res[1][1] > 0


def test_balanced_cuts():
    w = np.array([5, 0, 0, 1, 1, 1, 1, 1, 0, 10], dtype=float)
    c = shard.balanced_cuts(w, 3)
    assert c[0] == 0 and c[-1] == len(w) and all(a <= b for a, b in zip(c, c[1:]))
    pre = np.concatenate([[0], np.cumsum(w)])
    # each cut is the first value at which the prefix reaches r / world of the total
    for r in (1, 2):
        assert pre[c[r]] >= w.sum() * r / 3 and (c[r] == 0 or pre[c[r] - 1] < w.sum() * r / 3)
    assert shard.balanced_cuts(np.zeros(4), 2) == (0, 0, 4)
    assert shard.balanced_cuts(np.ones(8), 4) == (0, 2, 4, 6, 8)


def test_pair_weights_brute_force():
    rng = np.random.default_rng(1)
    ku = rng.integers(0, 6, size=(40, 2)).astype(np.int32)
    ku = np.unique(ku, axis=0)
    kv = np.unique(rng.integers(0, 6, size=(50, 2)), axis=0).astype(np.int32)
    # spec IJ,JK->IK: V's tuple (J, K) joins every U tuple with that J
    w = shard.pair_weights("IJ,JK->IK", [ku, kv], [(6, 6), (6, 6)], 1)
    want = np.array([np.sum(ku[:, 1] == j) for j, _ in kv], dtype=float)
    assert np.array_equal(w, want)
    # star join IJK,J,K->I: T's tuple weighs #B(J) * #C(K)
    kt = np.unique(rng.integers(0, 5, size=(60, 3)), axis=0).astype(np.int32)
    kb = np.array([[0], [2], [3]], np.int32)
    kc = np.array([[1], [2]], np.int32)
    w = shard.pair_weights("IJK,J,K->I", [kt, kb, kc], [(5, 5, 5), (5,), (5,)], 0)
    want = np.array([(j in (0, 2, 3)) * (k in (1, 2)) for _, j, k in kt], dtype=float)
    assert np.array_equal(w, want)
    # no shared label: a cross product weighs the other side's size
    w = shard.pair_weights("I,K->IK", [np.arange(3)[:, None], np.arange(7)[:, None]], [(3,), (7,)], 0)
    assert np.array_equal(w, np.full(3, 7.0))
