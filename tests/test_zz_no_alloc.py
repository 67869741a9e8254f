"""ucl_keys_check_noalloc: key validation for callers that cannot allocate
device memory (a device-memory budget owned by another component, or code
that must never call cudaMalloc because it can synchronise the device).

It must agree with the checks ucl_relation_create performs with allocated
workspace: the same status (OK / KEY_RANGE / DUP_KEY) and the same verdict
on ascending order, on two calls in a row (the scratch array it shares
between calls keeps the previous call's contents).  This file is collected
last so that a failure here stops a -x run only after every other test ran.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2603_08957_gb300 import Context, UclError, _lib

pytestmark = pytest.mark.gpu


def _cases():
    rng = np.random.default_rng(21)
    out = []
    # sorted, unique, 2 columns
    k = np.stack(np.meshgrid(np.arange(300), np.arange(7), indexing="ij"), -1).reshape(-1, 2).astype(np.int32)
    out.append(("sorted", k, (300, 7)))
    # the same tuples shuffled
    out.append(("unsorted", k[rng.permutation(len(k))], (300, 7)))
    # a duplicate far apart after shuffling
    d = k[rng.permutation(len(k))].copy()
    d[-1] = d[5]
    out.append(("duplicate", d, (300, 7)))
    # a key out of range
    r = k.copy()
    r[100, 1] = 7
    out.append(("range", r, (300, 7)))
    # a large random unique set near the size limit, three columns (54 bits)
    big = np.unique(rng.integers(0, 2**18, size=(900_000, 3)), axis=0)
    out.append(("large", big[rng.permutation(len(big))].astype(np.int32), (2**18,) * 3))
    # sorted except for one adjacent duplicate: flagged unsorted, then sorted and caught
    a = k.copy()
    a[41] = a[40]
    out.append(("adjacent duplicate", a, (300, 7)))
    # exactly the size limit, shuffled (the scan runs over the full histogram)
    m = 1 << 20
    full = np.stack([np.arange(m) // 1024, np.arange(m) % 1024], 1).astype(np.int32)
    out.append(("at the limit", full[rng.permutation(m)], (1024, 1024)))
    # every bound 1: zero key bits, so two tuples are the same key
    out.append(("zero bits", np.zeros((2, 3), np.int32), (1, 1, 1)))
    return out


def _noalloc(lib, keys_dev, n, u, bounds):
    b = (ctypes.c_int64 * max(1, u))(*bounds)
    srt = ctypes.c_int(-1)
    st = lib.ucl_keys_check_noalloc(0, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream), n, u,
                                    ctypes.c_void_p(keys_dev.data_ptr()), b, ctypes.byref(srt))
    return st, srt.value


def _ascending(keys):
    """Strictly ascending lexicographic order of the key rows (host check)."""
    if len(keys) < 2:
        return True
    a, b = keys[:-1].astype(np.int64), keys[1:].astype(np.int64)
    less = np.zeros(len(a), dtype=bool)
    undecided = np.ones(len(a), dtype=bool)
    for c in range(keys.shape[1]):
        less |= undecided & (a[:, c] < b[:, c])
        undecided &= a[:, c] == b[:, c]
    return bool(less.all())


def test_matches_relation_create_twice():
    ctx = Context(0)
    lib = _lib.load()
    cases = []
    for name, keys, bounds in _cases():
        n, u = keys.shape
        kd = torch.from_numpy(keys).cuda()
        tiles = torch.zeros((n, 1), dtype=torch.float32, device="cuda")
        try:
            ctx.relation(kd, bounds, tiles).destroy()   # the allocating entry point
            want = 0
        except UclError as e:
            want = e.status
        cases.append((name, keys, kd, bounds, want))
    expect = {"duplicate": 4, "adjacent duplicate": 4, "zero bits": 4, "range": 5}   # DUP_KEY, KEY_RANGE
    for name, _, _, _, want in cases:
        assert want == expect.get(name, 0), (name, want)
    ctx.close()

    def run_all():
        for name, keys, kd, bounds, want in cases:
            n, u = keys.shape
            for _ in range(2):
                st, srt = _noalloc(lib, kd, n, u, bounds)
                assert st == want, (name, st, want)
                if want == 0:
                    assert bool(srt) == _ascending(keys), name

    run_all()   # the first calls look up the scratch address and load the kernels
    torch.cuda.synchronize()
    torch_before = torch.cuda.memory_stats().get("allocation.all.allocated", 0)
    free_before, _ = torch.cuda.mem_get_info()
    dev = torch.cuda.current_device()
    run_all()
    torch.cuda.synchronize()
    assert torch.cuda.current_device() == dev
    assert torch.cuda.memory_stats().get("allocation.all.allocated", 0) == torch_before
    free_after, _ = torch.cuda.mem_get_info()
    assert free_after == free_before, (free_before, free_after)


def test_rejects_oversize_without_gpu_work():
    lib = _lib.load()
    b = (ctypes.c_int64 * 1)(10)
    srt = ctypes.c_int(-1)
    st = lib.ucl_keys_check_noalloc(0, None, (1 << 20) + 1, 1, ctypes.c_void_p(16), b, ctypes.byref(srt))
    assert st == 8  # UCL_ERR_UNSUPPORTED
