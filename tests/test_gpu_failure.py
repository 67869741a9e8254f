"""Failure detection on the GPU without a fault: the tcgen05 contraction's
bounded waits.  A test hook makes the producers skip one stage fill (no copy
issued, no arrival posted); with a short wait limit the roles waiting on it
give up, the CTA drains what it has in flight, frees its tensor memory and
returns, and the context reports UCL_ERR_TIMEOUT at its next synchronising
call.  The same context then evaluates the EinSum correctly."""
import time

import pytest
import torch

import workloads
from paper_2603_08957_gb300 import Context, UclError
from tests.parity import assert_parity, gpu_rel, oracle_ref

pytestmark = pytest.mark.gpu

UCL_ERR_TIMEOUT = 9


@pytest.mark.parametrize("window", ["0", "2"])
def test_withheld_stage_times_out_and_context_recovers(monkeypatch, window):
    """Both binary tcgen05 kernels: the plain one and the windowed one."""
    monkeypatch.setenv("UCL_WINDOW", window)
    ctx = Context(0)
    monkeypatch.delenv("UCL_WINDOW")
    w = workloads.gnn_chain(seed=6, n=4096, degree=16)
    X, Y = gpu_rel(ctx, w["X"]), gpu_rel(ctx, w["Y"])
    ref = oracle_ref(w["spec1"], [w["X"], w["Y"]])

    ctx.set_wait_limit(200_000)          # about 0.1 ms of SM clock
    ctx.withhold_stage(2)
    t0 = time.perf_counter()
    T = ctx.einsum(w["spec1"], X, Y, out_dtype="bf16", path="tc")
    with pytest.raises(UclError) as e:
        ctx.synchronize()
    dt = time.perf_counter() - t0
    assert e.value.status == UCL_ERR_TIMEOUT, e.value
    # the drain waited only for copies that were really in flight (the
    # withheld fill is skipped), well inside the default limit of ~1 s
    assert dt < 1.0, dt
    T.destroy()

    ctx.set_wait_limit(0)
    ctx.synchronize()                    # nothing left over
    T = ctx.einsum(w["spec1"], X, Y, out_dtype="bf16", path="tc")
    ctx.synchronize()
    assert_parity(T, ref, torch.bfloat16)
    for r in (X, Y, T):
        r.destroy()
    ctx.close()


def test_wait_limit_arguments():
    ctx = Context(0)
    with pytest.raises(UclError):
        ctx.set_wait_limit(-1)
    with pytest.raises(UclError):
        ctx.withhold_stage(-2)
    ctx.withhold_stage(-1)
    ctx.set_wait_limit(0)
    ctx.close()
