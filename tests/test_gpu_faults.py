"""Fault handling on the GPU without a fault: every device wait of the GEMM and attention
pipelines is bounded (2 s of %globaltimer), after which the kernel records a timeout and
returns.  dcl_selftest_wait_timeout runs those same bounded helpers on an mbarrier and on
a global counter that nothing signals; the call must report DCL_ERR_TIMEOUT and the
context must keep working (nothing traps, nothing hangs)."""
import time

import numpy as np
import pytest
import torch

import synthetic as syn

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ops():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as dcl
    ctx = dcl.Context(None, 1, 1)
    yield dcl, ctx
    ctx.close()


@pytest.mark.parametrize("which", [0, 1])
def test_unsignalled_wait_times_out_and_context_survives(ops, which):
    dcl, ctx = ops
    t = time.perf_counter()
    st = ctx.selftest_wait_timeout(which)
    dt = time.perf_counter() - t
    assert st == dcl.DCL_ERR_TIMEOUT, st
    assert 1.5 < dt < 60, dt  # the 2 s limit, not an early return nor a hang
    assert b"timed out" in dcl.lib().dcl_last_error(ctx.ptr)
    # the context (stream, error word, allocations) is still usable
    rng = np.random.default_rng(which)
    a = syn.round_bf16(rng.normal(0, 1, (300, 256)).astype(np.float32))
    w = syn.round_bf16(rng.normal(0, 0.0625, (512, 256)).astype(np.float32))
    out = torch.zeros(300, 512, dtype=torch.bfloat16, device="cuda")
    ctx.op_linear(torch.from_numpy(a).cuda().to(torch.bfloat16), torch.from_numpy(w).cuda().to(torch.bfloat16), out)
    torch.cuda.synchronize()
    ref = a.astype(np.float64) @ w.astype(np.float64).T
    assert np.abs(out.float().cpu().numpy() - ref).max() <= 2 ** -7 * np.abs(ref).max()


def test_selftest_rejects_unknown_kind(ops):
    dcl, ctx = ops
    assert ctx.selftest_wait_timeout(2) == dcl.DCL_ERR_INVALID_ARG
