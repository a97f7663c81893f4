"""dcl_accept_noalloc - the block acceptance for callers that cannot allocate device
memory (code inside another framework's memory pool, or on an allocation-free
real-time path, where cudaMalloc is forbidden or may stall; such callers cannot create
a dcl_ctx either).  Called through the C ABI, it must return exactly what dcl_accept
returns, on two calls in a row that share its static scratch, and must reject sizes
beyond that scratch and beyond dcl_accept's own limits.  This file is collected last."""
import ctypes

import numpy as np
import pytest
import torch

import synthetic as syn

pytestmark = pytest.mark.gpu

MAX_POSITIONS = 32768  # DCL_NOALLOC_MAX_POSITIONS


@pytest.fixture(scope="module")
def dcl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as pkg
    return pkg


def _inputs(seed, B, P, V):
    d = syn.accept_inputs(seed, B, P, V, V - 1)
    logits = torch.from_numpy(d["logits_bf16"].view(np.int16)).cuda().view(torch.bfloat16)
    committed = torch.from_numpy(d["committed"]).cuda()
    return d, logits, committed


def _both(dcl, ctx, d, logits, committed, cfg, B, P, V, stream=None):
    """dcl_accept (context) and dcl_accept_noalloc (no context) on the same inputs."""
    L = dcl.lib()
    x_ref = torch.from_numpy(d["x"].copy()).cuda()
    k_ref = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    ctx.accept(logits, committed, x_ref, cfg, k_ref)
    x = torch.from_numpy(d["x"].copy()).cuda()
    k = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    handle = None if stream is None else ctypes.c_void_p(stream.cuda_stream)
    st = L.dcl_accept_noalloc(logits.data_ptr(), B, P, V, committed.data_ptr(), x.data_ptr(),
                              ctypes.byref(cfg), k.data_ptr(), handle)
    torch.cuda.synchronize()
    assert st == dcl.DCL_OK, L.dcl_last_error(None)
    return k, k_ref, x, x_ref


@pytest.mark.parametrize("confidence", [0, 1])
def test_noalloc_matches_dcl_accept_on_two_calls(dcl, confidence):
    """Two calls in a row (the second reuses the scratch the first left behind), with the
    top-1 probability and with the marginal-entropy confidence."""
    ctx = dcl.Context(None, 1, 1)
    for seed, B, P, V, win, contig in [(11, 16, 32, 4096, 16, 0), (12, 8, 40, 3001, 7, 1)]:
        d, logits, committed = _inputs(seed, B, P, V)
        cfg = dcl.decode_config(tau_commit=0.7, tau_draft=0.9, max_window=win, gen_len=P,
                                contiguous_drafts=contig, confidence=confidence)
        k, k_ref, x, x_ref = _both(dcl, ctx, d, logits, committed, cfg, B, P, V)
        assert torch.equal(k, k_ref)
        assert torch.equal(x, x_ref)
        assert (k.cpu().numpy() >= 1).sum() == (d["committed"] < P).sum()
    ctx.close()


@pytest.mark.parametrize("P", [32, 128])
def test_noalloc_at_the_scratch_limit_on_a_side_stream(dcl, P):
    """B*P exactly DCL_NOALLOC_MAX_POSITIONS (the three scratch arrays reach the end of
    the static array), issued on a non-default stream, twice: with B = 1024 the
    statistics pass takes its positions in place, with B = 256 compacted."""
    ctx = dcl.Context(None, 1, 1)
    B, V = MAX_POSITIONS // P, 64
    d, logits, committed = _inputs(21, B, P, V)
    cfg = dcl.decode_config(tau_commit=0.5, tau_draft=0.9, max_window=8, gen_len=P)
    side = torch.cuda.Stream()
    for _ in range(2):
        k, k_ref, x, x_ref = _both(dcl, ctx, d, logits, committed, cfg, B, P, V, stream=side)
        assert torch.equal(k, k_ref)
        assert torch.equal(x, x_ref)
    ctx.close()


def test_noalloc_rejects_sizes_beyond_its_scratch(dcl):
    L = dcl.lib()
    cfg = dcl.decode_config(gen_len=32)
    t = torch.zeros(8, dtype=torch.int32, device="cuda")
    too_many = MAX_POSITIONS // 32 + 1
    st = L.dcl_accept_noalloc(t.data_ptr(), too_many, 32, 100, t.data_ptr(), t.data_ptr(),
                              ctypes.byref(cfg), t.data_ptr(), None)
    assert st == dcl.DCL_ERR_INVALID_ARG
    assert b"32768" in L.dcl_last_error(None)
    # dcl_accept's own limit on the block length holds here too, even when B*P fits
    st = L.dcl_accept_noalloc(t.data_ptr(), 1, 8192, 100, t.data_ptr(), t.data_ptr(),
                              ctypes.byref(cfg), t.data_ptr(), None)
    assert st == dcl.DCL_ERR_INVALID_ARG
    assert b"4096" in L.dcl_last_error(None)
