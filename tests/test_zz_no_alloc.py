"""dcl_accept_noalloc - the block acceptance for callers that cannot allocate device
memory (code inside another framework's memory pool, or on an allocation-free
real-time path, where cudaMalloc is forbidden or may stall; such callers cannot create
a dcl_ctx either).  Called through the C ABI, it must return exactly what dcl_accept
returns, on two calls in a row that share its static scratch, and must reject sizes
beyond that scratch.  This file is collected last."""
import ctypes

import numpy as np
import pytest
import torch

import synthetic as syn

pytestmark = pytest.mark.gpu


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


def test_noalloc_matches_dcl_accept_on_two_calls(dcl):
    ctx = dcl.Context(None, 1, 1)
    L = dcl.lib()
    for seed, B, P, V, win, contig in [(11, 16, 32, 4096, 16, 0), (12, 8, 40, 3001, 7, 1)]:
        d, logits, committed = _inputs(seed, B, P, V)
        cfg = dcl.decode_config(tau_commit=0.7, tau_draft=0.9, max_window=win, gen_len=P,
                                contiguous_drafts=contig)
        x_ref = torch.from_numpy(d["x"].copy()).cuda()
        k_ref = torch.full((B,), -1, dtype=torch.int32, device="cuda")
        ctx.accept(logits, committed, x_ref, cfg, k_ref)
        x = torch.from_numpy(d["x"].copy()).cuda()
        k = torch.full((B,), -1, dtype=torch.int32, device="cuda")
        torch.cuda.synchronize()
        st = L.dcl_accept_noalloc(logits.data_ptr(), B, P, V, committed.data_ptr(), x.data_ptr(),
                                  ctypes.byref(cfg), k.data_ptr(), None)
        torch.cuda.synchronize()
        assert st == dcl.DCL_OK, L.dcl_last_error(None)
        assert torch.equal(k, k_ref)
        assert torch.equal(x, x_ref)
        assert (k.cpu().numpy() >= 1).sum() == (d["committed"] < P).sum()
    ctx.close()


def test_noalloc_rejects_sizes_beyond_its_scratch(dcl):
    L = dcl.lib()
    cfg = dcl.decode_config(gen_len=32)
    t = torch.zeros(8, dtype=torch.int32, device="cuda")
    too_many = 32768 // 32 + 1
    st = L.dcl_accept_noalloc(t.data_ptr(), too_many, 32, 100, t.data_ptr(), t.data_ptr(),
                              ctypes.byref(cfg), t.data_ptr(), None)
    assert st == dcl.DCL_ERR_INVALID_ARG
    assert b"32768" in L.dcl_last_error(None)
