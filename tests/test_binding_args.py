"""The Python binding's argument checks (CPU only, no library call is made).

Every ``*_dev`` argument must be a CUDA tensor of the element size the C ABI states,
holding at least the elements the call touches: a host buffer or a short one is refused
in Python, before a kernel could read or write past it.  The checks run on stand-in
tensors, and on a Context whose library is a recorder, so no GPU is needed."""
import os
import sys

import numpy as np
import pytest
import torch

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import paper_2607_20467_gb300 as dcl  # noqa: E402
import synthetic as syn  # noqa: E402


class FakeCuda:
    """Stands in for a contiguous CUDA tensor: its size, element size and address."""

    is_cuda = True

    def __init__(self, n, itemsize, shape=None):
        self.n, self.itemsize, self.dtype = n, itemsize, f"{itemsize}-byte"
        self.shape = shape if shape is not None else (n,)

    def element_size(self):
        return self.itemsize

    def numel(self):
        return self.n

    def is_contiguous(self):
        return True

    def data_ptr(self):
        return 0x7000_0000


class Recorder:
    """A library whose every function records its call and returns DCL_OK."""

    def __init__(self):
        self.calls = []

    def __getattr__(self, name):
        def fn(*args):
            self.calls.append(name)
            return 0
        return fn


def _context(shape=None, batch=1, n_prompt=32, gen_len=64):
    ctx = object.__new__(dcl.Context)
    ctx._L, ctx.ptr, ctx.shape = Recorder(), None, shape
    ctx.batch, ctx.n_prompt, ctx.gen_len = batch, n_prompt, gen_len
    return ctx


def test_device_pointer_check():
    assert dcl._dev(None, "a", 4) is None
    assert dcl._dev(0x1234, "a", 4) == 0x1234  # a raw device address passes through
    with pytest.raises(ValueError, match="device buffer"):
        dcl._dev(np.zeros(4, np.int32), "a", 4)
    with pytest.raises(ValueError, match="device buffer"):
        dcl._dev(torch.zeros(4, dtype=torch.int32), "a", 4)
    with pytest.raises(TypeError, match="4 bytes"):
        dcl._dev(FakeCuda(8, 2), "a", 4)
    with pytest.raises(ValueError, match="at least 9"):
        dcl._dev(FakeCuda(8, 4), "a", 4, 9)
    assert dcl._dev(FakeCuda(9, 4), "a", 4, 9) == 0x7000_0000


def test_weight_elements_add_up_to_the_llada8b_weights():
    """Per layer (H + 2G) hd d + d H hd + 3 F d + 2 d elements: 13.96 GB of bf16 over the
    32 layers of the LLaDA-8B shape; embedding and LM head V d each."""
    sh = syn.SHAPES["llada8b"]
    layer = sum(dcl.weight_elements(sh, k) for k in (dcl.DCL_W_ATTN_NORM, dcl.DCL_W_Q, dcl.DCL_W_K, dcl.DCL_W_V,
                                                     dcl.DCL_W_O, dcl.DCL_W_MLP_NORM, dcl.DCL_W_GATE, dcl.DCL_W_UP,
                                                     dcl.DCL_W_DOWN))
    assert 2 * layer * sh.n_layers == pytest.approx(13.96e9, rel=1e-3)
    assert dcl.weight_elements(sh, dcl.DCL_W_LM_HEAD) == dcl.weight_elements(sh, dcl.DCL_W_EMBED) == 126464 * 4096
    g = syn.SHAPES["dream7b"]  # GQA: K and V have G = 4 heads of 128
    assert dcl.weight_elements(g, dcl.DCL_W_K) == 4 * 128 * 3584


def test_context_refuses_host_and_short_buffers_before_any_call():
    sh = syn.SHAPES["tiny"]
    ctx = _context(sh, batch=2)
    n = 2 * 64
    with pytest.raises(ValueError):
        ctx.forward_debug(top1=torch.zeros(n, dtype=torch.int32))
    with pytest.raises(ValueError):
        ctx.forward_debug(p1=FakeCuda(n - 1, 4))
    with pytest.raises(ValueError):
        ctx.forward_debug(logits=FakeCuda(n * sh.vocab - 1, 2))
    with pytest.raises(ValueError):
        ctx.debug_hidden(0, FakeCuda(2 * 96 * sh.d_model - 1, 4))
    with pytest.raises(TypeError):
        ctx.forward_debug_from(1, FakeCuda(2 * 96 * sh.d_model, 2))
    B, P, V = 4, 8, 16
    logits = torch.zeros(B, P, V, dtype=torch.bfloat16)  # host memory
    with pytest.raises(ValueError):
        ctx.accept(logits, FakeCuda(B, 4), FakeCuda(B * P, 4), dcl.decode_config(), FakeCuda(B, 4))
    with pytest.raises(ValueError):
        ctx.accept(FakeCuda(B * P * V, 2, (B, P, V)), FakeCuda(B, 4), FakeCuda(B * P - 1, 4), dcl.decode_config(),
                   FakeCuda(B, 4))
    with pytest.raises(TypeError):  # mode 1 adds into a float residual stream
        ctx.op_linear(FakeCuda(4 * 64, 2, (4, 64)), FakeCuda(128 * 64, 2, (128, 64)), FakeCuda(4 * 128, 2), mode=1)
    with pytest.raises(ValueError):
        ctx.set_weight(dcl.DCL_W_Q, 0, np.zeros(sh.n_heads * sh.head_dim * sh.d_model - 1, np.uint16))
    with pytest.raises(TypeError):
        ctx.set_weight(dcl.DCL_W_ATTN_NORM, 0, torch.zeros(sh.d_model))  # float32, not bf16
    assert ctx._L.calls == []


def test_context_passes_well_formed_buffers_through():
    sh = syn.SHAPES["tiny"]
    ctx = _context(sh, batch=2)
    n = 2 * 64
    ctx.forward_debug(FakeCuda(n * sh.vocab, 2), FakeCuda(n, 4), FakeCuda(n, 4), None, None, FakeCuda(n, 4))
    ctx.debug_hidden(0, FakeCuda(2 * 96 * sh.d_model, 4))
    B, P, V = 4, 8, 16
    ctx.accept(FakeCuda(B * P * V, 2, (B, P, V)), FakeCuda(B, 4), FakeCuda(B * P, 4), dcl.decode_config(),
               FakeCuda(B, 4))
    ctx.op_linear(FakeCuda(4 * 64, 2, (4, 64)), FakeCuda(128 * 64, 2, (128, 64)), FakeCuda(4 * 128, 4), mode=1)
    ctx.set_weight(dcl.DCL_W_ATTN_NORM, 0, np.zeros(sh.d_model, np.uint16))
    assert ctx._L.calls == ["dcl_forward_debug", "dcl_debug_hidden", "dcl_accept", "dcl_op_linear",
                            "dcl_set_weight"]
