"""The non-contiguous threshold rule (Eq. threshold_pd, Sec. 2.1; dcl_decode_config
acceptance = 1) on the GPU against the oracle:
  * the acceptance pass on given bf16 logits is bit-exact (same guard band as DCV's);
  * every step of a GPU generation applies the rule exactly to that step's own
    predictions (read back with dcl_forward_debug, which runs the same kernels): the
    oracle's threshold_commit on those predictions gives the same tokens, K and p;
  * closed forms: tau = 0 fills each block in one step; tau >= 1 with min_commit = k is
    the base sampler's low-confidence remasking, ceil(Bk / k) steps per block.
"""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import accept, decode

from test_gpu_accept import _guarded

pytestmark = pytest.mark.gpu

TINY = syn.SHAPES["tiny"]
N, M = 32, 64
T = N + M


@pytest.fixture(scope="module")
def dcl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as pkg
    return pkg


@pytest.fixture(scope="module")
def ctx(dcl):
    c = dcl.Context(TINY, max_batch=3, max_seq=T)
    c.load_weights(syn.model_weights(TINY, 0, lm_head_scale=40.0, norm_gain_std=0.1))
    yield c
    c.close()


@pytest.mark.parametrize("B,P,V,tau,k,conf", [(8, 32, 4096, 0.7, 1, 0), (64, 32, 126464, 0.7, 1, 0),
                                             (16, 40, 3001, 0.5, 3, 0), (16, 32, 4096, 1.0, 2, 0),
                                             (32, 32, 126464, 0.5, 1, 1)])
def test_accept_threshold_bit_exact(dcl, B, P, V, tau, k, conf):
    ops = dcl.Context(None, 1, 1)
    d, z = _guarded(B * 17 + P + k, B, P, V, (tau,), conf)
    logits = torch.from_numpy(d["logits_bf16"].view(np.int16)).cuda().view(torch.bfloat16)
    committed = torch.from_numpy(d["committed"]).cuda()
    x = torch.from_numpy(d["x"].copy()).cuda()
    kk = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    cfg = dcl.decode_config(tau_commit=tau, gen_len=P, min_commit=k, confidence=conf, acceptance=1)
    ops.accept(logits, committed, x, cfg, kk)
    torch.cuda.synchronize()
    ocfg = decode.DecodeConfig(tau_commit=tau, gen_len=P, min_commit=k, confidence=conf, acceptance=1)
    K, x_out, _, _, _ = accept.accept(z, d["committed"], d["x"], ocfg, P // 2)
    assert (kk.cpu().numpy() == K).all()
    assert (x.cpu().numpy() == x_out).all()
    ops.close()


@pytest.mark.parametrize("tau,Bk,k,conf", [(0.7, 32, 1, 0), (0.5, 16, 1, 0), (0.9, 32, 2, 0), (0.4, 8, 1, 1),
                                           (1.0, 32, 3, 0)])
def test_every_step_applies_the_rule_exactly(dcl, ctx, tau, Bk, k, conf):
    """A whole GPU generation, step by step: before each step the step's own predictions
    (top-1 ids and the confidence the threshold sees) are read with dcl_forward_debug; the
    oracle's threshold_commit applied to them, in the block holding p, must give exactly
    the GPU's next state."""
    B = 3
    prompt = syn.prompt_ids(40 + Bk + k, B, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=tau, gen_len=M, block_len=Bk, min_commit=k, confidence=conf, acceptance=1)
    ocfg = decode.DecodeConfig(tau_commit=tau, gen_len=M, block_len=Bk, min_commit=k, confidence=conf,
                               acceptance=1)
    ctx.set_prompt(prompt, cfg)
    top1 = torch.zeros(B * M, dtype=torch.int32, device="cuda")
    c = torch.zeros(B * M, device="cuda")
    x, p = ctx.get_state()
    flags = np.zeros((B, T), bool)
    flags[:, :N] = True
    steps = 0
    while (p < T).any():
        assert steps < 2 * M
        ctx.forward_debug(top1=top1, conf=c)
        ids, cv = top1.cpu().numpy().reshape(B, M), c.cpu().numpy().reshape(B, M)
        kk = ctx.step(return_k=True)
        x1, p1 = ctx.get_state()
        for b in range(B):
            if p[b] >= T:
                assert kk[b] == 0 and (x1[b] == x[b]).all() and p1[b] == p[b]
                continue
            xe = x[b].copy()
            fid = np.zeros(T, np.int32)
            fc = np.zeros(T)
            fid[N:], fc[N:] = ids[b], cv[b]
            lo = decode.prefix_end(int(p[b]), N, Bk)
            chosen = decode.threshold_commit(xe, flags[b], fid, fc, lo, min(lo + Bk, T), ocfg)
            assert (x1[b] == xe).all(), (steps, b)
            assert kk[b] == len(chosen)
            pe = int(p[b])
            while pe < T and flags[b, pe]:
                pe += 1
            assert p1[b] == pe
        x, p = x1, p1
        steps += 1
    assert (x[:, :N] == prompt).all()


def test_tau_zero_fills_each_block(dcl, ctx):
    prompt = syn.prompt_ids(5, 1, N, TINY.mask_id)
    ctx.set_prompt(prompt, dcl.decode_config(tau_commit=0.0, gen_len=M, block_len=16, acceptance=1))
    out, st, _ = ctx.generate(max_steps=4 * M)
    assert st.done == 1 and st.steps == M // 16 and st.tokens == M


@pytest.mark.parametrize("k", [1, 2, 3])
def test_tau_one_is_low_confidence_remasking(dcl, ctx, k):
    prompt = syn.prompt_ids(6, 2, N, TINY.mask_id)
    ctx.set_prompt(prompt, dcl.decode_config(tau_commit=1.0, gen_len=M, block_len=32, min_commit=k, acceptance=1))
    out, st, _ = ctx.generate(max_steps=4 * M)
    assert st.done == 1 and st.steps == (M // 32) * -(-32 // k) and st.tokens == 2 * M


def test_threshold_config_is_validated(dcl, ctx):
    prompt = syn.prompt_ids(0, 1, N, TINY.mask_id)
    for bad in (dcl.decode_config(gen_len=M, acceptance=2), dcl.decode_config(gen_len=M, acceptance=1, block_len=0)):
        with pytest.raises(dcl.DcleapError) as e:
            ctx.set_prompt(prompt, bad)
        assert e.value.status == dcl.DCL_ERR_INVALID_ARG
