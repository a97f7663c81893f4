"""The denoise step at full size, in the launch configuration the benchmark times: the
LLaDA-8B shape (32 layers, d 4096, 32 heads of 128, FFN 12288, vocab 126464), batch 1,
prompt 256 + generation 256, window 128, thresholds 0.7 / 0.98, LM head x12, weight seed
1, the step's CUDA graph on a caller stream; and the long-generation configuration
(prompt 512 + generation 1024, window 512).

A 32-layer forward of an 8B model in fp64 is out of reach of a test, so:
  * the residual stream after the embedding (exactly) and after blocks 0 and 1 is compared
    with the bf16-operand oracle on every one of the 512 rows.  Tolerance: at this size the
    fp32 accumulation alone moves values across bf16 rounding boundaries often enough
    that an IEEE-fp32 evaluation of block 0 with the same rounding points (PyTorch on the
    CPU) lies 2.1e-3 (mean) / 4.4e-3 (max) from the fp64 oracle in relative rms per row,
    the GPU 2.7e-3 / 4.2e-3; dropping any one of the bf16 rounding points moves the
    oracle by 2.5e-3 .. 6.8e-3 (mean).  Block 0 must stay within 3.5e-3 (mean) and 6e-3
    (max), block 1 (whose input already differs) within 5e-3 and 1e-2;
  * every step of a whole generation must apply the acceptance rule (Eq. compute_k,
    Eq. draft_update, Algorithm 1; strict thresholds in float32, K raised to 1, window
    clipped to the sequence end) to the step's own predictions, which
    dcl_forward_debug reproduces bit for bit (same kernels, deterministic reductions),
    and the generation must end with every position committed;
  * a second generation of the same prompt through dcl_generate gives the same tokens.
The rule is restated here in a few lines of numpy; the oracle is not fed GPU values.
"""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import model

pytestmark = pytest.mark.gpu

SH = syn.SHAPES["llada8b"]
SEED, STD, LM_SCALE = 1, 0.02, 12.0
TAU_C, TAU_D = 0.70, 0.98
CONFIGS = {  # name: (prompt, generation, window)
    "llada8b": (256, 256, 128),
    "llada8b-long": (512, 1024, 512),
}


@pytest.fixture(scope="module")
def dcl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as pkg
    return pkg


def _context(dcl, name):
    N, M, L = CONFIGS[name]
    stream = torch.cuda.Stream()
    ctx = dcl.Context(SH, max_batch=1, max_seq=N + M, stream=stream.cuda_stream)
    ctx.init_random_weights(SEED, STD, LM_SCALE, 0.0)
    prompt = syn.prompt_ids(1000, 1, N, SH.mask_id)
    cfg = dcl.decode_config(tau_commit=TAU_C, tau_draft=TAU_D, max_window=L, block_len=32, gen_len=M)
    ctx.set_prompt(prompt, cfg)
    return ctx, stream, prompt


def test_first_blocks_match_oracle(dcl):
    N, M, L = CONFIGS["llada8b"]
    T = N + M
    ctx, stream, prompt = _context(dcl, "llada8b")
    try:
        x = np.full(T, SH.mask_id, np.int32)
        x[:N] = prompt[0]
        with torch.cuda.stream(stream):
            ctx.forward_debug()
            h = torch.zeros(T, SH.d_model, device="cuda")
            got = []
            for layer in (-1, 0, 1):
                ctx.debug_hidden(layer, h)
                got.append(h.cpu().numpy().astype(np.float64))
        xin, _ = ctx.get_state()
        assert (xin[0] == x).all()  # the first window lies inside the all-MASK generation
    finally:
        ctx.close()
    # the oracle's weights: layers 0 and 1 and the embedding rows of the tokens present
    uniq, inv = np.unique(x, return_inverse=True)
    w = syn.model_weights(SH, SEED, STD, LM_SCALE, 0.0, layers=(0, 1), global_tensors=False)
    w["embed"] = syn.embed_rows(SH, SEED, uniq, STD)
    assert (got[0] == w["embed"][inv]).all()  # the embedding is an exact copy
    for layer, (tol_mean, tol_max) in ((0, (3.5e-3, 6e-3)), (1, (5e-3, 1e-2))):
        ref = model.forward_hidden(SH, w, inv, bf16_operands=True, upto_layer=layer)
        err = np.sqrt(((got[layer + 1] - ref) ** 2).mean(axis=1)) / np.sqrt((ref ** 2).mean(axis=1))
        print(f"block {layer}: relative rms error per row mean {err.mean():.2e} max {err.max():.2e}")
        assert err.mean() <= tol_mean and err.max() <= tol_max, (layer, float(err.mean()), float(err.max()))


def _expected_step(x0, p0, top1, c1, N, L):
    """The acceptance rule on one row (absolute positions; top1 / c1 over [N, T))."""
    T = x0.shape[0]
    w = min(L, T - p0)
    tc, td = np.float32(TAU_C), np.float32(TAU_D)
    run = 0
    while run < w and c1[p0 - N + run] > tc:
        run += 1
    K = min(max(run, 1), w)
    x = x0.copy()
    x[p0:p0 + w] = SH.mask_id
    x[p0:p0 + K] = top1[p0 - N:p0 - N + K]
    for i in range(p0 + L, T):
        if c1[i - N] > td:
            x[i] = top1[i - N]
    return x, K


@pytest.mark.parametrize("name", list(CONFIGS))
def test_generation_follows_acceptance_rule(dcl, name):
    N, M, L = CONFIGS[name]
    T = N + M
    ctx, stream, prompt = _context(dcl, name)
    try:
        top1 = torch.zeros(M, dtype=torch.int32, device="cuda")
        c1 = torch.zeros(M, device="cuda")
        c2 = torch.zeros(M, device="cuda")
        torch.cuda.synchronize()  # the buffers exist before the context's stream writes them
        steps = 0
        ks = []
        while True:
            x0, p0 = ctx.get_state()
            p0 = int(p0[0])
            if p0 >= T:
                break
            with torch.cuda.stream(stream):
                ctx.forward_debug(None, top1, c1, c2)
            ids, conf, conf2 = top1.cpu().numpy(), c1.cpu().numpy(), c2.cpu().numpy()
            assert ((ids >= 0) & (ids < SH.vocab)).all()
            assert (conf2 <= conf).all() and (conf <= 1.0).all() and (conf2 >= 0.0).all()
            k = int(ctx.step(return_k=True)[0])
            x1, p1 = ctx.get_state()
            x_exp, K = _expected_step(x0[0], p0, ids, conf, N, L)
            assert k == K, (steps, k, K)
            assert int(p1[0]) == p0 + K
            assert (x1[0] == x_exp).all(), (steps, np.nonzero(x1[0] != x_exp)[0][:8])
            ks.append(k)
            steps += 1
            assert steps <= M
        x_final, p_final = ctx.get_state()
        assert int(p_final[0]) == T and sum(ks) == M
        assert (x_final[0, :N] == prompt[0]).all()
        assert (x_final[0, N:] != SH.mask_id).all()
        # the same generation again through the public entry point: same tokens, same count
        ctx.restart()
        out, stats, status = ctx.generate()
        assert (out[0] == x_final[0, N:]).all()
        assert stats.steps == steps
    finally:
        ctx.close()
