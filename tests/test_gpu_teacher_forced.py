"""Teacher-forced parity of the whole denoise step, block by block, at the 2-layer test
size and at the sizes the benchmark runs: the LLaDA-8B shape (batch 1, prompt 256 + gen
256, window 128) and the Dream-7B shape (GQA 28 / 4, prompt 384 + gen 512, window 256;
the 16 rows of the batch hold the same state), thresholds 0.7 / 0.98.

Inputs flow oracle -> GPU only.  Each state (a committed prefix, the MASKed window and
drafts beyond it, from the seeded generator of synthetic/) is run through the oracle's
forward (bf16 operands, fp64 accumulation), whose residual stream entering block l
(rounded to fp32, the GPU's stream format) is loaded into the GPU with
dcl_forward_debug_from; the GPU's stream after block l is then compared with the
oracle's block l on the same input, for every block:
  * blocks: relative rms error per row <= 3.5e-3 mean, 6e-3 max (the bound the block-0
    test of tests/test_gpu_fullsize.py derives; an IEEE-fp32 evaluation with the same
    rounding points stays inside it, tests/test_fp32_restatement.py);
  * LM head and confidence (Eq. 2) on identical inputs: the oracle's final-normed rows,
    rounded to bf16, through the GPU's fused LM head + softmax (dcl_op_lmhead_top2, the
    full vocabulary, the same weights generated on the host) give the top-1 and top-2
    probabilities within 1e-3 and the top-1 id wherever the top-1/top-2 gap exceeds 1e-3;
  * the same from the oracle's final stream through the step's own final RMSNorm and LM
    head (dcl_forward_debug_from at layer n_layers): logits within max relative error
    2e-2 per row, and the top-1 probability within TOL_PATH = 5e-3.  The final RMSNorm is
    rounded to bf16 from fp32 on the GPU and from fp64 in the oracle, so an element within
    fp32 rounding (~2^-22 relative) of a bf16 midpoint rounds one bf16 ulp apart (about
    5e-5 of the elements, 0.2 per row at d = 3584); such an element moves a logit by at
    most |w| ulp(x), ~ 3 sigma_w 2^-8 |x| ~ 9e-3 at the LM-head scale (sigma_w = 0.02 x
    12.8), and the top-1 probability by at most a quarter of that, ~2.3e-3: TOL_PATH
    allows two such elements on the top logit (measured: 1.3e-3 over 1024 Dream rows);
  * decisions (Eq. compute_k, Eq. draft_update): the GPU's acceptance on those
    predictions (commit = 1) equals the oracle's commit_and_draft on its own predictions,
    exactly, unless a decision's margin is within TOL_PATH (a near tie: counted, and the
    outcome must then be one of the valid ones).
The oracle's accumulated forward (no teacher forcing) is also compared with the GPU's
whole forward from the tokens, for the record (printed).
"""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import decode, model

pytestmark = pytest.mark.gpu

STD = 0.02
TAU_C, TAU_D = 0.70, 0.98
TOL_P = 1e-3                 # top-1 / top-2 probability on identical LM-head inputs (absolute)
TOL_PATH = 5e-3              # the same through the step's final RMSNorm (its bf16 rounding, above)
TOL_BLOCK = (3.5e-3, 6e-3)   # relative rms per row: mean, max
# name: shape, batch, prompt, generation, window, weight seed, LM-head scale, norm-gain std,
#       offsets p - N of the states checked
CONFIGS = {
    "tiny": ("tiny", 2, 32, 64, 32, 0, 40.0, 0.1, (0, 24)),
    "llada8b": ("llada8b", 1, 256, 256, 128, 1, 12.0, 0.0, (0, 120)),
    "dream7b": ("dream7b", 16, 384, 512, 256, 2, 12.8, 0.0, (0, 200)),
}


@pytest.fixture(scope="module")
def dcl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as pkg
    return pkg


def _rel_rms(got, ref):
    return np.sqrt(((got - ref) ** 2).mean(axis=1)) / np.sqrt((ref ** 2).mean(axis=1))


def _oracle_decision(x0, p0, ids, c1, c2, N, L, ocfg):
    """The oracle's step on one row with a guard band: (x1, K, near) where near counts the
    decisions whose margin is within TOL_PATH (K and the affected positions are then None /
    left to the validity check)."""
    T = x0.shape[0]
    full_id = np.zeros(T, np.int32)
    full_c = np.zeros(T)
    gap = np.full(T, np.inf)
    full_id[N:], full_c[N:], gap[N:] = ids, c1, c1 - c2
    x1 = x0.copy()
    K = decode.commit_and_draft(x1, p0, full_id, full_c, ocfg, L)
    w = min(L, T - p0)
    k_lo = min(max(decode.window_length(full_c[p0:p0 + w], TAU_C + TOL_PATH), 1), w)
    k_hi = min(max(decode.window_length(full_c[p0:p0 + w], TAU_C - TOL_PATH), 1), w)
    unsure = np.zeros(T, bool)
    unsure[p0 + k_lo:p0 + k_hi] = True                            # committed or not
    unsure[p0:p0 + k_hi] |= gap[p0:p0 + k_hi] <= TOL_PATH         # committed id may differ
    fut = np.arange(T) >= p0 + L
    unsure |= fut & (np.abs(full_c - TAU_D) <= TOL_PATH)          # draft decision may differ
    unsure |= fut & (full_c > TAU_D) & (gap <= TOL_PATH)          # drafted id may differ
    near = int(k_lo != k_hi) + int(unsure.sum())
    return x1, (K if k_lo == k_hi else None), (k_lo, k_hi), unsure, full_id, near


@pytest.mark.parametrize("name", list(CONFIGS))
def test_teacher_forced_blocks_head_and_decisions(dcl, name):
    shape, B, N, M, L, seed, lm_scale, gstd, offsets = CONFIGS[name]
    sh = syn.SHAPES[shape]
    T = N + M
    d = sh.d_model
    ocfg = decode.DecodeConfig(tau_commit=TAU_C, tau_draft=TAU_D, max_window=L, gen_len=M)
    prompt1 = syn.prompt_ids(2000, 1, N, sh.mask_id)
    states = [syn.decode_state(77, prompt1, M, off, L, sh.mask_id) for off in offsets]
    stream = torch.cuda.Stream()
    ctx = dcl.Context(sh, max_batch=B, max_seq=T, stream=stream.cuda_stream)
    try:
        if name == "tiny":
            w_all = syn.model_weights(sh, seed, STD, lm_scale, gstd)
            ctx.load_weights(w_all)
        else:
            w_all = None
            ctx.init_random_weights(seed, STD, lm_scale, gstd)
        ctx.set_prompt(np.repeat(prompt1, B, axis=0),
                       dcl.decode_config(tau_commit=TAU_C, tau_draft=TAU_D, max_window=L, block_len=32, gen_len=M))
        h_dev = torch.zeros(B * T, d, device="cuda")
        got = torch.zeros(B * T, d, device="cuda")
        torch.cuda.synchronize()

        def load_state(s):
            x, p = states[s]
            ctx.set_state(np.repeat(x, B, axis=0), np.repeat(p, B))

        def run_from(layer, h_in, commit=False, **outs):
            h_dev.copy_(torch.from_numpy(np.tile(h_in.astype(np.float32), (B, 1))))
            torch.cuda.synchronize()
            with torch.cuda.stream(stream):
                ctx.forward_debug_from(layer, h_dev, commit, **outs)

        # embedding: the oracle's rows of the tokens present
        h = []
        for x, _ in states:
            if w_all is not None:
                h.append(np.asarray(w_all["embed"], np.float64)[x[0]])
            else:
                uniq, inv = np.unique(x[0], return_inverse=True)
                h.append(syn.embed_rows(sh, seed, uniq, STD)[inv].astype(np.float64))
        angles = model.rope_angles(T, sh.head_dim, sh.rope_theta)
        worst = [0.0, 0.0]
        # block 1 from the GPU's own block-0 output (its attn_norm is the RMSNorm that the
        # previous block's MLP launch runs at its end), and the input of the last block
        second, last_in = {}, {}
        for layer in range(sh.n_layers):
            lw = (w_all if w_all is not None else
                  syn.model_weights(sh, seed, STD, lm_scale, gstd, layers=(layer,), global_tensors=False))["layers"][layer]
            for s in range(len(states)):
                h_in = h[s].astype(np.float32)
                if layer == sh.n_layers - 1:
                    last_in[s] = h_in
                ref = model.block(sh, lw, h_in.astype(np.float64), angles, bf16_operands=True)
                load_state(s)
                run_from(layer, h_in)
                with torch.cuda.stream(stream):
                    ctx.debug_hidden(layer, got)
                g = got.cpu().numpy()
                assert (g[:T] == g.reshape(B, T, d)).all(), "rows holding the same state differ"
                err = _rel_rms(g[:T].astype(np.float64), ref)
                worst = [max(worst[0], float(err.mean())), max(worst[1], float(err.max()))]
                assert err.mean() <= TOL_BLOCK[0] and err.max() <= TOL_BLOCK[1], (layer, s, err.mean(), err.max())
                if layer == 0 and sh.n_layers > 1:
                    with torch.cuda.stream(stream):
                        ctx.debug_hidden(1, got)
                    second[s] = (g[:T].astype(np.float64), got.cpu().numpy()[:T].astype(np.float64))
                if layer == 1:
                    ref2 = model.block(sh, lw, second[s][0], angles, bf16_operands=True)
                    err2 = _rel_rms(second[s][1], ref2)
                    assert err2.mean() <= TOL_BLOCK[0] and err2.max() <= TOL_BLOCK[1], (s, err2.mean(), err2.max())
                h[s] = ref
        print(f"{name}: every block teacher-forced, relative rms per row: worst mean {worst[0]:.2e}, "
              f"worst max {worst[1]:.2e}")

        # final RMSNorm + LM head + confidence, from the oracle's final stream
        gw = syn.model_weights(sh, seed, STD, lm_scale, gstd, layers=(), embed=False) if w_all is None else w_all
        w_lm = torch.from_numpy(np.asarray(gw["lm_head"], np.float32)).to(torch.bfloat16).cuda()
        ops = dcl.Context(None, 1, 1)
        near_total = exact_total = 0
        for s, (x, p) in enumerate(states):
            h_in = h[s].astype(np.float32)
            hn = model.rms_norm(h_in.astype(np.float64)[N:], gw["final_norm"], sh.rms_eps)
            z = model.logits(gw, hn)                                       # pure definition
            hb = model.to_bf16(hn)
            ids_o, p1_o, p2_o = model.confidence(model.logits(gw, hb))    # bf16 operand
            sure = p1_o - p2_o > TOL_P
            # the fused LM head + softmax on identical inputs
            top1 = torch.zeros(B * M, dtype=torch.int32, device="cuda")
            q1 = torch.zeros(B * M, device="cuda")
            q2 = torch.zeros(B * M, device="cuda")
            ops.op_lmhead_top2(torch.from_numpy(hb.astype(np.float32)).to(torch.bfloat16).cuda(), w_lm,
                               top1[:M], q1[:M], q2[:M])
            g1, g2, gi = q1.cpu().numpy()[:M], q2.cpu().numpy()[:M], top1.cpu().numpy()[:M]
            assert np.abs(g1 - p1_o).max() <= TOL_P, float(np.abs(g1 - p1_o).max())
            assert np.abs(g2 - p2_o).max() <= TOL_P, float(np.abs(g2 - p2_o).max())
            assert (gi[sure] == ids_o[sure]).all()
            e_same = float(np.abs(g1 - p1_o).max())
            # the step's final RMSNorm + LM head from the oracle's final stream
            logits = torch.zeros(B * M, sh.vocab, dtype=torch.bfloat16, device="cuda")
            torch.cuda.synchronize()
            load_state(s)
            run_from(sh.n_layers, h_in, logits=logits, top1=top1, p1=q1, p2=q2)
            g1, gi = q1.cpu().numpy()[:M], top1.cpu().numpy()[:M]
            assert np.abs(g1 - p1_o).max() <= TOL_PATH, float(np.abs(g1 - p1_o).max())
            clear = p1_o - p2_o > TOL_PATH
            assert (gi[clear] == ids_o[clear]).all()
            zg = logits[:M].float().cpu().numpy()
            assert (np.abs(zg - z).max(axis=1) / np.abs(z).max(axis=1)).max() <= 2e-2
            print(f"{name} state {s}: max |p1 - p1_oracle| = {e_same:.2e} on identical LM-head inputs "
                  f"({int(sure.sum())}/{M} ids exact), {np.abs(g1 - p1_o).max():.2e} through the final RMSNorm")

            # the acceptance on those predictions against the oracle's
            x1_o, K_o, (k_lo, k_hi), unsure, full_id, near = _oracle_decision(x[0], int(p[0]), ids_o, p1_o, p2_o,
                                                                               N, L, ocfg)
            load_state(s)
            run_from(sh.n_layers, h_in, commit=True, top1=top1)
            x1, p1 = ctx.get_state()
            gtop = np.full(T, -1, np.int64)
            for b in range(B):
                k = int(p1[b]) - int(p[0])
                assert k_lo <= k <= k_hi, (k_lo, k, k_hi)
                if K_o is not None:
                    assert k == K_o
                same = x1[b] == x1_o
                assert same[~unsure].all(), np.nonzero(~same & ~unsure)[0][:8]
                # unsure positions: the old token, or the oracle's or the GPU's top-1 id
                gtop[N:] = top1.cpu().numpy()[b * M:(b + 1) * M]
                assert ((x1[b] == x[0]) | (x1[b] == full_id) | (x1[b] == gtop) | same)[unsure].all()
            near_total += near
            exact_total += int((~unsure).sum()) + int(K_o is not None)
        print(f"{name}: decisions exact {exact_total}, near ties (margin <= {TOL_PATH}) {near_total}")

        # the final RMSNorm as the last MLP launch runs it, on the GPU's own last block
        # output: p1 against the oracle's final norm + LM head of that output
        for s in range(len(states)):
            load_state(s)
            run_from(sh.n_layers - 1, last_in[s], top1=top1, p1=q1, p2=q2)
            with torch.cuda.stream(stream):
                ctx.debug_hidden(sh.n_layers - 1, got)
            g = got.cpu().numpy()[:T].astype(np.float64)
            hn = model.rms_norm(g[N:], gw["final_norm"], sh.rms_eps)
            ids_o, p1_o, p2_o = model.confidence(model.logits(gw, model.to_bf16(hn)))
            g1, gi = q1.cpu().numpy()[:M], top1.cpu().numpy()[:M]
            assert np.abs(g1 - p1_o).max() <= TOL_PATH, float(np.abs(g1 - p1_o).max())
            clear = p1_o - p2_o > TOL_PATH
            assert (gi[clear] == ids_o[clear]).all()
        ops.close()

        # for the record: the accumulated forward from the tokens (no teacher forcing)
        x, p = states[0]
        load_state(0)
        with torch.cuda.stream(stream):
            ctx.forward_debug()
            ctx.debug_hidden(sh.n_layers - 1, got)
        acc = _rel_rms(got.cpu().numpy()[:T].astype(np.float64), h[0])
        print(f"{name}: accumulated forward, last block relative rms per row: mean {acc.mean():.2e}, "
              f"max {acc.max():.2e}")
    finally:
        ctx.close()
