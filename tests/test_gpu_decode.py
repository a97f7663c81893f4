"""The whole denoise step and Algorithm 1 on the GPU (through the C ABI) against the
oracle, on the 2-layer / d 256 / 4x64 heads / vocab 4096 model (prompt 32, gen 64).

Tolerances.  Kernels fed identical inputs agree tightly (tests/test_gpu_ops.py: the
fused LM head + softmax gives top-1/top-2 probabilities within 1e-3).  End to end the
GPU keeps matrix-product operands in bf16 and accumulates in fp32; the oracle used
for decisions stores the same operands in bf16 but accumulates in fp64.  Values that
land on different sides of a bf16 rounding boundary are then amplified by this random
model: attention is nearly uniform, so its output averages ~T cancelling value
vectors and relative differences grow ~sqrt(T) per layer; with logits up to ~45
(LM head x40) a final-hidden difference of ~1e-3 moves logits by up to ~0.1 and the
top-1 probability by up to ~3e-2.  Hence:
  * logits: max |z_gpu - z| <= 2e-2 max |z| per row (pure fp64 oracle);
  * residual stream after each layer: relative rms error <= 3e-3;
  * confidences: |p1_gpu - p1| <= E2E_TOL = 5e-2;
  * decisions: every decision whose oracle margin exceeds E2E_TOL (|c - tau| for the
    commit and draft thresholds, top-1/top-2 gap for the committed id) must agree
    exactly; the others must be one of the valid outcomes.
Teacher forcing flows oracle -> GPU only: oracle states are loaded with dcl_set_state.
"""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import decode, model

pytestmark = pytest.mark.gpu

TINY = syn.SHAPES["tiny"]
N, M = 32, 64
T = N + M
E2E_TOL = 5e-2


@pytest.fixture(scope="module")
def dcl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as pkg
    return pkg


@pytest.fixture(scope="module")
def weights():
    return syn.model_weights(TINY, 0, lm_head_scale=40.0, norm_gain_std=0.1)


@pytest.fixture(scope="module")
def ctx(dcl, weights):
    c = dcl.Context(TINY, max_batch=4, max_seq=T)
    c.load_weights(weights)
    yield c
    c.close()


def _predict(w, with_entropy=False):
    return lambda tokens: model.predict(TINY, w, tokens, rows=slice(N, T), bf16_operands=True,
                                        with_entropy=with_entropy)


def test_forward_parity(dcl, ctx, weights):
    prompt = syn.prompt_ids(3, 2, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=0.7, tau_draft=0.98, max_window=32, gen_len=M)
    ctx.set_prompt(prompt, cfg)
    # drafts beyond the window (from the input generator) so the forward input is not all MASK
    x = np.full((2, T), TINY.mask_id, np.int32)
    x[:, :N] = prompt
    x[:, N + 40:] = np.random.default_rng(0).integers(0, TINY.mask_id, (2, M - 40))
    ctx.set_state(x, np.full(2, N, np.int32))
    logits = torch.zeros(2 * M, TINY.vocab, dtype=torch.bfloat16, device="cuda")
    top1 = torch.zeros(2 * M, dtype=torch.int32, device="cuda")
    p1 = torch.zeros(2 * M, device="cuda")
    p2 = torch.zeros(2 * M, device="cuda")
    ctx.forward_debug(logits, top1, p1, p2)
    xin, _ = ctx.get_state()
    xr = x.copy()
    xr[:, N:N + 32] = TINY.mask_id                          # Eq. remasking of [p, p+L)
    assert (xin == xr).all()
    h = torch.zeros(2 * T, TINY.d_model, device="cuda")
    for b in range(2):
        z = model.logits(weights, model.forward_hidden(TINY, weights, xr[b])[N:])
        zg = logits[b * M:(b + 1) * M].float().cpu().numpy()
        assert (np.abs(zg - z).max(axis=1) / np.abs(z).max(axis=1)).max() <= 2e-2
        ids_o, p1_o, p2_o = _predict(weights)(xr[b])
        sl = slice(b * M, (b + 1) * M)
        assert np.abs(p1[sl].cpu().numpy() - p1_o).max() <= E2E_TOL
        assert np.abs(p2[sl].cpu().numpy() - p2_o).max() <= E2E_TOL
        sure = p1_o - p2_o > E2E_TOL
        assert (top1[sl].cpu().numpy()[sure] == ids_o[sure]).all()
        for layer in range(-1, TINY.n_layers):
            ref = model.forward_hidden(TINY, weights, xr[b], bf16_operands=True, upto_layer=layer)
            ctx.debug_hidden(layer, h)
            got = h[b * T:(b + 1) * T].cpu().numpy()
            err = np.sqrt(((got - ref) ** 2).mean(axis=1)) / np.sqrt((ref ** 2).mean(axis=1))
            assert err.max() <= 3e-3, (layer, err.max())


def _check_step(x0, p0, x1, k1, ids, c1, c2, cfg, L, tol, conf=None):
    """Check one GPU step (x0, p0) -> (x1, p0 + k1) of one row against the oracle's
    predictions (ids, c1, c2 over the generation positions; conf, if given, is the
    confidence the thresholds see instead of c1).  Decisions with a margin above tol
    must match the oracle; the rest must be valid outcomes.  Returns (number of
    decisions checked exactly, number of near ties)."""
    full_id = np.zeros(T, np.int64)
    full_c = np.zeros(T)
    gap = np.full(T, np.inf)
    full_id[N:], full_c[N:], gap[N:] = ids, c1 if conf is None else conf, c1 - c2
    w_eff = min(L, T - p0)
    exact = near = 0
    # K: between the prefix lengths obtained with the threshold moved by -tol / +tol
    k_lo = min(max(decode.window_length(full_c[p0:p0 + w_eff], cfg.tau_commit + tol), cfg.min_commit), w_eff)
    k_hi = min(max(decode.window_length(full_c[p0:p0 + w_eff], cfg.tau_commit - tol), cfg.min_commit), w_eff)
    assert k_lo <= k1 <= k_hi, (k_lo, k1, k_hi)
    if k_lo == k_hi:
        exact += 1
    else:
        near += 1
    # committed ids: the oracle's top-1 wherever its top-1/top-2 gap exceeds tol
    for i in range(p0, p0 + k1):
        if gap[i] > tol:
            assert x1[i] == full_id[i]
            exact += 1
        else:
            near += 1
    assert (x1[:p0] == x0[:p0]).all()                         # committed prefix unchanged
    assert (x1[p0 + k1:min(p0 + L, T)] == TINY.mask_id).all()  # rest of the window stays masked
    # drafts at i >= p + L: replaced by the top-1 id exactly when c_i > tau_draft; in the
    # App. E mode only along the unbroken chain from p + L
    chain = "open"  # "open": chain intact so far; "broken": surely broken; "unknown"
    for i in range(p0 + L, T):
        near_thr = abs(full_c[i] - cfg.tau_draft) <= tol
        passes = full_c[i] > cfg.tau_draft
        valid = x1[i] == x0[i] or x1[i] == full_id[i] or gap[i] <= tol
        if cfg.contiguous_drafts and chain == "broken":
            assert x1[i] == x0[i]
            exact += 1
        elif (cfg.contiguous_drafts and chain == "unknown") or near_thr:
            assert valid
            near += 1
            if cfg.contiguous_drafts:
                chain = "unknown"
        elif not passes:
            assert x1[i] == x0[i]
            exact += 1
            chain = "broken"
        elif gap[i] > tol:
            assert x1[i] == full_id[i]
            exact += 1
        else:
            assert valid and x1[i] != -1
            near += 1
    return exact, near


@pytest.mark.parametrize("seed,tau_c,tau_d,L,contig,conf", [(0, 0.7, 0.98, 32, 0, 0), (1, 0.5, 0.8, 16, 0, 0),
                                                            (2, 0.9, 0.6, 8, 1, 0), (3, 0.3, 0.95, 64, 0, 0),
                                                            (4, 0.3, 0.6, 32, 0, 1), (5, 0.5, 0.9, 16, 1, 1)])
def test_teacher_forced_steps(dcl, ctx, weights, seed, tau_c, tau_d, L, contig, conf):
    """Every state of the oracle's own trajectory is loaded into the GPU, one GPU step
    runs, and the result is checked against the oracle's decision at that state (conf
    = 1: the thresholds see exp(-H); the step's Eq. entropy_bound is checked too)."""
    B = 2
    prompt = syn.prompt_ids(100 + seed, B, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=tau_c, tau_draft=tau_d, max_window=L, gen_len=M,
                            contiguous_drafts=contig, confidence=conf)
    ocfg = decode.DecodeConfig(tau_commit=tau_c, tau_draft=tau_d, max_window=L, gen_len=M,
                               contiguous_drafts=bool(contig), confidence=conf)
    ref = decode.generate(_predict(weights, with_entropy=True), prompt, ocfg, TINY.mask_id)
    ctx.set_prompt(prompt, cfg)
    p = np.full(B, N, np.int64)
    exact = near = 0
    for s, (xin, pr) in enumerate(zip(ref["inputs"], ref["preds"])):
        ctx.set_state(xin, p.astype(np.int32))  # also clears the entropy-bound accumulators
        _, st, _ = ctx.generate(max_steps=1, out=False, check=False)
        x1, p1 = ctx.get_state()
        k = p1 - p
        bound = 0.0
        for b in range(B):
            if p[b] >= T:
                assert k[b] == 0 and (x1[b] == xin[b]).all() and p1[b] == p[b]
                continue
            assert p1[b] == p[b] + k[b] and 1 <= k[b] <= min(L, T - p[b])
            c = decode.entropy_confidence(pr[3, b]) if conf else None
            e, n = _check_step(xin[b], int(p[b]), x1[b], int(k[b]), pr[0, b], pr[1, b], pr[2, b],
                               ocfg, L, E2E_TOL, conf=c)
            exact += e
            near += n
            H = pr[3, b][int(p[b]) - N:int(p[b]) - N + int(k[b])]
            bound += decode.jpde_bound(H)
        # Eq. entropy_bound of the sets the GPU committed, with the oracle's entropies:
        # each H within the end-to-end tolerance scaled by H (|dH| <= 2 H |dz|)
        assert abs(st.jpde_bound - bound) <= 0.05 * (bound + 1.0) * max(1, int(k.max())), (s, st.jpde_bound, bound)
        p = p + ref["k"][s]
    assert exact > 0
    print(f"teacher-forced: {exact} decisions exact, {near} near ties (|margin| <= {E2E_TOL})")


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_free_running_generation(dcl, ctx, weights, seed):
    """GPU and oracle generations agree up to the first step whose oracle decision had a
    margin below E2E_TOL; the fraction of such divergences is reported."""
    prompt = syn.prompt_ids(200 + seed, 1, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=0.7, tau_draft=0.98, max_window=32, gen_len=M)
    ocfg = decode.DecodeConfig(tau_commit=0.7, tau_draft=0.98, max_window=32, gen_len=M)
    ctx.set_prompt(prompt, cfg)
    states = []
    for _ in range(2 * M):
        x, p = ctx.get_state()
        states.append((x[0].copy(), int(p[0])))
        if p[0] >= T:
            break
        ctx.step()
    assert states[-1][1] == T
    ref = decode.generate(_predict(weights), prompt, ocfg, TINY.mask_id)
    p_o = N
    L = ocfg.window()
    outside = lambda p: (np.arange(T) < p) | (np.arange(T) >= p + L)  # not re-masked this step
    for s, (xin, pr) in enumerate(zip(ref["inputs"], ref["preds"])):
        xg, pg = states[s]
        if pg != p_o or not (xg == xin[0])[outside(p_o)].all():
            # the trajectories split at step s-1: that decision must have been a near tie
            prev = ref["preds"][s - 1][:, 0]
            c = np.zeros(T)
            c[N:] = prev[1]
            g = np.full(T, np.inf)
            g[N:] = prev[1] - prev[2]
            p_prev = p_o - int(ref["k"][s - 1, 0])
            assert (np.abs(c[p_prev:] - ocfg.tau_commit) <= E2E_TOL).any() or \
                (np.abs(c[p_prev:] - ocfg.tau_draft) <= E2E_TOL).any() or (g[p_prev:] <= E2E_TOL).any(), \
                "GPU and oracle diverged at a decision with a clear margin"
            print(f"seed {seed}: trajectories split after {s} of {ref['n_iter']} steps at a near tie")
            return
        p_o += int(ref["k"][s, 0])
    out_g = states[-1][0][N:]
    assert (out_g == ref["x"][0, N:]).all()
    assert len(states) - 1 == ref["n_iter"]
    print(f"seed {seed}: identical trajectories ({ref['n_iter']} steps)")


def test_forward_entropy_parity(dcl, ctx, weights):
    """The marginal entropy from the fused LM head against the oracle (bf16 operands), and
    the confidence the thresholds see with confidence = 1: exp(-H) <= p1."""
    prompt = syn.prompt_ids(13, 2, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=0.5, tau_draft=0.9, max_window=32, gen_len=M, confidence=1)
    ctx.set_prompt(prompt, cfg)
    x = np.full((2, T), TINY.mask_id, np.int32)
    x[:, :N] = prompt
    x[:, N + 40:] = np.random.default_rng(1).integers(0, TINY.mask_id, (2, M - 40))
    ctx.set_state(x, np.full(2, N, np.int32))
    p1 = torch.zeros(2 * M, device="cuda")
    conf = torch.zeros(2 * M, device="cuda")
    ent = torch.zeros(2 * M, device="cuda")
    ctx.forward_debug(p1=p1, conf=conf, entropy=ent)
    xr = x.copy()
    xr[:, N:N + 32] = TINY.mask_id
    worst = 0.0
    for b in range(2):
        sl = slice(b * M, (b + 1) * M)
        _, p1_o, _, H_o = _predict(weights, with_entropy=True)(xr[b])
        gH, gc, gp1 = ent[sl].cpu().numpy(), conf[sl].cpu().numpy(), p1[sl].cpu().numpy()
        worst = max(worst, float(np.abs(gH - H_o).max()))
        # the end-to-end logit drift (up to ~0.1 on this model) moves H by <= 2 H |dz|
        assert (np.abs(gH - H_o) <= 0.2 * H_o + 1e-3).all()
        assert np.abs(gc - np.exp(-gH.astype(np.float64))).max() <= 1e-6
        assert (gc <= gp1 + 1e-6).all()
    print(f"entropy: max |H_gpu - H| = {worst:.2e}")


def test_entropy_bound_of_sequential_decoding_is_zero(dcl, ctx, weights):
    prompt = syn.prompt_ids(17, 2, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=1.0, tau_draft=2.0, max_window=16, gen_len=M, confidence=1)
    ctx.set_prompt(prompt, cfg)
    out, st, _ = ctx.generate(max_steps=2 * M)
    assert st.steps == M and st.tokens == 2 * M and st.jpde_bound == 0.0
    cfg = dcl.decode_config(tau_commit=0.0, tau_draft=2.0, max_window=16, gen_len=M, confidence=1)
    ctx.set_prompt(prompt, cfg)
    _, st, _ = ctx.generate(max_steps=2 * M)
    assert st.steps == M // 16 and st.jpde_bound > 0.0
    ctx.restart()  # restart clears the accumulated bound: the same run gives the same total
    _, st2, _ = ctx.generate(max_steps=2 * M)
    assert st2.jpde_bound == st.jpde_bound


def test_generate_counts_and_progress(dcl, ctx, weights):
    prompt = syn.prompt_ids(9, 3, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=0.7, tau_draft=0.98, max_window=32, gen_len=M)
    ctx.set_prompt(prompt, cfg)
    out, st, status = ctx.generate(max_steps=4 * M)
    assert status == dcl.DCL_OK and st.done == 1 and st.tokens == 3 * M and 1 <= st.steps <= M
    x, p = ctx.get_state()
    assert (p == T).all() and (x[:, N:] == out).all() and (x[:, :N] == prompt).all()
    # restart replays the same trajectory (the step is deterministic)
    ctx.restart()
    out2, st2, _ = ctx.generate(max_steps=4 * M)
    assert (out2 == out).all() and st2.steps == st.steps


def test_tau_commit_one_is_sequential(dcl, ctx, weights):
    prompt = syn.prompt_ids(7, 1, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=1.0, tau_draft=2.0, max_window=16, gen_len=M)
    ctx.set_prompt(prompt, cfg)
    out, st, _ = ctx.generate(max_steps=2 * M)
    assert st.steps == M and st.tokens == M


def test_tau_commit_zero_fills_windows(dcl, ctx, weights):
    prompt = syn.prompt_ids(8, 1, N, TINY.mask_id)
    cfg = dcl.decode_config(tau_commit=0.0, tau_draft=0.98, max_window=24, gen_len=M)
    ctx.set_prompt(prompt, cfg)
    ks = []
    for _ in range(M):
        ks.append(int(ctx.step(return_k=True)[0]))
        if sum(ks) >= M:
            break
    assert ks == [24, 24, 16]


def test_error_statuses(dcl, weights):
    with dcl.Context(TINY, max_batch=1, max_seq=T) as c:
        assert dcl.lib().dcl_step(c.ptr, None) == dcl.DCL_ERR_STATE
        assert dcl.lib().dcl_restart(c.ptr) == dcl.DCL_ERR_STATE
        cfg = dcl.decode_config(gen_len=M)
        bad = syn.prompt_ids(0, 1, N, TINY.mask_id)
        bad[0, 3] = TINY.vocab
        with pytest.raises(dcl.DcleapError) as e:
            c.set_prompt(bad, cfg)
        assert e.value.status == dcl.DCL_ERR_INVALID_ARG
        with pytest.raises(dcl.DcleapError):
            c.set_prompt(syn.prompt_ids(0, 2, N, TINY.mask_id), cfg)   # batch > max_batch
        with pytest.raises(dcl.DcleapError) as e:  # the cache needs 32-aligned blocks
            c.set_prompt(syn.prompt_ids(0, 1, N, TINY.mask_id), dcl.decode_config(gen_len=M, kv_cache=1, block_len=16))
        assert e.value.status == dcl.DCL_ERR_UNSUPPORTED
        with pytest.raises(dcl.DcleapError) as e:
            c.set_prompt(syn.prompt_ids(0, 1, N, TINY.mask_id), dcl.decode_config(gen_len=M, kv_cache=3))
        assert e.value.status == dcl.DCL_ERR_INVALID_ARG
        c.load_weights(weights)
        c.set_prompt(syn.prompt_ids(0, 1, N, TINY.mask_id), cfg)
        x, p = c.get_state()
        with pytest.raises(dcl.DcleapError):
            c.set_state(x, np.array([T + 1], np.int32))
        out, st, status = c.generate(max_steps=1, check=False)
        assert status == dcl.DCL_ERR_TIMEOUT and st.done == 0 and st.steps == 1
        out, st, status = c.generate(max_steps=10 * M)
        assert status == dcl.DCL_OK and st.done == 1
    with pytest.raises(dcl.DcleapError) as e:
        dcl.Context(syn.ModelShape(1, 100, 2, 2, 64, 128, 64, 63, 1e4), 1, 8)  # d_model % 128
    assert e.value.status == dcl.DCL_ERR_UNSUPPORTED


def test_near_tie_divergence_fraction(dcl, ctx, weights):
    """32 free-running generations (prompt 32, gen 64, window 32, thresholds 0.7 / 0.98) on
    the GPU and in the oracle: no split may follow a decision whose oracle margin exceeds
    the end-to-end drift E2E_TOL; the fraction of diverged sequences and the margins at the
    splits are reported."""
    import bench
    r = bench.near_tie_study(ctx, dcl, TINY, weights, N, M, 32, 0.7, 0.98, range(32), tol=1e-3, drift=E2E_TOL)
    print("near-tie study:", {k: v for k, v in r.items() if k != "split_margins"},
          "margins at the splits:", [f"{m:.1e}" for m in sorted(r["split_margins"])])
    assert r["split_clear"] == 0
    assert r["identical"] + r["split_near_tie"] + r["split_within_drift"] == 32
