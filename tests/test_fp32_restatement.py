"""Where the full-size block tolerance and the end-to-end splits come from (no GPU).

The GPU accumulates every matrix product in fp32; the oracle in fp64.  Both round the same
operands to bf16 (the RMSNorm outputs, q / k after RoPE, v, the attention output and the
SwiGLU output).  At the LLaDA-8B and Dream-7B shapes, fp32 accumulation over K = 4096 ..
18944 products moves enough values across bf16 rounding boundaries that even an exact
IEEE-fp32 evaluation differs visibly from the fp64 oracle.  This test makes that
evaluation, in PyTorch on the CPU from the same seeded weights and tokens, and checks that
it lies within the bound the GPU parity tests use for one block (relative rms error per
row: 3.5e-3 mean, 6e-3 max) but clearly away from zero: the bound is what a correct fp32
implementation reaches, not slack.

The same fp32 evaluation, run through whole generations of the 2-layer model, also
shows where the GPU's free-running generations part from the oracle's: an exact fp32
implementation parts from the fp64 oracle about as often, and at decisions whose oracle
margins lie in the same band (above the 1e-3 near-tie margin, inside the 5e-2 end-to-end
drift of this random model).
"""
import numpy as np
import pytest
import torch

import synthetic as syn
from oracle import model

TOL_BLOCK = (3.5e-3, 6e-3)


def _bf(t):
    return t.to(torch.bfloat16).to(torch.float32)


def _block_fp32(shape, lw, h, angles):
    """One block in IEEE fp32 (torch, CPU) with the oracle's bf16 rounding points."""
    T = h.shape[0]
    H, G, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    f = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))  # noqa: E731

    def rms(x, g):
        return x * torch.rsqrt((x * x).mean(dim=-1, keepdim=True) + shape.rms_eps) * f(g)

    def rope(x):
        c, s = torch.cos(angles)[:, None, :], torch.sin(angles)[:, None, :]
        x1, x2 = x[..., :hd // 2], x[..., hd // 2:]
        return torch.cat([x1 * c - x2 * s, x2 * c + x1 * s], dim=-1)

    xn = _bf(rms(h, lw["attn_norm"]))
    q = _bf(rope((xn @ f(lw["wq"]).T).reshape(T, H, hd)))
    k = _bf(rope((xn @ f(lw["wk"]).T).reshape(T, G, hd)))
    v = _bf((xn @ f(lw["wv"]).T).reshape(T, G, hd))
    rep = H // G
    k = k.repeat_interleave(rep, dim=1)
    v = v.repeat_interleave(rep, dim=1)
    s = torch.einsum("thd,shd->hts", q, k) / np.float32(np.sqrt(hd))
    a = torch.einsum("hts,shd->thd", torch.softmax(s, dim=-1), v).reshape(T, H * hd)
    h = h + _bf(a) @ f(lw["wo"]).T
    xn = _bf(rms(h, lw["mlp_norm"]))
    g = xn @ f(lw["w_gate"]).T
    act = _bf(g * torch.sigmoid(g) * (xn @ f(lw["w_up"]).T))
    return h + act @ f(lw["w_down"]).T


@pytest.mark.parametrize("name,seed,N,M", [("llada8b", 1, 256, 256), ("dream7b", 2, 384, 512)])
def test_fp32_block_zero_lies_within_the_gpu_bound(name, seed, N, M):
    sh = syn.SHAPES[name]
    T = N + M
    torch.set_num_threads(max(1, torch.get_num_threads()))
    prompt = syn.prompt_ids(1000, 1, N, sh.mask_id)[0]
    x = np.concatenate([prompt, np.full(M, sh.mask_id, np.int32)])
    uniq, inv = np.unique(x, return_inverse=True)
    h0 = syn.embed_rows(sh, seed, uniq, 0.02)[inv]
    lw = syn.model_weights(sh, seed, 0.02, 12.0, 0.0, layers=(0,), global_tensors=False)["layers"][0]
    angles = model.rope_angles(T, sh.head_dim, sh.rope_theta)
    ref = model.block(sh, lw, h0.astype(np.float64), angles, bf16_operands=True)
    with torch.no_grad():
        got = _block_fp32(sh, lw, torch.from_numpy(h0), torch.from_numpy(angles.astype(np.float32))).numpy()
    err = np.sqrt(((got - ref) ** 2).mean(axis=1)) / np.sqrt((ref ** 2).mean(axis=1))
    print(f"{name} block 0, IEEE fp32 vs fp64 oracle: relative rms per row mean {err.mean():.2e} max {err.max():.2e}")
    assert err.mean() <= TOL_BLOCK[0] and err.max() <= TOL_BLOCK[1]
    assert err.mean() >= 0.1 * TOL_BLOCK[0]  # the rounding-boundary effect is real, not slack


def _predict_fp32(shape, w, N):
    """Forward + confidence of the bf16-operand model in IEEE fp32 (torch, CPU), the way
    the GPU evaluates it: fp32 logits of the bf16 final-normed rows, p1 = 1 / sum exp(z - m),
    p2 from the largest logit at another index."""
    f = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))  # noqa: E731
    E, LM, gain = f(w["embed"]), f(w["lm_head"]), f(w["final_norm"])

    def predict(tokens):
        T = len(tokens)
        angles = torch.from_numpy(model.rope_angles(T, shape.head_dim, shape.rope_theta).astype(np.float32))
        with torch.no_grad():
            h = E[torch.from_numpy(np.asarray(tokens, np.int64))]
            for lw in w["layers"]:
                h = _block_fp32(shape, lw, h, angles)
            g = h[N:]
            z = _bf(g * torch.rsqrt((g * g).mean(dim=-1, keepdim=True) + shape.rms_eps) * gain) @ LM.T
            m = z.max(dim=-1, keepdim=True).values
            S = torch.exp(z - m).sum(dim=-1)
            ids = torch.argmax(z, dim=-1)
            z2 = z.clone()
            z2[torch.arange(z.shape[0]), ids] = -torch.inf
            p2 = torch.exp(z2.max(dim=-1).values - m[:, 0]) / S
        return ids.numpy().astype(np.int32), (1.0 / S).double().numpy(), p2.double().numpy()
    return predict


def test_fp32_generations_part_from_the_oracle_as_the_gpu_does():
    """32 free-running generations of the 2-layer model (prompt 32, gen 64, window 32,
    thresholds 0.7 / 0.98; the GPU near-tie study's settings and prompts), fp32 against the
    fp64 oracle: none parts at a decision whose oracle margin exceeds the 5e-2 drift, and
    some part between 1e-3 and 5e-2, as the GPU's do: those splits are the arithmetic's,
    not a kernel's."""
    import bench
    from oracle import decode
    sh = syn.SHAPES["tiny"]
    N, M, L, tc, td = 32, 64, 32, 0.7, 0.98
    w = syn.model_weights(sh, 0, lm_head_scale=40.0, norm_gain_std=0.1)
    cfg = decode.DecodeConfig(tau_commit=tc, tau_draft=td, max_window=L, gen_len=M)
    pred64 = lambda t: model.predict(sh, w, t, rows=slice(N, N + M), bf16_operands=True)  # noqa: E731
    pred32 = _predict_fp32(sh, w, N)
    counts = {"identical": 0, "near_tie": 0, "within_drift": 0, "clear": 0}
    margins = []
    for seed in range(32):
        prompt = syn.prompt_ids(3000 + seed, 1, N, sh.mask_id)
        ref = decode.generate(pred64, prompt, cfg, sh.mask_id)
        alt = decode.generate(pred32, prompt, cfg, sh.mask_id)
        split, p = None, N
        for s, xin in enumerate(ref["inputs"]):
            if s >= len(alt["inputs"]) or not (alt["inputs"][s][0] == xin[0]).all():
                split = s
                break
            p += int(ref["k"][s, 0])
        if split is None and (alt["x"][0] == ref["x"][0]).all():
            counts["identical"] += 1
            continue
        s = (split if split is not None else len(ref["inputs"])) - 1  # the last step both took
        k = int(ref["k"][s, 0])
        mg = bench._step_margin(ref["preds"][s][:, 0], ref["inputs"][s][0], p - k, k, N, L, tc, td)
        margins.append(mg)
        counts["near_tie" if mg <= 1e-3 else "within_drift" if mg <= 5e-2 else "clear"] += 1
    print("fp32 vs fp64 oracle:", counts, "margins at the splits:", [f"{m:.1e}" for m in sorted(margins)])
    assert counts["clear"] == 0
    assert counts["within_drift"] >= 1


def test_fp32_forward_confidence_drift_sets_the_end_to_end_bound():
    """The end-to-end confidence bound of the 2-layer model's GPU tests (5e-2 between the
    GPU's and the bf16-operand oracle's top-1 probability after a whole forward) is what an
    exact fp32 evaluation reaches: over 32 prompts (drafts beyond the window) the fp32
    restatement's p1 drifts from the fp64 oracle's by more than 1e-2 at worst, and stays
    inside 5e-2.  The 1e-3 bound holds for the LM head on identical inputs, where no
    forward precedes it (the GPU tests check that separately)."""
    sh = syn.SHAPES["tiny"]
    N, M = 32, 64
    w = syn.model_weights(sh, 0, lm_head_scale=40.0, norm_gain_std=0.1)
    pred32 = _predict_fp32(sh, w, N)
    worst = []
    for seed in range(32):
        rng = np.random.default_rng(seed)
        x = np.concatenate([syn.prompt_ids(3000 + seed, 1, N, sh.mask_id)[0], np.full(M, sh.mask_id, np.int32)])
        x[N + 40:] = rng.integers(0, sh.mask_id, M - 40)
        p1_64 = model.predict(sh, w, x, rows=slice(N, N + M), bf16_operands=True)[1]
        worst.append(float(np.abs(pred32(x)[1] - p1_64).max()))
    print(f"fp32 vs fp64 top-1 probability after one forward: median {np.median(worst):.2e}, max {max(worst):.2e}")
    assert 1e-2 < max(worst) <= 5e-2
