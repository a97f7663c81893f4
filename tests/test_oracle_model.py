"""Pins of the forward / confidence oracle (Sec. 2.1 Eq. 2; top-1 of Eq. threshold_pd;
top-2 of Sec. 2.2; bidirectional attention of App. B.2).

The oracle is checked against library routines written independently of it
(scipy softmax, torch scaled_dot_product_attention / rms_norm / silu, RoPE as a
complex rotation), closed forms, invariants and brute force.
"""
import itertools
import math

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

from oracle import model
import synthetic as syn

TINY = syn.SHAPES["tiny"]


# ------------------------------------------------------------- softmax, top-1/2

def test_softmax_normalised_and_matches_library():
    rng = np.random.default_rng(0)
    z = rng.normal(0, 8, size=(50, 1000))
    p = model.softmax(z)
    assert np.abs(p.sum(axis=1) - 1.0).max() < 1e-12
    assert np.allclose(p, scipy.special.softmax(z, axis=1), rtol=1e-12, atol=0)


def test_confidence_matches_library_softmax():
    rng = np.random.default_rng(1)
    z = rng.normal(0, 6, size=(64, 4096))
    ids, p1, p2 = model.confidence(z)
    ref = scipy.special.softmax(z, axis=1)
    srt = np.sort(ref, axis=1)
    assert (ids == np.argmax(ref, axis=1)).all()
    assert np.allclose(p1, srt[:, -1], rtol=1e-12, atol=0)
    assert np.allclose(p2, srt[:, -2], rtol=1e-12, atol=0)
    V = z.shape[1]
    assert (p1 >= 1.0 / V).all() and (p1 <= 1.0).all() and (p2 <= p1).all()


@pytest.mark.parametrize("V", [2, 3, 8])
def test_confidence_brute_force_small_vocab(V):
    grid = [-1.0, 0.0, 0.5, 2.0]
    rows = list(itertools.product(grid, repeat=V)) if V <= 3 else \
        [tuple(np.random.default_rng(s).choice(grid, V)) for s in range(400)]
    ids, p1, p2 = model.confidence(np.array(rows))
    for r, (row) in enumerate(rows):
        e = [math.exp(v) for v in row]
        tot = sum(e)
        best = max(row)
        first = row.index(best)                       # ties: lowest index
        others = [e[i] for i in range(V) if i != first]
        assert ids[r] == first
        assert abs(p1[r] - e[first] / tot) < 1e-14
        assert abs(p2[r] - max(others) / tot) < 1e-14


def test_confidence_tie_gives_equal_top2():
    ids, p1, p2 = model.confidence(np.array([[1.0, 3.0, 3.0, 0.0]]))
    assert ids[0] == 1 and p1[0] == p2[0]


# ----------------------------------------------------------------- RMSNorm, RoPE

def test_rms_norm_unit_rms_and_library():
    rng = np.random.default_rng(2)
    x = rng.normal(0, 3, size=(17, 96))
    y = model.rms_norm(x, np.ones(96), 0.0)
    assert np.allclose(np.sqrt((y * y).mean(axis=1)), 1.0, atol=1e-12)
    g = rng.normal(1, 0.2, 96)
    ref = F.rms_norm(torch.tensor(x), (96,), torch.tensor(g), eps=1e-5).numpy()
    assert np.allclose(model.rms_norm(x, g, 1e-5), ref, rtol=1e-12, atol=1e-12)


def test_rope_is_complex_rotation():
    rng = np.random.default_rng(3)
    T, heads, hd, theta = 33, 3, 16, 500.0
    x = rng.normal(size=(T, heads, hd))
    y = model.apply_rope(x, model.rope_angles(T, hd, theta))
    half = hd // 2
    zc = x[..., :half] + 1j * x[..., half:]
    w = np.array([theta ** (-(2 * j) / hd) for j in range(half)])
    rot = np.exp(1j * np.arange(T)[:, None, None] * w[None, None, :])
    ref = zc * rot
    assert np.allclose(y[..., :half], ref.real, atol=1e-12)
    assert np.allclose(y[..., half:], ref.imag, atol=1e-12)
    # position 0 is the identity; norms are preserved
    assert np.allclose(y[0], x[0], atol=0)
    assert np.allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), atol=1e-12)


def test_rope_scores_depend_only_on_relative_position():
    rng = np.random.default_rng(4)
    hd, theta = 32, 10000.0
    q, k = rng.normal(size=(1, 1, hd)), rng.normal(size=(1, 1, hd))
    ang = model.rope_angles(64, hd, theta)

    def score(m, n):
        return float((model.apply_rope(q, ang[m:m + 1]) * model.apply_rope(k, ang[n:n + 1])).sum())
    assert abs(score(5, 2) - score(40, 37)) < 1e-10
    assert abs(score(0, 9) - score(50, 59)) < 1e-10


# --------------------------------------------------------------------- attention

def test_attention_matches_library_non_causal_gqa():
    rng = np.random.default_rng(5)
    T, H, G, hd = 23, 6, 2, 16
    q, k, v = rng.normal(size=(T, H, hd)), rng.normal(size=(T, G, hd)), rng.normal(size=(T, G, hd))
    out = model.attention(q, k, v).reshape(T, H, hd)
    kt = torch.tensor(k).repeat_interleave(H // G, dim=1)
    vt = torch.tensor(v).repeat_interleave(H // G, dim=1)
    ref = F.scaled_dot_product_attention(torch.tensor(q).transpose(0, 1), kt.transpose(0, 1),
                                         vt.transpose(0, 1), is_causal=False).transpose(0, 1)
    assert np.allclose(out, ref.numpy(), rtol=1e-10, atol=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(6)
    # a single position attends only to itself: output = V
    v = rng.normal(size=(1, 2, 8))
    out = model.attention(rng.normal(size=(1, 4, 8)), rng.normal(size=(1, 2, 8)), v)
    assert np.allclose(out.reshape(1, 4, 8), np.repeat(v, 2, axis=1))
    # zero queries give uniform weights over ALL positions (non-causal): every row is the mean of V
    T = 9
    v = rng.normal(size=(T, 1, 8))
    out = model.attention(np.zeros((T, 1, 8)), rng.normal(size=(T, 1, 8)), v)
    assert np.allclose(out, np.broadcast_to(v.mean(axis=0).reshape(1, 8), (T, 8)))


def test_silu_matches_library():
    x = np.linspace(-30, 30, 1001)
    assert np.allclose(model.silu(x), F.silu(torch.tensor(x)).numpy(), rtol=1e-13, atol=1e-300)
    assert model.silu(np.array([0.0]))[0] == 0.0


# --------------------------------------------------------------- whole forward

def test_to_bf16_matches_torch_rounding():
    rng = np.random.default_rng(9)
    x = np.concatenate([rng.normal(0, 1, 10000), rng.normal(0, 1e4, 1000),
                        # exact halfway cases between bf16 neighbours (ties to even)
                        (np.arange(1, 200, dtype=np.float64) * 2 + 1) * 2 ** -8 + 1.0])
    ref = torch.tensor(x).float().bfloat16().double().numpy()
    assert (model.to_bf16(x) == ref).all()


def _torch_forward(shape, w, tokens, bf16=False):
    """Independent fp64 restatement with torch library ops (F.linear, F.rms_norm, SDPA, F.silu)
    and RoPE as a complex multiplication; bf16=True casts matrix-product operands with
    torch's own bf16 conversion at the points a bf16 model stores them."""
    t = lambda a: torch.tensor(np.asarray(a, np.float64))
    c = (lambda a: a.float().bfloat16().double()) if bf16 else (lambda a: a)
    T = len(tokens)
    H, G, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    h = t(w["embed"])[torch.tensor(tokens, dtype=torch.long)]
    freqs = torch.tensor([shape.rope_theta ** (-(2 * j) / hd) for j in range(hd // 2)], dtype=torch.float64)
    rot = torch.polar(torch.ones(T, hd // 2, dtype=torch.float64),
                      torch.arange(T, dtype=torch.float64)[:, None] * freqs[None, :])

    def rope(x):                               # x [T, heads, hd]
        zc = torch.complex(x[..., :hd // 2], x[..., hd // 2:]) * rot[:, None, :]
        return torch.cat([zc.real, zc.imag], dim=-1)
    for lw in w["layers"]:
        xn = c(F.rms_norm(h, (shape.d_model,), t(lw["attn_norm"]), eps=shape.rms_eps))
        q = c(rope(F.linear(xn, t(lw["wq"])).view(T, H, hd)))
        k = c(rope(F.linear(xn, t(lw["wk"])).view(T, G, hd))).repeat_interleave(H // G, dim=1)
        v = c(F.linear(xn, t(lw["wv"])).view(T, G, hd)).repeat_interleave(H // G, dim=1)
        a = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                           is_causal=False).transpose(0, 1).reshape(T, H * hd)
        h = h + F.linear(c(a), t(lw["wo"]))
        xn = c(F.rms_norm(h, (shape.d_model,), t(lw["mlp_norm"]), eps=shape.rms_eps))
        h = h + F.linear(c(F.silu(F.linear(xn, t(lw["w_gate"]))) * F.linear(xn, t(lw["w_up"]))),
                         t(lw["w_down"]))
    h = c(F.rms_norm(h, (shape.d_model,), t(w["final_norm"]), eps=shape.rms_eps))
    return F.linear(h, t(w["lm_head"])).numpy()


def test_tiny_forward_matches_torch_restatement():
    w = syn.model_weights(TINY, 0, lm_head_scale=40.0, norm_gain_std=0.1)
    tokens = np.concatenate([syn.prompt_ids(0, 1, 32, TINY.mask_id)[0],
                             np.full(64, TINY.mask_id, np.int32)])
    tokens[40] = 7
    z = model.logits(w, model.forward_hidden(TINY, w, tokens))
    ref = _torch_forward(TINY, w, tokens)
    assert np.abs(z - ref).max() <= 1e-9 * np.abs(ref).max()


def test_tiny_forward_bf16_operands_matches_torch_restatement():
    w = syn.model_weights(TINY, 0, lm_head_scale=40.0, norm_gain_std=0.1)
    tokens = np.concatenate([syn.prompt_ids(5, 1, 32, TINY.mask_id)[0],
                             np.full(64, TINY.mask_id, np.int32)])
    z = model.logits(w, model.forward_hidden(TINY, w, tokens, bf16_operands=True))
    ref = _torch_forward(TINY, w, tokens, bf16=True)
    # identical rounding points; only fp64 summation order differs (it may move a value
    # across a bf16 rounding boundary, so allow a few bf16 ulps in rare elements)
    assert np.abs(z - ref).max() <= 1e-4 * np.abs(ref).max()
    # and the rounding is real: the pure forward differs
    z0 = model.logits(w, model.forward_hidden(TINY, w, tokens))
    assert np.abs(z0 - z).max() > 1e-3


def test_upto_layer_returns_residual_stream():
    w = syn.model_weights(TINY, 1)
    tokens = syn.prompt_ids(2, 1, 20, TINY.mask_id)[0]
    h_emb = model.forward_hidden(TINY, w, tokens, upto_layer=-1)
    assert np.array_equal(h_emb, np.asarray(w["embed"], np.float64)[tokens])
    h0 = model.forward_hidden(TINY, w, tokens, upto_layer=0)
    ang = model.rope_angles(20, TINY.head_dim, TINY.rope_theta)
    assert np.array_equal(h0, model.block(TINY, w["layers"][0], h_emb, ang))


def test_gqa_forward_matches_torch_restatement():
    shape = syn.ModelShape(2, 64, 4, 2, 16, 128, 97, 96, 1e6)
    w = syn.model_weights(shape, 3, lm_head_scale=10.0, norm_gain_std=0.2)
    tokens = syn.prompt_ids(4, 1, 21, shape.mask_id)[0]
    z = model.logits(w, model.forward_hidden(shape, w, tokens))
    ref = _torch_forward(shape, w, tokens)
    assert np.abs(z - ref).max() <= 1e-9 * np.abs(ref).max()


def test_forward_is_bidirectional():
    """Changing the LAST token changes the prediction at the first generation position;
    a causal forward would leave every earlier position unchanged."""
    w = syn.model_weights(TINY, 0, lm_head_scale=40.0)
    tokens = np.concatenate([syn.prompt_ids(1, 1, 32, TINY.mask_id)[0],
                             np.full(64, TINY.mask_id, np.int32)])
    h0 = model.forward_hidden(TINY, w, tokens)
    tokens2 = tokens.copy()
    tokens2[-1] = 5
    h1 = model.forward_hidden(TINY, w, tokens2)
    assert np.abs(h0[32] - h1[32]).max() > 1e-6
    assert np.abs(h0[0] - h1[0]).max() > 1e-6


def test_forward_rejects_bad_token():
    w = syn.model_weights(TINY, 0)
    with pytest.raises(ValueError):
        model.forward_hidden(TINY, w, np.array([0, TINY.vocab]))
