"""Oracle: bidirectional transformer forward and per-position confidence, fp64.

Test infrastructure only (see ``oracle/__init__.py``).

The paper fixes what the forward produces (Sec. 2.1, Eq. 2: a categorical
distribution per position from one non-causal pass over prompt + generation,
bidirectional per App. B.2) but not the architecture; the architecture below is
the LLaDA/Dream family as configured: RMSNorm, rotate-half RoPE, multi-head (or
grouped-query) attention over ALL positions, SwiGLU MLP, final RMSNorm, untied LM
head, no biases.  Weights are read as given (bf16-exact values) and every
operation runs in float64.

Precision reading.  The paper evaluates bf16 checkpoints but never states where
activations are rounded.  ``bf16_operands=False`` (default) is the pure definition:
nothing is rounded.  ``bf16_operands=True`` is a bf16 model: every operand of a
matrix product is stored in bf16 exactly where a bf16 model stores it - the RMSNorm
outputs, q/k (after RoPE) and v, the attention output, the SwiGLU output and the
final hidden state - while products accumulate, and norms, softmax and the residual
stream are computed, in float64.  The rounding is value -> float32 -> bf16, both
round-to-nearest-even.
"""
from __future__ import annotations

import numpy as np


def to_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bf16 value (via float32; both steps round to nearest even)."""
    b = np.ascontiguousarray(np.asarray(x, dtype=np.float64).astype(np.float32)).view(np.uint32)
    r = ((b + np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)) << np.uint32(16)
    return r.view(np.float32).astype(np.float64).reshape(np.shape(x))


def _maybe_bf16(x, on):
    return to_bf16(x) if on else x


def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * gain over the last axis."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(gain, np.float64)


def rope_angles(n_pos: int, head_dim: int, theta: float) -> np.ndarray:
    """Angle[t, j] = t * theta^(-2j/head_dim) for j < head_dim/2 (positions 0..n_pos-1)."""
    j = np.arange(head_dim // 2, dtype=np.float64)
    inv_freq = theta ** (-2.0 * j / head_dim)
    return np.outer(np.arange(n_pos, dtype=np.float64), inv_freq)


def apply_rope(x: np.ndarray, angles: np.ndarray) -> np.ndarray:
    """Rotate-half RoPE: pairs (j, j + hd/2) rotated by angle[t, j].  x: [T, heads, hd]."""
    half = x.shape[-1] // 2
    c = np.cos(angles)[:, None, :]
    s = np.sin(angles)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """Non-causal softmax(q k^T / sqrt(hd)) v; every query sees every key.

    q: [T, H, hd]; k, v: [T, G, hd] with H a multiple of G (query head h reads kv head
    h // (H/G)).  Returns [T, H*hd].
    """
    T, H, hd = q.shape
    G = k.shape[1]
    rep = H // G
    out = np.empty((T, H, hd), dtype=np.float64)
    for h in range(H):
        g = h // rep
        s = q[:, h, :] @ k[:, g, :].T / np.sqrt(hd)
        s = s - s.max(axis=1, keepdims=True)
        w = np.exp(s)
        w = w / w.sum(axis=1, keepdims=True)
        out[:, h, :] = w @ v[:, g, :]
    return out.reshape(T, H * hd)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def _f64(a):
    return np.asarray(a, dtype=np.float64)


def block(shape, lw: dict, h: np.ndarray, angles: np.ndarray, bf16_operands: bool = False) -> np.ndarray:
    """One transformer block on the residual stream h [T, d] (returns the new stream)."""
    T = h.shape[0]
    H, G, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    r = bf16_operands
    xn = _maybe_bf16(rms_norm(h, lw["attn_norm"], shape.rms_eps), r)
    q = (xn @ _f64(lw["wq"]).T).reshape(T, H, hd)
    k = (xn @ _f64(lw["wk"]).T).reshape(T, G, hd)
    v = _maybe_bf16((xn @ _f64(lw["wv"]).T).reshape(T, G, hd), r)
    q = _maybe_bf16(apply_rope(q, angles), r)
    k = _maybe_bf16(apply_rope(k, angles), r)
    h = h + _maybe_bf16(attention(q, k, v), r) @ _f64(lw["wo"]).T
    xn = _maybe_bf16(rms_norm(h, lw["mlp_norm"], shape.rms_eps), r)
    a = _maybe_bf16(silu(xn @ _f64(lw["w_gate"]).T) * (xn @ _f64(lw["w_up"]).T), r)
    return h + a @ _f64(lw["w_down"]).T


def forward_hidden(shape, weights: dict, tokens: np.ndarray, bf16_operands: bool = False,
                   upto_layer: int = None) -> np.ndarray:
    """Final-normed hidden states [T, d] of one sequence (one full bidirectional pass).

    With ``upto_layer`` = l the un-normed residual stream after block l is returned
    instead (l = -1: after the embedding)."""
    tokens = np.asarray(tokens)
    if tokens.min() < 0 or tokens.max() >= shape.vocab:
        raise ValueError("token id out of range")
    h = _f64(weights["embed"])[tokens]
    if upto_layer == -1:
        return h
    angles = rope_angles(len(tokens), shape.head_dim, shape.rope_theta)
    for li, lw in enumerate(weights["layers"]):
        h = block(shape, lw, h, angles, bf16_operands)
        if upto_layer == li:
            return h
    return _maybe_bf16(rms_norm(h, weights["final_norm"], shape.rms_eps), bf16_operands)


# ---------------------------------------------------------------- approximate prefix cache
# The paper's accelerated setting pairs DC-Leap with a dLLM cache (Sec. 4, Tab. 6) whose
# policy it does not describe.  The reading built here keeps, per layer, the keys and
# values of all T positions of a sequence between steps.  At the first step and whenever
# the block-aligned prefix end N + Bk * floor((p - N) / Bk) changes, a step computes all
# T positions (refreshing every stored key and value); otherwise it computes only the
# positions from that prefix end on: their fresh keys and values overwrite the stored
# ones, and their queries attend to all T stored positions, so the prefix contributes the
# keys and values of its last refresh.


def block_rows(shape, lw: dict, h: np.ndarray, pos: np.ndarray, kv, angles: np.ndarray,
               bf16_operands: bool = False) -> np.ndarray:
    """One block for the rows h [len(pos), d] at positions ``pos`` of one sequence.

    kv = [k, v], each [T, G, hd]: the layer's stored keys and values; the rows' own keys
    and values (after RoPE, rounded like the model stores them) are written at ``pos``
    before their queries attend to all T stored positions.  ``angles`` are the RoPE angles
    of ``pos``."""
    n = h.shape[0]
    H, G, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    r = bf16_operands
    xn = _maybe_bf16(rms_norm(h, lw["attn_norm"], shape.rms_eps), r)
    q = (xn @ _f64(lw["wq"]).T).reshape(n, H, hd)
    k = (xn @ _f64(lw["wk"]).T).reshape(n, G, hd)
    v = _maybe_bf16((xn @ _f64(lw["wv"]).T).reshape(n, G, hd), r)
    q = _maybe_bf16(apply_rope(q, angles), r)
    kv[0][pos] = _maybe_bf16(apply_rope(k, angles), r)
    kv[1][pos] = v
    h = h + _maybe_bf16(attention(q, kv[0], kv[1]), r) @ _f64(lw["wo"]).T
    xn = _maybe_bf16(rms_norm(h, lw["mlp_norm"], shape.rms_eps), r)
    a = _maybe_bf16(silu(xn @ _f64(lw["w_gate"]).T) * (xn @ _f64(lw["w_up"]).T), r)
    return h + a @ _f64(lw["w_down"]).T


def forward_rows(shape, weights: dict, tokens: np.ndarray, pos: np.ndarray, kv_store: list,
                 bf16_operands: bool = False) -> np.ndarray:
    """Final-normed hidden states [len(pos), d] of positions ``pos`` of one sequence,
    reading and updating ``kv_store`` (one [k, v] pair of [T, G, hd] arrays per layer).
    With every position and any store this is ``forward_hidden``."""
    tokens = np.asarray(tokens)
    pos = np.asarray(pos, dtype=np.int64)
    if tokens.min() < 0 or tokens.max() >= shape.vocab:
        raise ValueError("token id out of range")
    h = _f64(weights["embed"])[tokens[pos]]
    angles = rope_angles(len(tokens), shape.head_dim, shape.rope_theta)[pos]
    for lw, kv in zip(weights["layers"], kv_store):
        h = block_rows(shape, lw, h, pos, kv, angles, bf16_operands)
    return _maybe_bf16(rms_norm(h, weights["final_norm"], shape.rms_eps), bf16_operands)


def new_kv_store(shape, T: int) -> list:
    G, hd = shape.n_kv_heads, shape.head_dim
    return [[np.zeros((T, G, hd)), np.zeros((T, G, hd))] for _ in range(shape.n_layers)]


def predict_from(shape, weights: dict, tokens: np.ndarray, start: int, state: dict, n_prompt: int,
                 bf16_operands: bool = False, with_entropy: bool = False, end: int | None = None):
    """(ids, p1, p2) over the generation positions [n_prompt, T) computing only positions
    in [start, end) (end = T by default; the others are returned as -1 / NaN);
    ``state["kv"]`` is the sequence's key / value store, created on first use.  With
    ``with_entropy`` the marginal entropy H of every computed position follows (NaN
    elsewhere)."""
    T = len(tokens)
    if state.get("kv") is None:
        state["kv"] = new_kv_store(shape, T)
    pos = np.arange(start, T if end is None else end)
    hid = forward_rows(shape, weights, tokens, pos, state["kv"], bf16_operands)
    M = T - n_prompt
    ids = np.full(M, -1, np.int32)
    p1 = np.full(M, np.nan)
    p2 = np.full(M, np.nan)
    gen = pos >= n_prompt
    z = logits(weights, hid[gen])
    i, c1, c2 = confidence(z)
    ids[pos[gen] - n_prompt], p1[pos[gen] - n_prompt], p2[pos[gen] - n_prompt] = i, c1, c2
    if not with_entropy:
        return ids, p1, p2
    H = np.full(M, np.nan)
    H[pos[gen] - n_prompt] = entropy(z)
    return ids, p1, p2, H


def logits(weights: dict, hidden: np.ndarray) -> np.ndarray:
    """LM-head logits z = hidden @ W_lm^T, [R, V]."""
    return np.asarray(hidden, np.float64) @ _f64(weights["lm_head"]).T


def softmax(z: np.ndarray) -> np.ndarray:
    """Eq. 2: softmax over the whole vocabulary, per row."""
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - z.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def confidence(z: np.ndarray):
    """Top-1 id, top-1 probability c = max_v P (Eq. threshold_pd) and top-2 probability.

    Ties go to the lowest index; the top-2 probability is the largest probability at an
    index other than the top-1 index, so a tie at the top gives p2 == p1.
    Returns (ids int32 [R], p1 float64 [R], p2 float64 [R]).
    """
    z = np.atleast_2d(np.asarray(z, dtype=np.float64))
    ids = np.argmax(z, axis=1)                      # first maximal index
    m = z[np.arange(z.shape[0]), ids]
    e = np.exp(z - m[:, None])
    s = e.sum(axis=1)
    rest = z.copy()
    rest[np.arange(z.shape[0]), ids] = -np.inf
    z2 = rest.max(axis=1)
    return ids.astype(np.int32), 1.0 / s, np.exp(z2 - m) / s


def entropy(z: np.ndarray) -> np.ndarray:
    """Marginal entropy H = -sum_v P(v) ln P(v) of the Eq. 2 distribution, in nats, per row.

    This is the per-token H(x_i | C) of Eq. entropy_bound; a term with P(v) = 0 (an
    underflowed probability) contributes 0, its limit.
    """
    p = softmax(np.atleast_2d(z))
    with np.errstate(divide="ignore", invalid="ignore"):
        t = np.where(p > 0, p * np.log(p), 0.0)
    return -t.sum(axis=-1)


def predict(shape, weights: dict, tokens: np.ndarray, rows=None, bf16_operands: bool = False,
            with_entropy: bool = False):
    """Forward + confidence: (ids, p1, p2) for positions ``rows`` (all positions by
    default), and the marginal entropy H of every position when ``with_entropy``."""
    hid = forward_hidden(shape, weights, tokens, bf16_operands)
    if rows is not None:
        hid = hid[rows]
    z = logits(weights, hid)
    return confidence(z) + ((entropy(z),) if with_entropy else ())
