"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in the oracle (on the CPU, by replacing one of its functions
for the duration of the test) of the kind a reader could make when restating the paper:
a dropped term, a wrong sign, index or axis, a transposed operand, `>=` for `>`.  The
named pin tests, run against the planted oracle, must fail.  Nothing here touches the
CUDA path.
"""
import os
from dataclasses import replace

import numpy as np
import pytest

from oracle import accept, decode, fp8, model

import synthetic as syn
import test_oracle_accept as tacc
import test_oracle_cache as tcache
import test_oracle_decode as tdec
import test_oracle_entropy as tent
import test_oracle_fp8 as tfp8
import test_oracle_model as tmod
import test_oracle_threshold as tthr

ROOT_GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


# ----------------------------------------------------------------- planted mistakes

def _rms_no_mean(x, gain, eps):  # sum of squares instead of their mean
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.sum(x * x, axis=-1, keepdims=True) + eps) * np.asarray(gain, np.float64)


def _rms_eps_outside(x, gain, eps):  # eps added after the square root
    x = np.asarray(x, dtype=np.float64)
    return x / (np.sqrt(np.mean(x * x, axis=-1, keepdims=True)) + eps) * np.asarray(gain, np.float64)


def _rope_wrong_sign(x, angles):  # rotation by -angle
    half = x.shape[-1] // 2
    c, s = np.cos(angles)[:, None, :], np.sin(angles)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c + x2 * s, x2 * c - x1 * s], axis=-1)


def _rope_interleaved(x, angles):  # pairs (2j, 2j + 1) instead of (j, j + hd/2)
    c, s = np.cos(angles)[:, None, :], np.sin(angles)[:, None, :]
    x1, x2 = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x1 * c - x2 * s
    out[..., 1::2] = x2 * c + x1 * s
    return out


def _rope_angles_wrong_freq(n_pos, head_dim, theta):  # theta^(-j/hd) instead of theta^(-2j/hd)
    j = np.arange(head_dim // 2, dtype=np.float64)
    return np.outer(np.arange(n_pos, dtype=np.float64), theta ** (-1.0 * j / head_dim))


def _attention_variant(causal=False, scale=True, gqa_mod=False, softmax_axis=1):
    def att(q, k, v):
        T, H, hd = q.shape
        G = k.shape[1]
        rep = H // G
        out = np.empty((T, H, hd))
        for h in range(H):
            g = h % G if gqa_mod else h // rep
            s = q[:, h, :] @ k[:, g, :].T
            if scale:
                s = s / np.sqrt(hd)
            if causal:
                s = s + np.triu(np.full((T, T), -np.inf), 1)
            s = s - s.max(axis=softmax_axis, keepdims=True)
            w = np.exp(s)
            w = w / w.sum(axis=softmax_axis, keepdims=True)
            out[:, h, :] = w @ v[:, g, :]
        return out.reshape(T, H * hd)
    return att


def _silu_sigmoid(x):  # sigmoid instead of x * sigmoid
    return 1.0 / (1.0 + np.exp(-x))


def _block_without_mlp_residual(shape, lw, h, angles, bf16_operands=False):
    T = h.shape[0]
    H, G, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    f = lambda a: np.asarray(a, np.float64)  # noqa: E731
    xn = model.rms_norm(h, lw["attn_norm"], shape.rms_eps)
    q = model.apply_rope((xn @ f(lw["wq"]).T).reshape(T, H, hd), angles)
    k = model.apply_rope((xn @ f(lw["wk"]).T).reshape(T, G, hd), angles)
    v = (xn @ f(lw["wv"]).T).reshape(T, G, hd)
    h = h + model.attention(q, k, v) @ f(lw["wo"]).T
    xn = model.rms_norm(h, lw["mlp_norm"], shape.rms_eps)
    a = model.silu(xn @ f(lw["w_gate"]).T) * (xn @ f(lw["w_up"]).T)
    return a @ f(lw["w_down"]).T  # the residual h dropped


def _block_gate_up_swapped(shape, lw, h, angles, bf16_operands=False):
    lw = dict(lw, w_gate=lw["w_up"], w_up=lw["w_gate"])
    return _ORIG["block"](shape, lw, h, angles, bf16_operands)


def _confidence_p2_includes_top(z):
    ids, p1, _ = _ORIG["confidence"](z)
    return ids, p1, p1.copy()  # the "second" is the top itself


def _confidence_last_argmax(z):  # ties to the highest index
    z = np.asarray(z, dtype=np.float64)
    ids = z.shape[-1] - 1 - np.argmax(z[..., ::-1], axis=-1)
    _, p1, p2 = _ORIG["confidence"](z)
    return ids, p1, p2


def _entropy_log2(z):  # bits instead of nats
    return _ORIG["entropy"](z) / np.log(2.0)


def _exceeds_ge(c, tau):  # c >= tau instead of c > tau
    return np.asarray(c, dtype=np.float32) >= np.float32(tau)


def _commit_drafts_from_p_plus_k(x, p, ids, c, cfg, window, k_max=None):  # future region from p + K
    T = x.shape[0]
    w_eff = min(window, T - p)
    K = min(max(decode.window_length(c[p:p + w_eff], cfg.tau_commit), cfg.min_commit), w_eff)
    x[p:p + K] = ids[p:p + K]
    lo = p + K
    ok = decode.exceeds(c[lo:T], cfg.tau_draft)
    seg = x[lo:T]
    seg[ok] = ids[lo:T][ok]
    return K


def _remask_shifted(x, p, window, mask_id):  # one position late
    x[p + 1:min(p + 1 + window, x.shape[0])] = mask_id


def _jpde_sum_only(H_set):  # the max term dropped
    H_set = np.asarray(H_set, dtype=np.float64)
    return float(H_set.sum()) if H_set.size >= 2 else 0.0


def _forward_rows_rope_at_row_index(shape, weights, tokens, pos, kv_store, bf16_operands=False):
    """Suffix rows rotated by their index in the suffix, not their position in the sequence."""
    pos = np.asarray(pos, dtype=np.int64)
    h = np.asarray(weights["embed"], np.float64)[np.asarray(tokens)[pos]]
    angles = model.rope_angles(len(pos), shape.head_dim, shape.rope_theta)
    for lw, kv in zip(weights["layers"], kv_store):
        h = model.block_rows(shape, lw, h, pos, kv, angles, bf16_operands)
    return model.rms_norm(h, weights["final_norm"], shape.rms_eps)


def _block_rows_no_store(shape, lw, h, pos, kv, angles, bf16_operands=False):
    """The rows' fresh keys / values never reach the store their queries attend to."""
    n = h.shape[0]
    H, G, hd = shape.n_heads, shape.n_kv_heads, shape.head_dim
    f = lambda a: np.asarray(a, np.float64)  # noqa: E731
    xn = model.rms_norm(h, lw["attn_norm"], shape.rms_eps)
    q = model.apply_rope((xn @ f(lw["wq"]).T).reshape(n, H, hd), angles)
    h = h + model.attention(q, kv[0], kv[1]) @ f(lw["wo"]).T
    xn = model.rms_norm(h, lw["mlp_norm"], shape.rms_eps)
    a = model.silu(xn @ f(lw["w_gate"]).T) * (xn @ f(lw["w_up"]).T)
    return h + a @ f(lw["w_down"]).T


def _accept_window_from_zero(logits, committed, x, cfg, window):
    """The window taken from position 0 instead of the committed prefix."""
    return _ORIG["accept"](logits, np.zeros_like(committed), x, cfg, window)


def _prefix_end_unaligned(p, n_prompt, block_len):  # p itself, not the block boundary
    return p


def _forward_without_final_norm(shape, weights, tokens, bf16_operands=False, upto_layer=None):
    h = np.asarray(weights["embed"], np.float64)[np.asarray(tokens)]
    if upto_layer == -1:
        return h
    angles = model.rope_angles(len(tokens), shape.head_dim, shape.rope_theta)
    for li, lw in enumerate(weights["layers"]):
        h = model.block(shape, lw, h, angles, bf16_operands)
        if upto_layer == li:
            return h
    return h  # the final RMSNorm dropped


def _entropy_confidence_wrong_sign(H):  # exp(+H)
    return np.exp(np.asarray(H, dtype=np.float64))


def _commit_drafts_ignore_chain(x, p, ids, c, cfg, window, k_max=None):  # App. E flag ignored
    return _ORIG["commit_and_draft"](x, p, ids, c, replace(cfg, contiguous_drafts=False), window, k_max)


def _dual_range_to_the_end(p, n_prompt, T, cfg, refresh):
    """The dual cache computing the whole suffix between refreshes (the prefix cache's range)."""
    if refresh:
        return 0, T
    return decode.prefix_end(p, n_prompt, cfg.block_len), T


def _commit_uncapped(x, p, ids, c, cfg, window, k_max=None):  # the dual cache's block cap ignored
    return _ORIG["commit_and_draft"](x, p, ids, c, cfg, window)


def _threshold_forced_leftmost(x, committed, ids, c, lo, hi, cfg):
    """Forced progress commits the leftmost masked positions, not the most confident."""
    cand = [i for i in range(lo, hi) if not committed[i]]
    passing = [i for i in cand if decode.exceeds(c[i], cfg.tau_commit)]
    chosen = passing if len(passing) >= cfg.min_commit else cand[:cfg.min_commit]
    for i in chosen:
        x[i] = ids[i]
        committed[i] = True
    return chosen


def _threshold_ties_high(x, committed, ids, c, lo, hi, cfg):
    """Equal confidences ranked to the higher position."""
    cand = [i for i in range(lo, hi) if not committed[i]]
    passing = [i for i in cand if decode.exceeds(c[i], cfg.tau_commit)]
    if len(passing) >= cfg.min_commit:
        chosen = passing
    else:
        chosen = sorted(sorted(cand, key=lambda i: (-float(np.float32(c[i])), -i))[:cfg.min_commit])
    for i in chosen:
        x[i] = ids[i]
        committed[i] = True
    return chosen


def _threshold_whole_sequence(x, committed, ids, c, lo, hi, cfg):
    """The rule applied to every masked position to the sequence end, not the block."""
    return _ORIG["threshold_commit"](x, committed, ids, c, lo, x.shape[0], cfg)


def _threshold_recommits(x, committed, ids, c, lo, hi, cfg):
    """Committed positions taken as candidates again (their flags ignored when choosing)."""
    chosen = _ORIG["threshold_commit"](x, np.zeros_like(committed), ids, c, lo, hi, cfg)
    committed[chosen] = True
    return chosen


_ORIG = {"block": model.block, "confidence": model.confidence, "entropy": model.entropy,
         "accept": accept.accept, "commit_and_draft": decode.commit_and_draft,
         "threshold_commit": decode.threshold_commit}
_TINY_W = syn.model_weights(syn.SHAPES["tiny"], 0, lm_head_scale=40.0, norm_gain_std=0.1)


# ------------------------------------------------------ planted mistake -> its pins

def _fp8_exponent_floor(w):  # the row scale rounded down: the row maximum overflows 448
    amax = np.max(np.abs(np.asarray(w, np.float64)), axis=1)
    e = np.zeros(amax.shape, np.int64)
    nz = amax > 0
    e[nz] = np.floor(np.log2(amax[nz] / fp8.E4M3_MAX)).astype(np.int64)
    return e


def _fp8_round_half_away(x):  # ties away from zero instead of to the even mantissa
    x = np.asarray(x, np.float64)
    a = np.abs(x)
    _, ex = np.frexp(a)
    spacing = np.exp2(np.maximum(ex - 1, -6).astype(np.float64) - 3.0)
    return np.sign(x) * np.floor(a / spacing + 0.5) * spacing


def _fp8_round_subnormal_spacing(x):  # the subnormals spaced 2^-10 (the normal rule continued)
    x = np.asarray(x, np.float64)
    a = np.abs(x)
    _, ex = np.frexp(a)
    spacing = np.exp2(np.maximum(ex - 1, -7).astype(np.float64) - 3.0)
    return np.sign(x) * np.rint(a / spacing) * spacing


def _fp8_values_bias8():  # exponent bias 8 instead of 7
    codes = np.arange(256)
    sign = np.where(codes & 0x80, -1.0, 1.0)
    f = (codes >> 3) & 0xF
    m = (codes & 0x7).astype(np.float64)
    mag = np.where(f == 0, m * 2.0 ** -10, (1.0 + m / 8.0) * np.exp2(f.astype(np.float64) - 8.0))
    mag = np.where((f == 0xF) & (codes & 0x7 == 0x7), np.nan, mag)
    return sign * mag


def _fp8_quantise_per_tensor(w):  # one scale for the whole matrix instead of one per row
    w = np.asarray(w, np.float64)
    e_row = fp8.row_exponents(w)
    e = np.full(e_row.shape, int(e_row.max()))
    q = fp8.e4m3_round(w / np.exp2(e.astype(np.float64))[:, None])
    return fp8.e4m3_encode(q), e

CASES = [
    ("rms_norm sum not mean", model, "rms_norm", _rms_no_mean,
     [tmod.test_rms_norm_unit_rms_and_library, tmod.test_tiny_forward_matches_torch_restatement]),
    ("rms_norm eps outside sqrt", model, "rms_norm", _rms_eps_outside,
     [tmod.test_rms_norm_unit_rms_and_library]),
    ("rope wrong sign", model, "apply_rope", _rope_wrong_sign,
     [tmod.test_rope_is_complex_rotation, tmod.test_tiny_forward_matches_torch_restatement]),
    ("rope interleaved pairs", model, "apply_rope", _rope_interleaved,
     [tmod.test_rope_is_complex_rotation, tmod.test_tiny_forward_matches_torch_restatement]),
    ("rope frequency exponent", model, "rope_angles", _rope_angles_wrong_freq,
     [tmod.test_rope_is_complex_rotation, tmod.test_tiny_forward_matches_torch_restatement]),
    ("attention causal", model, "attention", _attention_variant(causal=True),
     [tmod.test_attention_matches_library_non_causal_gqa, tmod.test_attention_special_cases,
      tmod.test_forward_is_bidirectional]),
    ("attention unscaled", model, "attention", _attention_variant(scale=False),
     [tmod.test_attention_matches_library_non_causal_gqa]),
    ("attention GQA head map", model, "attention", _attention_variant(gqa_mod=True),
     [tmod.test_attention_matches_library_non_causal_gqa, tmod.test_gqa_forward_matches_torch_restatement]),
    ("attention softmax over queries", model, "attention", _attention_variant(softmax_axis=0),
     [tmod.test_attention_matches_library_non_causal_gqa]),
    ("silu as sigmoid", model, "silu", _silu_sigmoid,
     [tmod.test_silu_matches_library, tmod.test_tiny_forward_matches_torch_restatement]),
    ("block drops the MLP residual", model, "block", _block_without_mlp_residual,
     [tmod.test_tiny_forward_matches_torch_restatement]),
    ("block swaps gate and up", model, "block", _block_gate_up_swapped,
     [tmod.test_tiny_forward_matches_torch_restatement]),
    ("p2 includes the top-1", model, "confidence", _confidence_p2_includes_top,
     [tmod.test_confidence_matches_library_softmax]),
    ("argmax ties to the highest id", model, "confidence", _confidence_last_argmax,
     [tmod.test_confidence_tie_gives_equal_top2]),
    ("entropy in bits", model, "entropy", _entropy_log2,
     [lambda: tent.test_entropy_uniform_is_log_v(8), tent.test_entropy_matches_scipy_on_random_rows]),
    (">= instead of >", decode, "exceeds", _exceeds_ge,
     [tdec.test_window_length_equals_first_failure_brute_force]),
    ("drafts from p + K", decode, "commit_and_draft", _commit_drafts_from_p_plus_k,
     [lambda: tdec.test_golden_scripted_trajectories(ROOT_GOLDEN)]),
    ("remask one late", decode, "remask", _remask_shifted,
     [tdec.test_remask_sets_exactly_the_clipped_window, lambda: tdec.test_golden_scripted_trajectories(ROOT_GOLDEN)]),
    ("entropy bound without the max", decode, "jpde_bound", _jpde_sum_only,
     [tent.test_jpde_bound_special_cases]),
    ("cache: RoPE at the row index", model, "forward_rows", _forward_rows_rope_at_row_index,
     [lambda: tcache.test_suffix_with_fresh_store_equals_full_forward(_TINY_W, tcache.N + 32)]),
    ("cache: fresh keys not stored", model, "block_rows", _block_rows_no_store,
     [lambda: tcache.test_all_rows_equal_full_forward(_TINY_W, False)]),
    ("acceptance window from position 0", accept, "accept", _accept_window_from_zero,
     [tacc.test_accept_matches_brute_force]),
    ("forward without the final RMSNorm", model, "forward_hidden", _forward_without_final_norm,
     [tmod.test_tiny_forward_matches_torch_restatement, tmod.test_gqa_forward_matches_torch_restatement]),
    ("entropy confidence exp(+H)", decode, "entropy_confidence", _entropy_confidence_wrong_sign,
     [tent.test_entropy_shift_invariance_bounds_and_order, tdec.test_decision_confidence_modes]),
    ("contiguous drafts ignored", decode, "commit_and_draft", _commit_drafts_ignore_chain,
     [lambda: tdec.test_golden_scripted_trajectories(ROOT_GOLDEN),
      lambda: tdec.test_golden_after_states_step_by_step(ROOT_GOLDEN)]),
    ("threshold rule: forced commit leftmost", decode, "threshold_commit", _threshold_forced_leftmost,
     [lambda: tthr.test_golden_threshold_trajectories(ROOT_GOLDEN)]),
    ("threshold rule: ties to the higher position", decode, "threshold_commit", _threshold_ties_high,
     [lambda: tthr.test_golden_threshold_trajectories(ROOT_GOLDEN)]),
    ("threshold rule: block ignored", decode, "threshold_commit", _threshold_whole_sequence,
     [lambda: tthr.test_golden_threshold_trajectories(ROOT_GOLDEN)]),
    ("threshold rule: committed flags ignored", decode, "threshold_commit", _threshold_recommits,
     [lambda: tthr.test_golden_threshold_trajectories(ROOT_GOLDEN)]),
    ("dual cache: suffix computed to the end", decode, "computed_range", _dual_range_to_the_end,
     [lambda: tcache.test_dual_steps_between_refreshes_stay_in_the_block(_TINY_W, 10, 0.7, 16)]),
    ("dual cache: K not capped at the block end", decode, "commit_and_draft", _commit_uncapped,
     [lambda: tcache.test_dual_cap_binds_where_the_window_runs_past_the_block(_TINY_W),
      lambda: tcache.test_dual_steps_between_refreshes_stay_in_the_block(_TINY_W, 16, 0.7, 8)]),
    ("fp8: row scale rounded down", fp8, "row_exponents", _fp8_exponent_floor,
     [tfp8.test_row_scale_is_the_least_power_of_two]),
    ("fp8: ties away from zero", fp8, "e4m3_round", _fp8_round_half_away,
     [tfp8.test_rounding_matches_the_library, tfp8.test_rounding_is_the_nearest_value_brute_force]),
    ("fp8: subnormal spacing 2^-10", fp8, "e4m3_round", _fp8_round_subnormal_spacing,
     [tfp8.test_rounding_matches_the_library, tfp8.test_rounding_is_the_nearest_value_brute_force]),
    ("fp8: exponent bias 8", fp8, "e4m3_values", _fp8_values_bias8,
     [tfp8.test_code_table_matches_the_library, tfp8.test_code_table_closed_forms]),
    ("fp8: one scale per tensor", fp8, "quantise", _fp8_quantise_per_tensor,
     [tfp8.test_quantisation_error_representability_and_idempotence]),
    ("prefix end not block-aligned", decode, "prefix_end", _prefix_end_unaligned,
     [tdec.test_prefix_end_is_the_start_of_the_current_block,
      lambda: tcache.test_refresh_exactly_at_block_changes(_TINY_W)]),
]


@pytest.mark.parametrize("name,mod,attr,bad,pins", CASES, ids=[c[0] for c in CASES])
def test_planted_mistake_fails_its_pins(monkeypatch, name, mod, attr, bad, pins):
    monkeypatch.setattr(mod, attr, bad)
    for pin in pins:
        with pytest.raises(AssertionError):
            pin()


@pytest.mark.parametrize("name,mod,attr,bad,pins", CASES, ids=[c[0] for c in CASES])
def test_pins_pass_on_the_oracle_as_written(name, mod, attr, bad, pins):
    """The same pins pass without the planted mistake (so the failures above are caused by it)."""
    for pin in pins:
        pin()
