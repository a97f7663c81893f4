"""Pins of the FP8 weight oracle (oracle/fp8.py) against what fixes it independently:
the library's float8_e4m3fn type (code table and rounding), brute force over the 254
finite values, the format's closed forms, and the definition of the row scale."""
import os
import sys

import numpy as np
import pytest
import torch

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import synthetic as syn  # noqa: E402
from oracle import fp8  # noqa: E402


def _torch_table():
    return torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).double().numpy()


def _finite_positive():
    v = fp8.e4m3_values()[:127]  # codes 0x00..0x7E
    return v


def _inputs(seed, n=20000):
    """Log-uniform magnitudes over the normal and subnormal ranges, both signs, and every
    midpoint between neighbouring values (the ties), with their negatives."""
    rng = np.random.default_rng(seed)
    mag = np.exp2(rng.uniform(-12, np.log2(448), n))
    x = np.where(rng.random(n) < 0.5, -mag, mag)
    v = _finite_positive()
    mids = (v[:-1] + v[1:]) / 2
    return np.concatenate([x, mids, -mids, v, -v, [0.0, 448.0, -448.0]])


def test_code_table_matches_the_library():
    assert np.array_equal(fp8.e4m3_values(), _torch_table(), equal_nan=True)


def test_code_table_closed_forms():
    v = fp8.e4m3_values()
    assert v[0x7E] == 448.0 and np.isnan(v[0x7F]) and np.isnan(v[0xFF])
    assert v[0x01] == 2.0 ** -9 and v[0x07] == 7 * 2.0 ** -9 and v[0x08] == 2.0 ** -6
    assert v[0x38] == 1.0 and v[0x39] == 1.125  # exponent field 7 = 2^0, mantissa steps of 1/8
    pos = v[:0x7F]
    assert np.all(np.diff(pos) > 0)  # codes 0x00..0x7E in increasing order
    assert np.array_equal(v[0x80:0xFF], -pos)  # the sign bit mirrors them
    assert np.count_nonzero(np.isfinite(v)) == 254


def test_rounding_matches_the_library():
    x = _inputs(1)
    assert np.array_equal(fp8.e4m3_round(x), torch.from_numpy(x).to(torch.float8_e4m3fn).double().numpy())


def test_rounding_is_the_nearest_value_brute_force():
    """argmin |x - v| over the finite values; at a tie the value whose code has an even
    mantissa (the last code bit clear)."""
    x = _inputs(2, 3000)
    v = fp8.e4m3_values()
    codes = np.flatnonzero(np.isfinite(v) & ~((v == 0) & (np.arange(256) >= 0x80)))  # one zero
    d = np.abs(x[:, None] - v[codes][None, :])
    best = d.min(axis=1, keepdims=True)
    ties = d == best
    pick = np.where(ties.sum(axis=1) > 1,
                    np.argmax(ties & ((codes[None, :] & 1) == 0), axis=1),
                    np.argmax(ties, axis=1))
    assert np.array_equal(fp8.e4m3_round(x), v[codes][pick])


def test_rounding_refuses_out_of_range():
    for bad in (448.5, -1e4, np.inf, np.nan):
        with pytest.raises(ValueError):
            fp8.e4m3_round(np.array([bad]))


def test_encode_decode_round_trip():
    v = fp8.e4m3_values()
    codes = np.flatnonzero(np.isfinite(v))
    assert np.array_equal(fp8.e4m3_encode(v[codes]), codes.astype(np.uint8))
    x = _inputs(3)
    r = fp8.e4m3_round(x)
    x = np.concatenate([x, [-0.0, -2.0 ** -11, 2.0 ** -11]])  # signed zeros, and values rounding to them
    r = fp8.e4m3_round(x)
    lib = torch.from_numpy(x).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(fp8.e4m3_encode(r), lib)
    assert np.array_equal(fp8.e4m3_decode(fp8.e4m3_encode(r)), r)
    for bad in (1.0 + 2.0 ** -4, 480.0, 2.0 ** -10):
        with pytest.raises(ValueError):
            fp8.e4m3_encode(np.array([bad]))


def _weights(seed):
    """A weight-like matrix: N(0, 0.02) rows, rows scaled by powers of two, a row with one
    large outlier, a row of zeros and rows whose maximum sits exactly on (or just past) a
    power-of-two multiple of 448."""
    rng = np.random.default_rng(seed)
    w = rng.normal(0, 0.02, (24, 64))
    w[3] *= 2.0 ** 9
    w[4] *= 2.0 ** -9
    w[5, 7] = 3.7
    w[6] = 0.0
    w[7] = np.clip(w[7], -0.1, 0.1)
    w[7, 0] = 448.0 * 2.0 ** -12
    w[8, 1] = -448.0 * 2.0 ** -12 * (1 + 2.0 ** -40)
    return w


def test_row_scale_is_the_least_power_of_two():
    w = _weights(4)
    e = fp8.row_exponents(w)
    amax = np.abs(w).max(axis=1)
    nz = amax > 0
    assert np.all(amax[nz] <= 448.0 * np.exp2(e[nz].astype(float)))
    assert np.all(amax[nz] > 448.0 * np.exp2(e[nz].astype(float) - 1))
    assert e[6] == 0 and e[7] == -12 and e[8] == -11


def test_quantisation_error_representability_and_idempotence():
    w = _weights(5)
    codes, e = fp8.quantise(w)
    w_hat = fp8.dequantise(codes, e)
    scale = np.exp2(e.astype(float))[:, None]
    normal = np.abs(w) / scale >= 2.0 ** -6
    err = np.abs(w_hat - w)
    assert np.all(err[normal] <= 2.0 ** -4 * np.abs(w[normal]))          # half a spacing: 2^-4 relative
    assert np.all(err[~normal] <= (2.0 ** -10 * np.broadcast_to(scale, w.shape))[~normal])  # half of 2^-9
    q_max = np.abs(fp8.e4m3_decode(codes)).max(axis=1)
    nz = q_max > 0
    # each row's maximum lands in (224, 448] before rounding, [224, 448] after it
    assert np.all((q_max[nz] >= 224) & (q_max[nz] <= 448))
    as_bf16 = torch.from_numpy(w_hat.astype(np.float32)).to(torch.bfloat16).double().numpy()
    assert np.array_equal(as_bf16, w_hat)                                  # exact in bf16
    # W_hat is a fixed point (a row whose maximum rounded to 224 * 2^e is stored again one
    # scale lower, with the same values)
    assert np.array_equal(fp8.dequantise(*fp8.quantise(w_hat)), w_hat)


def test_weights_fp8_quantises_the_matrices_only():
    sh = syn.SHAPES["tiny"]
    w = syn.model_weights(sh, 0, lm_head_scale=40.0, norm_gain_std=0.1)
    q = fp8.weights_fp8(w)
    assert q["embed"] is w["embed"] and q["final_norm"] is w["final_norm"]
    for lw, lq in zip(w["layers"], q["layers"]):
        assert lq["attn_norm"] is lw["attn_norm"] and lq["mlp_norm"] is lw["mlp_norm"]
        for k in fp8.QUANTISED:  # (the error bound is pinned above; here: which tensors)
            a, b = np.asarray(lw[k], np.float64), lq[k].astype(np.float64)
            assert b.shape == a.shape and not np.array_equal(a, b)
            assert np.array_equal(b, fp8.dequantise(*fp8.quantise(a)))
    assert np.array_equal(q["lm_head"], fp8.dequantise(*fp8.quantise(w["lm_head"])))
    assert not np.array_equal(q["lm_head"], w["lm_head"])
