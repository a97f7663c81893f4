"""dcl_fp8_quantise (host code in libdcleap.so, no GPU) against the FP8 oracle: the same
bf16 weights give bit-identical E4M3 codes and row exponents."""
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import synthetic as syn  # noqa: E402
from oracle import fp8  # noqa: E402


@pytest.fixture(scope="module")
def dcl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as pkg
    return pkg


def _bits(a):
    """bf16 bit patterns of float32 values that are bf16 values."""
    b = np.ascontiguousarray(a, np.float32).view(np.uint32)
    assert not np.any(b & 0xFFFF), "not bf16 values"
    return (b >> 16).astype(np.uint16)


def _values(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _same(dcl, bits):
    codes, exps = dcl.fp8_quantise(bits)
    c_o, e_o = fp8.quantise(_values(bits))
    assert np.array_equal(exps, e_o.astype(np.int32))
    assert np.array_equal(codes, c_o)


def test_model_matrices_match_the_oracle(dcl):
    w = syn.model_weights(syn.SHAPES["tiny"], 0, lm_head_scale=40.0, norm_gain_std=0.1)
    for lw in w["layers"]:
        for k in fp8.QUANTISED:
            _same(dcl, _bits(syn.round_bf16(np.asarray(lw[k], np.float32))))
    _same(dcl, _bits(syn.round_bf16(np.asarray(w["lm_head"], np.float32))))


def test_edge_rows_match_the_oracle(dcl):
    """Rows of zeros (both signs), bf16 subnormals, the largest bf16 value, maxima exactly
    at 448 * 2^k, and every tie between neighbouring E4M3 values scaled into a row."""
    v = fp8.e4m3_values()[:127]
    mids = (v[:-1] + v[1:]) / 2
    n = 1 + len(mids)  # 127 columns: a row maximum, then the 126 midpoints
    rows = [
        np.zeros(n),
        -np.zeros(n),
        np.concatenate([[448.0 * 2.0 ** -12], np.linspace(-1e-4, 1e-4, n - 1)]),
        np.concatenate([[448.0], mids]),
        np.concatenate([[-448.0 * 2.0 ** 20], -mids * 2.0 ** 20]),
        np.concatenate([[448.0 * 2.0 ** -3], mids * 2.0 ** -3]),
    ]
    bits = np.stack([_bits(syn.round_bf16(np.asarray(r, np.float32))) for r in rows])
    sub = np.zeros((2, n), np.uint16)
    sub[0, :8] = np.arange(1, 9)            # bf16 subnormals only
    sub[1, :] = 0x8001                       # the negative smallest subnormal
    big = np.full((1, n), 0x7F7F, np.uint16)  # the largest finite bf16 value
    big[0, 1::2] = 0x0001
    _same(dcl, np.concatenate([bits, sub, big]))


def test_random_bit_patterns_match_the_oracle(dcl):
    rng = np.random.default_rng(11)
    bits = rng.integers(0, 1 << 16, (64, 96), dtype=np.uint64).astype(np.uint16)
    bits[(bits & 0x7F80) == 0x7F80] &= 0xBFFF  # no infinities or NaNs (clear an exponent bit)
    _same(dcl, bits)
    # weight-like rows across twelve binades of scale
    w = rng.normal(0, 1, (48, 200)) * np.exp2(rng.integers(-30, 10, 48))[:, None]
    _same(dcl, _bits(syn.round_bf16(w.astype(np.float32))))


def test_refuses_non_finite_and_bad_arguments(dcl):
    for bad in (0x7F80, 0xFF80, 0x7FC0):  # +inf, -inf, NaN
        bits = np.zeros((2, 4), np.uint16)
        bits[1, 2] = bad
        with pytest.raises(dcl.DcleapError) as e:
            dcl.fp8_quantise(bits)
        assert e.value.status == dcl.DCL_ERR_INVALID_ARG and "row 1, column 2" in str(e.value)
    with pytest.raises(TypeError):
        dcl.fp8_quantise(np.zeros((2, 4), np.float32))
    L = dcl.lib()
    assert L.dcl_fp8_quantise(None, 1, 1, None, None) == dcl.DCL_ERR_INVALID_ARG
    z = np.zeros((1, 1), np.uint16)
    assert L.dcl_fp8_quantise(z.ctypes.data, 0, 1, z.ctypes.data, z.ctypes.data) == dcl.DCL_ERR_INVALID_ARG
