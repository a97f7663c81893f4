"""Oracle: FP8 (E4M3) weight storage with one power-of-two scale per output row, fp64.

Test infrastructure only (see ``oracle/__init__.py``).

Not in the paper.  A serving refinement for the steps that stream every weight once for
few rows (the cached suffix steps of the decoder): storing the linear weights in 8 bits
halves the bytes those steps must read.  This module fixes what the stored weights mean;
the forward is then the model's forward with each quantised matrix W replaced by its
dequantised value W_hat (``oracle.model`` unchanged).

The format (the readings this module takes):

* E4M3 as in the OCP 8-bit floating-point specification ("E4M3FN"): a sign bit, four
  exponent bits with bias 7, three mantissa bits.  Exponent field 0 holds zero and the
  subnormals m * 2^-9 (m = 1..7); field f = 1..15 the normals (1 + m/8) * 2^(f-7); there
  are no infinities, and the code with every exponent and mantissa bit set is NaN, so
  the largest finite magnitude is 1.75 * 2^8 = 448.
* Rounding to the nearest representable value, ties to the even mantissa, the sign of
  the operand kept (a negative value that rounds to zero gives -0): IEEE 754's default
  rounding.
* One scale per output feature, i.e. per row n of a weight in the [out][in] layout:
  2^e_n with e_n the least integer for which max_k |W[n,k]| / 2^e_n <= 448.  A power of
  two costs a floating-point format almost nothing (the relative spacing of E4M3 values
  does not depend on where the row maximum lands in [224, 448]), and it keeps
  W_hat = q * 2^e_n exactly representable in bf16 (q has at most 4 significant bits, bf16
  8; the lowest bit of any W_hat in row n is at least 2^(e_n - 9), bf16's least
  subnormal 2^-133, so this holds whenever e_n >= -124, i.e. for every row whose largest
  magnitude exceeds 2^-116), so a kernel can widen the bytes to bf16 and run the
  unchanged bf16 contraction.  A row of zeros takes e_n = 0.
* Which weights: the seven matrices of every block (q, k, v, o, gate, up, down) and the
  LM head.  The embedding is a gather of the rows in use, and the norm gains are a few
  KB, so both stay bf16.
"""
from __future__ import annotations

import numpy as np

E4M3_MAX = 448.0
E4M3_MIN_NORMAL = 2.0 ** -6
E4M3_MIN_SUBNORMAL = 2.0 ** -9
QUANTISED = ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")


def e4m3_values() -> np.ndarray:
    """The value of each of the 256 codes (sign bit 7, exponent bits 6..3, mantissa bits
    2..0), NaN for the two NaN codes."""
    codes = np.arange(256)
    sign = np.where(codes & 0x80, -1.0, 1.0)
    f = (codes >> 3) & 0xF
    m = (codes & 0x7).astype(np.float64)
    mag = np.where(f == 0, m * E4M3_MIN_SUBNORMAL, (1.0 + m / 8.0) * np.exp2(f.astype(np.float64) - 7.0))
    mag = np.where((f == 0xF) & (codes & 0x7 == 0x7), np.nan, mag)
    return sign * mag


def e4m3_decode(codes: np.ndarray) -> np.ndarray:
    """Values (float64) of uint8 codes."""
    return e4m3_values()[np.asarray(codes, dtype=np.uint8)]


def e4m3_round(x: np.ndarray) -> np.ndarray:
    """The nearest E4M3 value to each x (ties to the even mantissa), |x| <= 448 required.

    The spacing of E4M3 values near |x| is 2^(E-3) for |x| in [2^E, 2^(E+1)), E >= -6, and
    the subnormal spacing 2^-9 below 2^-6; |x| divided by that spacing is exact in fp64,
    and numpy's rint rounds half to even."""
    x = np.asarray(x, dtype=np.float64)
    a = np.abs(x)
    if np.any(~np.isfinite(a)) or np.any(a > E4M3_MAX):
        raise ValueError("e4m3_round: |x| must be finite and at most 448")
    _, ex = np.frexp(a)  # a = frac * 2^ex, frac in [0.5, 1): the binade's exponent is ex - 1
    spacing = np.exp2(np.maximum(ex - 1, -6).astype(np.float64) - 3.0)
    return np.copysign(np.rint(a / spacing) * spacing, x)  # (the sign kept, zeros included)


def e4m3_encode(v: np.ndarray) -> np.ndarray:
    """Codes (uint8) of values that are E4M3 values (e.g. the output of e4m3_round)."""
    v = np.asarray(v, dtype=np.float64)
    a = np.abs(v)
    sign = np.where(np.signbit(v), 0x80, 0)
    _, ex = np.frexp(a)
    normal = a >= E4M3_MIN_NORMAL
    f = np.where(normal, ex - 1 + 7, 0)
    m = np.where(normal, a / np.exp2((ex - 1).astype(np.float64)) * 8.0 - 8.0, a / E4M3_MIN_SUBNORMAL)
    if np.any(m != np.rint(m)) or np.any(m < 0) or np.any(m > 7) or np.any(f > 15) or np.any((f == 15) & (m == 7)):
        raise ValueError("e4m3_encode: not an E4M3 value")
    return (sign | (f << 3) | m.astype(np.int64)).astype(np.uint8)


def row_exponents(w: np.ndarray) -> np.ndarray:
    """e_n = the least integer with max_k |w[n,k]| <= 448 * 2^e_n (0 for a row of zeros)."""
    amax = np.max(np.abs(np.asarray(w, dtype=np.float64)), axis=1)
    e = np.zeros(amax.shape, dtype=np.int64)
    nz = amax > 0
    e[nz] = np.ceil(np.log2(amax[nz] / E4M3_MAX)).astype(np.int64)
    # log2 is not exact: step to the least integer by the defining comparison
    for n in np.flatnonzero(nz):
        while amax[n] > E4M3_MAX * 2.0 ** e[n]:
            e[n] += 1
        while amax[n] <= E4M3_MAX * 2.0 ** (e[n] - 1):
            e[n] -= 1
    return e


def quantise(w: np.ndarray):
    """(codes uint8 [N][K], exponents int64 [N]) of a weight [N][K]: each row divided by
    its scale 2^e_n (exact) and rounded to E4M3."""
    w = np.asarray(w, dtype=np.float64)
    e = row_exponents(w)
    q = e4m3_round(w / np.exp2(e.astype(np.float64))[:, None])
    return e4m3_encode(q), e


def dequantise(codes: np.ndarray, e: np.ndarray) -> np.ndarray:
    """W_hat[n,k] = value(codes[n,k]) * 2^e_n (float64)."""
    return e4m3_decode(codes) * np.exp2(np.asarray(e, dtype=np.float64))[:, None]


def weights_fp8(w: dict) -> dict:
    """The weights dict of ``synthetic.model_weights`` with every quantised matrix replaced
    by W_hat (float32, exact): the model the FP8 weights store."""
    def q(a):
        return dequantise(*quantise(a)).astype(np.float32)
    out = dict(w)
    out["lm_head"] = q(w["lm_head"])
    out["layers"] = [{k: (q(v) if k in QUANTISED else v) for k, v in lw.items()} for lw in w["layers"]]
    return out
