"""Seeded synthetic inputs shared by the CPU oracle and the CUDA path.

This module holds random draws, bf16 packing and workload shapes only; none of
the decoding method's arithmetic lives here.  Both sides of every parity test
take their inputs from it:

* ``weight_values`` is the counter-based weight generator.  It is defined from
  the published SplitMix64 output function (Steele, Lea and Flood, "Fast
  splittable pseudorandom number generators", OOPSLA 2014) and a sum of four
  16-bit uniforms (an Irwin-Hall approximation of a normal draw), so that it can
  be evaluated exactly, element by element, in integer arithmetic plus one
  IEEE fp32 multiply and one fp32 add.  The CUDA library carries its own
  implementation of the same definition (``dcl_init_random_weights``) so that
  multi-GB weights never cross the host link; a GPU test checks the two agree
  bit for bit.
* ``prompt_ids`` and ``accept_inputs`` draw prompts and acceptance-kernel
  inputs with numpy's PCG64 generator.
"""
from __future__ import annotations

import concurrent.futures as cf
import dataclasses
import math
import os

import numpy as np

__all__ = [
    "ModelShape", "SHAPES", "TensorKind", "tensor_id", "splitmix64",
    "weight_values", "embed_rows", "bf16_bits", "bf16_to_f32", "round_bf16",
    "model_weights", "prompt_ids", "accept_inputs", "GEN_SIGMA4",
]

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)

# standard deviation of the sum of four independent uniform draws on {0..65535}
GEN_SIGMA4 = math.sqrt(4.0 * (65536.0 ** 2 - 1.0) / 12.0)
GEN_MEAN4 = 2 * 65535  # mean of that sum


@dataclasses.dataclass(frozen=True)
class ModelShape:
    """Transformer shape of a masked-diffusion LM (no biases, untied head)."""
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int
    vocab: int
    mask_id: int
    rope_theta: float
    rms_eps: float = 1e-5


SHAPES = {
    # 2 layers, d 256, 4x64 MHA, ffn 1024, vocab 4096 (mask 4095)
    "tiny": ModelShape(2, 256, 4, 4, 64, 1024, 4096, 4095, 10000.0),
    # LLaDA-8B-shaped: 32 layers, d 4096, 32x128 MHA, ffn 12288, vocab 126464
    "llada8b": ModelShape(32, 4096, 32, 32, 128, 12288, 126464, 126463, 500000.0),
    # the LLaDA-8B shape with 2 layers (profiling captures of the same kernels)
    "llada8b-2l": ModelShape(2, 4096, 32, 32, 128, 12288, 126464, 126463, 500000.0),
    # Dream-7B-shaped: 28 layers, d 3584, 28 query / 4 kv heads x128, ffn 18944, vocab 152064
    "dream7b": ModelShape(28, 3584, 28, 4, 128, 18944, 152064, 152063, 1000000.0),
}


class TensorKind:
    """Tensor kinds; the numbering is part of the weight generator's counter."""
    EMBED = 0        # [V][d]
    ATTN_NORM = 1    # [d]
    WQ = 2           # [H*hd][d]
    WK = 3           # [G*hd][d]
    WV = 4           # [G*hd][d]
    WO = 5           # [d][H*hd]
    MLP_NORM = 6     # [d]
    W_GATE = 7       # [F][d]
    W_UP = 8         # [F][d]
    W_DOWN = 9       # [d][F]
    FINAL_NORM = 10  # [d]
    LM_HEAD = 11     # [V][d]

    GLOBAL = (EMBED, FINAL_NORM, LM_HEAD)
    NORMS = (ATTN_NORM, MLP_NORM, FINAL_NORM)


def tensor_id(kind: int, layer: int) -> int:
    """Counter block of a tensor: 16*layer + kind; global tensors use layer 4095."""
    if kind in TensorKind.GLOBAL:
        layer = 4095
    return 16 * layer + kind


def splitmix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function (published constants), on uint64 arrays."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = z + _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def weight_values(seed: int, tid: int, start: int, count: int, std: float,
                  mean: float = 0.0) -> np.ndarray:
    """Elements [start, start+count) of tensor ``tid`` as bf16-exact float32.

    key   = seed << 48 | tid << 32 | index           (index < 2**32)
    h     = splitmix64(key)
    s     = sum of the four 16-bit fields of h         (integer in [0, 262140])
    w32   = fp32(s - 131070) * fp32(std / GEN_SIGMA4) (one IEEE fp32 multiply)
    w32   = w32 + fp32(mean)                           (one IEEE fp32 add, if mean != 0)
    value = bf16 round-to-nearest-even of w32
    """
    if not (0 <= seed < 65536 and 0 <= tid < 65536 and start >= 0 and start + count <= 2 ** 32):
        raise ValueError("generator counter out of range")
    out = np.empty(count, np.float32)
    threads = min(16, os.cpu_count() or 1)
    if count < (1 << 22) or threads == 1:
        _weight_chunks(seed, tid, start, count, std, mean, out)
    else:  # elementwise and counter-based: independent sub-ranges, numpy releases the GIL
        step = -(-count // threads)

        def job(i):
            a, b = i * step, min(count, (i + 1) * step)
            if a < b:
                _weight_chunks(seed, tid, start + a, b - a, std, mean, out[a:b])

        with cf.ThreadPoolExecutor(threads) as ex:
            list(ex.map(job, range(threads)))
    return out


def _weight_chunks(seed, tid, start, count, std, mean, out):
    """weight_values written into out (float32 [count]), in cache-sized chunks with
    in-place integer steps."""
    hi = (np.uint64(seed) << np.uint64(48)) | (np.uint64(tid) << np.uint64(32))
    std32 = float(np.float32(std))        # the C ABI receives std as a float
    scale = np.float32(std32 / GEN_SIGMA4)
    m16 = np.uint64(0xFFFF)
    chunk = 1 << 16
    for c0 in range(0, count, chunk):
        n = min(chunk, count - c0)
        z = np.arange(start + c0, start + c0 + n, dtype=np.uint64)
        z |= hi                                       # key = seed << 48 | tid << 32 | index
        t = np.empty_like(z)
        with np.errstate(over="ignore"):              # SplitMix64, as splitmix64() above
            z += _GOLDEN
            np.right_shift(z, np.uint64(30), out=t)
            z ^= t
            z *= _M1
            np.right_shift(z, np.uint64(27), out=t)
            z ^= t
            z *= _M2
            np.right_shift(z, np.uint64(31), out=t)
            z ^= t
        s = z & m16                                   # sum of the four 16-bit fields
        for sh in (16, 32):
            np.right_shift(z, np.uint64(sh), out=t)
            t &= m16
            s += t
        np.right_shift(z, np.uint64(48), out=t)
        s += t
        w = (s.view(np.int64) - GEN_MEAN4).astype(np.float32)
        w *= scale
        if mean != 0.0:
            w += np.float32(mean)
        out[c0:c0 + n] = round_bf16(w)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even (finite inputs)."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = (b + np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return rounded.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float32 values."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 value (returned as float32)."""
    return bf16_to_f32(bf16_bits(x))


def model_weights(shape: ModelShape, seed: int, std: float = 0.02,
                  lm_head_scale: float = 1.0, norm_gain_std: float = 0.0,
                  layers=None, global_tensors: bool = True, embed: bool = True) -> dict:
    """Weights of ``shape`` from the counter-based generator, as bf16-exact float32.

    Matrices are [out][in] (the nn.Linear layout).  Norm gains are 1 + N(0, norm_gain_std).
    ``layers`` restricts the per-layer tensors generated (all by default);
    ``global_tensors=False`` leaves out the embedding, final norm and LM head (None);
    ``embed=False`` leaves out only the embedding table (see embed_rows).
    """
    d, hd, H, G, F, V = (shape.d_model, shape.head_dim, shape.n_heads,
                         shape.n_kv_heads, shape.ffn_dim, shape.vocab)
    dims = {
        TensorKind.EMBED: (V, d), TensorKind.ATTN_NORM: (d,), TensorKind.WQ: (H * hd, d),
        TensorKind.WK: (G * hd, d), TensorKind.WV: (G * hd, d), TensorKind.WO: (d, H * hd),
        TensorKind.MLP_NORM: (d,), TensorKind.W_GATE: (F, d), TensorKind.W_UP: (F, d),
        TensorKind.W_DOWN: (d, F), TensorKind.FINAL_NORM: (d,), TensorKind.LM_HEAD: (V, d),
    }

    def gen(kind, layer):
        n = int(np.prod(dims[kind]))
        if kind in TensorKind.NORMS:
            v = weight_values(seed, tensor_id(kind, layer), 0, n, norm_gain_std, 1.0)
        else:
            s = np.float32(std)
            if kind == TensorKind.LM_HEAD:
                s = s * np.float32(lm_head_scale)   # fp32 product, as on the device
            v = weight_values(seed, tensor_id(kind, layer), 0, n, float(s))
        return v.reshape(dims[kind])

    names = {TensorKind.ATTN_NORM: "attn_norm", TensorKind.WQ: "wq", TensorKind.WK: "wk",
             TensorKind.WV: "wv", TensorKind.WO: "wo", TensorKind.MLP_NORM: "mlp_norm",
             TensorKind.W_GATE: "w_gate", TensorKind.W_UP: "w_up", TensorKind.W_DOWN: "w_down"}
    if global_tensors:
        out = {"embed": gen(TensorKind.EMBED, 0) if embed else None, "final_norm": gen(TensorKind.FINAL_NORM, 0),
               "lm_head": gen(TensorKind.LM_HEAD, 0), "layers": []}
    else:
        out = {"embed": None, "final_norm": None, "lm_head": None, "layers": []}
    for li in range(shape.n_layers):
        if layers is not None and li not in layers:
            out["layers"].append(None)
            continue
        out["layers"].append({names[k]: gen(k, li) for k in names})
    return out


def embed_rows(shape: ModelShape, seed: int, ids, std: float = 0.02) -> np.ndarray:
    """Rows ``ids`` of the embedding table of ``model_weights(shape, seed, std)`` (float32
    [len(ids)][d]) without generating the whole table."""
    d = shape.d_model
    tid = tensor_id(TensorKind.EMBED, 0)
    ids = np.asarray(ids, dtype=np.int64).reshape(-1)
    out = np.empty((len(ids), d), np.float32)
    for r, i in enumerate(ids):
        if not 0 <= i < shape.vocab:
            raise ValueError("token id out of range")
        out[r] = weight_values(seed, tid, int(i) * d, d, std)
    return out


def prompt_ids(seed: int, batch: int, n_prompt: int, mask_id: int) -> np.ndarray:
    """Uniform random prompt ids in [0, mask_id) (never the mask id), int32 [batch][N]."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.integers(0, mask_id, size=(batch, n_prompt), dtype=np.int64).astype(np.int32)


def decode_state(seed: int, prompt: np.ndarray, gen_len: int, p_offset: int, window: int, mask_id: int,
                 draft_frac: float = 0.4):
    """A decoding state of Algorithm 1's shape for every row of ``prompt`` (int32 [B][N]):
    x = prompt ++ committed ids on [N, p) ++ MASK on the window [p, p + window) ++ draft
    ids on about ``draft_frac`` of the future positions (MASK elsewhere), p = N + p_offset.
    Ids are uniform in [0, mask_id).  Returns (x int32 [B][N + M], p int32 [B])."""
    rng = np.random.Generator(np.random.PCG64([seed, p_offset]))
    prompt = np.atleast_2d(np.asarray(prompt, dtype=np.int32))
    B, N = prompt.shape
    T = N + gen_len
    p = N + p_offset
    x = np.full((B, T), mask_id, np.int32)
    x[:, :N] = prompt
    x[:, N:p] = rng.integers(0, mask_id, size=(B, p - N))
    lo = min(p + window, T)
    drafts = rng.random((B, T - lo)) < draft_frac
    ids = rng.integers(0, mask_id, size=(B, T - lo))
    x[:, lo:] = np.where(drafts, ids, mask_id)
    return x, np.full(B, p, np.int32)


def _beta_mixture(rng, n):
    """Top-1 target probabilities: 50% in (0.65, 0.9), 25% above 0.9, 25% below 0.65."""
    comp = rng.choice(3, size=n, p=[0.5, 0.25, 0.25])
    b = rng.beta(2.0, 2.0, size=n)
    lo = np.array([0.65, 0.90, 0.05])[comp]
    width = np.array([0.25, 0.0999, 0.60])[comp]
    return lo + width * b


def accept_inputs(seed: int, batch: int, positions: int, vocab: int, mask_id: int,
                  rows=None) -> dict:
    """Inputs of the acceptance kernel: bf16 logits [B][P][V] plus block state.

    Per position a top-1 target probability q is drawn from the Beta mixture above,
    the other logits g_v ~ N(0, 1), and the top logit (at a uniform random index) is
    set to log(q/(1-q) * sum_{v != top} exp(g_v)); all logits are then rounded to bf16.
    The realised top-1 probability differs from q by the bf16 rounding.  Each row has
    c_b ~ U{0..P} committed positions (left-aligned); uncommitted positions hold MASK
    or a random draft id with equal odds.  ``rows`` limits logits generation to the
    listed (b, i) pairs (others are zero) to keep small samples cheap.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    committed = rng.integers(0, positions + 1, size=batch).astype(np.int32)
    x = rng.integers(0, mask_id, size=(batch, positions)).astype(np.int32)
    is_mask = rng.random((batch, positions)) < 0.5
    for b in range(batch):
        for i in range(positions):
            if i >= committed[b] and is_mask[b, i]:
                x[b, i] = mask_id
    q = _beta_mixture(rng, batch * positions).reshape(batch, positions)
    top = rng.integers(0, vocab, size=(batch, positions))
    logits = np.zeros((batch, positions, vocab), dtype=np.uint16)
    for b in range(batch):
        for i in range(positions):
            if rows is not None and (b, i) not in rows:
                continue
            prng = np.random.Generator(np.random.PCG64([seed, b, i]))
            g = prng.standard_normal(vocab, dtype=np.float32)
            g[top[b, i]] = -np.inf
            rest = float(np.exp(g.astype(np.float64)).sum())
            g[top[b, i]] = math.log(q[b, i] / (1.0 - q[b, i]) * rest)
            logits[b, i] = bf16_bits(g)
    return {"logits_bf16": logits, "committed": committed, "x": x, "target_p1": q,
            "top_index": top.astype(np.int32)}
