"""Per-kernel parity of the CUDA path (through the C ABI) against the CPU oracle.

Tolerances follow from the arithmetic: GEMM/attention outputs are rounded to bf16
(relative 2^-9) after fp32 accumulation; confidences must agree within 1e-3 absolute
and top-1 ids wherever the oracle's top-1/top-2 gap exceeds that tolerance.
"""
import numpy as np
import pytest
import torch

import paper_2607_20467_gb300 as dcl
import synthetic as syn
from oracle import model

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ops():
    import __graft_entry__
    __graft_entry__.build()
    ctx = dcl.Context(None, 1, 1)
    yield ctx
    ctx.close()


def _bf16(a):
    return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(torch.bfloat16).cuda()


def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


# ------------------------------------------------------------------ generator
@pytest.mark.parametrize("tid,start,count,std,mean", [
    (syn.tensor_id(syn.TensorKind.WQ, 0), 0, 100_003, 0.02, 0.0),
    (syn.tensor_id(syn.TensorKind.LM_HEAD, 0), 12_345, 65_536, 0.8, 0.0),
    (syn.tensor_id(syn.TensorKind.ATTN_NORM, 5), 0, 4096, 0.1, 1.0),
    (syn.tensor_id(syn.TensorKind.W_UP, 31), 2 ** 31 + 7, 5000, 0.02, 0.0),
])
def test_generator_bit_exact(ops, tid, start, count, std, mean):
    dst = torch.empty(count, dtype=torch.bfloat16, device="cuda")
    ops.op_generate(dst, 1, tid, start, count, std, mean)
    torch.cuda.synchronize()
    ref = syn.weight_values(1, tid, start, count, std, mean)
    assert (dst.float().cpu().numpy() == ref).all()


# ------------------------------------------------------------------ RMSNorm
@pytest.mark.parametrize("rows,d", [(1, 256), (96, 256), (7, 4096), (3, 3584), (33, 128)])
def test_rmsnorm(ops, rows, d):
    rng = np.random.default_rng(rows * d)
    x = (rng.normal(0, 3, (rows, d))).astype(np.float32)
    g = syn.round_bf16(rng.normal(1, 0.2, d).astype(np.float32))
    y = torch.empty(rows, d, dtype=torch.bfloat16, device="cuda")
    ops.op_rmsnorm(torch.from_numpy(x).cuda(), _bf16(g), y, 1e-5)
    torch.cuda.synchronize()
    ref = model.rms_norm(x, g, 1e-5)
    err = np.abs(_f64(y) - ref)
    assert (err <= 2 ** -8 * np.abs(ref) + 1e-6).all()


# ------------------------------------------------------------------ tcgen05 GEMM
PAIR, SK, HALF, DS = 2, 1 << 16, 1 << 18, 1 << 19
# auto, one-CTA 128 / 256 columns, CTA pair (library's K schedule), CTA pair unsplit,
# CTA pair with 2 / 3 K splits, CTA pair with stream-K over all pairs / in K halves,
# left-over tiles as two half-width pieces, left-over tiles split by K over a cluster's
# two pairs (DSMEM sum)
TILES = [0, 128, 256, PAIR, PAIR | (1 << 8), PAIR | (2 << 8), PAIR | (3 << 8), PAIR | SK, PAIR | SK | (2 << 8),
         PAIR | HALF, PAIR | DS]


def _splits(tile):
    if (tile & 0xff) != PAIR or tile & SK:
        return 1
    return max(1, (tile >> 8) & 0xff)


def _streamk_possible(M, N, K, segments):
    """Stream-K needs a partly filled last round of pair tiles and at least one 64-wide
    K block for every sharing CTA pair."""
    pairs = torch.cuda.get_device_properties(0).multi_processor_count // 2
    left = ((M + 255) // 256) * ((N + 255) // 256) % pairs
    sharing = pairs if segments == 0 else min(pairs, segments * left)
    return segments != 1 and left > 0 and left * (K // 64) >= sharing


def _unsupported(M, N, K, tile):
    """True when the tile choice cannot run this shape (then the call must be refused)."""
    if tile & DS:  # (and at most one left-over tile per cluster: every shape here has <= 32)
        return K // 64 < 2
    if tile & SK:
        return not _streamk_possible(M, N, K, (tile >> 8) & 0xff)
    return K // 64 < _splits(tile)


@pytest.mark.parametrize("tile", TILES)
@pytest.mark.parametrize("M,N,K", [(96, 768, 256), (128, 256, 64), (300, 512, 1024), (1, 128, 64),
                                   (257, 384, 192), (512, 4096, 4096), (200, 1024, 12288),
                                   (300, 1280, 4096)])
def test_linear_bf16(ops, M, N, K, tile):
    rng = np.random.default_rng(M + N + K)
    a = syn.round_bf16(rng.normal(0, 1, (M, K)).astype(np.float32))
    w = syn.round_bf16(rng.normal(0, K ** -0.5, (N, K)).astype(np.float32))
    out = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    if _unsupported(M, N, K, tile):
        with pytest.raises(dcl.DcleapError):
            ops.op_linear(_bf16(a), _bf16(w), out, mode=0, tile=tile)
        return
    ops.op_linear(_bf16(a), _bf16(w), out, mode=0, tile=tile)
    torch.cuda.synchronize()
    ref = a.astype(np.float64) @ w.astype(np.float64).T
    got = _f64(out)
    assert np.isfinite(got).all()
    err = np.abs(got - ref)
    assert (err <= 2 ** -8 * np.abs(ref) + 1e-3 * np.sqrt((ref ** 2).mean())).all()


@pytest.mark.parametrize("tile", TILES)
@pytest.mark.parametrize("M,N,K", [(96, 256, 256), (512, 4096, 4096), (70, 3584, 3584), (300, 1280, 4096)])
def test_linear_residual(ops, M, N, K, tile):
    rng = np.random.default_rng(7 * M + N)
    a = syn.round_bf16(rng.normal(0, 1, (M, K)).astype(np.float32))
    w = syn.round_bf16(rng.normal(0, K ** -0.5, (N, K)).astype(np.float32))
    h0 = rng.normal(0, 2, (M, N)).astype(np.float32)
    h = torch.from_numpy(h0).cuda()
    if _unsupported(M, N, K, tile):
        with pytest.raises(dcl.DcleapError):
            ops.op_linear(_bf16(a), _bf16(w), h, mode=1, tile=tile)
        return
    ops.op_linear(_bf16(a), _bf16(w), h, mode=1, tile=tile)
    torch.cuda.synchronize()
    ref = h0.astype(np.float64) + a.astype(np.float64) @ w.astype(np.float64).T
    assert np.abs(h.cpu().numpy() - ref).max() <= 1e-4 * np.sqrt((ref ** 2).mean()) * 10


@pytest.mark.parametrize("tile,mode", [(PAIR | (3 << 8), 1), (PAIR | (2 << 8), 0), (0, 1), (0, 0),
                                       (PAIR | SK, 0), (PAIR | SK, 1), (PAIR | SK | (2 << 8), 1),
                                       (PAIR | DS, 1), (PAIR | DS, 0)])
def test_linear_split_k_is_deterministic(ops, tile, mode):
    """Split-K and stream-K partial sums are combined in K order: two runs give the same
    bits."""
    rng = np.random.default_rng(5)
    M, N, K = 512, 4096, 12288
    a = _bf16(rng.normal(0, 1, (M, K)).astype(np.float32))
    w = _bf16(rng.normal(0, K ** -0.5, (N, K)).astype(np.float32))
    outs = []
    for _ in range(2):
        if mode == 1:
            o = torch.ones(M, N, device="cuda")
        else:
            o = torch.zeros(M, N, dtype=torch.bfloat16, device="cuda")
        ops.op_linear(a, w, o, mode=mode, tile=tile)
        outs.append(o)
    torch.cuda.synchronize()
    assert torch.equal(outs[0], outs[1])


@pytest.mark.parametrize("M,N,K,mode", [(512, 12288, 4096, 0), (512, 4096, 4096, 1), (300, 1280, 4096, 0),
                                        (512, 4096, 12288, 1), (1, 128, 64, 0)])
def test_linear_half_pieces_equal_whole_tiles(ops, M, N, K, mode):
    """Half-width pieces accumulate each output over all of K in the same order as whole
    tiles: the same bits (whole tiles forced by an unsplit pair tile), run after run."""
    rng = np.random.default_rng(M + 3 * N + K)
    a = _bf16(rng.normal(0, 1, (M, K)).astype(np.float32))
    w = _bf16(rng.normal(0, K ** -0.5, (N, K)).astype(np.float32))
    h0 = torch.from_numpy(rng.normal(0, 2, (M, N)).astype(np.float32)).cuda()
    outs = []
    for tile in (PAIR | (1 << 8), PAIR | HALF, PAIR | HALF):
        o = h0.clone() if mode == 1 else torch.zeros(M, N, dtype=torch.bfloat16, device="cuda")
        ops.op_linear(a, w, o, mode=mode, tile=tile)
        outs.append(o)
    torch.cuda.synchronize()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


# ------------------------------------------------------------------ attention
@pytest.mark.parametrize("B,T,H,G,hd,qr", [(1, 96, 4, 4, 64, 0), (2, 65, 4, 2, 128, 0), (1, 1, 2, 1, 64, 0),
                                           (1, 512, 32, 32, 128, 0), (2, 200, 28, 4, 128, 0), (1, 1536, 4, 4, 128, 0),
                                           # queries = the last qr positions (the suffix of a cached step),
                                           # keys = all T positions; a ragged last key block; GQA; hd 64
                                           (1, 1536, 32, 32, 128, 32), (2, 300, 4, 2, 128, 160),
                                           (1, 1000, 28, 4, 128, 192), (1, 640, 2, 2, 64, 64)])
def test_attention_non_causal(ops, B, T, H, G, hd, qr):
    rng = np.random.default_rng(B * T * H + hd + qr)
    cols = (H + 2 * G) * hd
    qkv = syn.round_bf16(rng.normal(0, 1, (B * T, cols)).astype(np.float32))
    out = torch.full((B * T, H * hd), float("nan"), dtype=torch.bfloat16, device="cuda")
    ops.op_attention(_bf16(qkv), out, B, T, H, G, hd, qr)
    torch.cuda.synchronize()
    got = _f64(out)
    q0 = T - qr if qr else 0
    for b in range(B):
        blk = qkv[b * T:(b + 1) * T].astype(np.float64)
        q = blk[q0:, :H * hd].reshape(T - q0, H, hd)
        k = blk[:, H * hd:(H + G) * hd].reshape(T, G, hd)
        v = blk[:, (H + G) * hd:].reshape(T, G, hd)
        ref = model.attention(q, k, v)
        g = got[b * T + q0:(b + 1) * T]
        if q0:
            assert np.isnan(got[b * T:b * T + q0]).all()  # rows outside the query set untouched
        assert np.isfinite(g).all()
        assert np.abs(g - ref).max() <= 1.5e-2 * np.abs(ref).max() + 1e-3
        assert np.abs(g - ref).mean() <= 3e-3 * np.sqrt((ref ** 2).mean())


# ------------------------------------------------------------------ LM head + confidence
@pytest.mark.parametrize("tile", [0, 256, PAIR, PAIR | SK, PAIR | SK | (2 << 8)])
@pytest.mark.parametrize("R,V,d,sz", [(37, 4096, 256, 12.0), (5, 1000, 128, 6.0), (130, 4096, 64, 20.0),
                                      (300, 4096, 256, 12.0), (64, 126464, 4096, 15.0),
                                      (300, 126464, 4096, 15.0)])
def test_lmhead_top2(ops, R, V, d, sz, tile):
    rng = np.random.default_rng(R * V + d)
    x = syn.round_bf16(rng.normal(0, 1, (R, d)).astype(np.float32))
    w = syn.round_bf16(rng.normal(0, sz / np.sqrt(d), (V, d)).astype(np.float32))
    tie = None
    if R > 8:  # plant an exact tie: row 3's top column duplicated at another index
        z3 = x[3].astype(np.float64) @ w.astype(np.float64).T
        j = int(np.argmax(z3))
        w[(j + 17) % V] = w[j]
        tie = min(j, (j + 17) % V)
    top1 = torch.zeros(R, dtype=torch.int32, device="cuda")
    p1 = torch.zeros(R, dtype=torch.float32, device="cuda")
    p2 = torch.zeros(R, dtype=torch.float32, device="cuda")
    ent = torch.full((R,), -1.0, dtype=torch.float32, device="cuda")
    if _unsupported(R, V, d, tile):
        with pytest.raises(dcl.DcleapError):
            ops.op_lmhead_top2(_bf16(x), _bf16(w), top1, p1, p2, tile=tile)
        return
    ops.op_lmhead_top2(_bf16(x), _bf16(w), top1, p1, p2, tile=tile, entropy=ent)
    torch.cuda.synchronize()
    rows = np.arange(R) if R <= 64 else rng.choice(R, 32, replace=False)
    z = x[rows].astype(np.float64) @ w.astype(np.float64).T
    ids_o, p1_o, p2_o = model.confidence(z)
    g1, gp1, gp2 = top1.cpu().numpy()[rows], p1.cpu().numpy()[rows], p2.cpu().numpy()[rows]
    assert np.abs(gp1 - p1_o).max() <= 1e-3
    assert np.abs(gp2 - p2_o).max() <= 1e-3
    # marginal entropy: |dH| <= 2 H max|dz| for a logit error dz (|dH/dz_v| = P(v)|ln P(v) + H|);
    # fp32 accumulation of d bf16 products leaves |dz| ~1e-4 at these scales
    H_o = model.entropy(z)
    gH = ent.cpu().numpy()[rows]
    assert (gH >= 0).all() and (gH <= np.log(V) + 1e-4).all()
    assert np.abs(gH - H_o).max() <= 5e-3, float(np.abs(gH - H_o).max())
    assert (np.exp(-gH) <= gp1 + 2e-3).all()
    sure = (p1_o - p2_o) > 1e-3
    assert (g1[sure] == ids_o[sure]).all()
    assert ((g1 >= 0) & (g1 < V)).all()
    if tie is not None:  # ties go to the lowest index and give p2 == p1
        assert int(top1[3]) == tie
        assert abs(float(p1[3]) - float(p2[3])) <= 1e-6
