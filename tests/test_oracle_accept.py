"""Pins of the block acceptance oracle (Eq. 2 + Eq. compute_k + Eq. draft_update)."""
import math

import numpy as np

from oracle import accept, decode
import synthetic as syn


def _brute(logits, committed, x, L, tau_c, tau_d):
    """Per row: Python-loop softmax (math.exp), first-failure K, plain draft loop."""
    B, P, V = logits.shape
    x = [list(map(int, r)) for r in x]
    ks = []
    for b in range(B):
        p = int(committed[b])
        if p >= P:
            ks.append(0)
            continue
        ids, c = [], []
        for i in range(P):
            if i < p:
                ids.append(-1)
                c.append(0.0)
                continue
            row = [float(v) for v in logits[b, i]]
            m = max(row)
            ids.append(row.index(m))
            c.append(float(np.float32(1.0 / sum(math.exp(v - m) for v in row))))
        tc, td = float(np.float32(tau_c)), float(np.float32(tau_d))
        K = 0
        while K < min(L, P - p) and c[p + K] > tc:
            K += 1
        K = max(K, 1)
        for i in range(p, p + K):
            x[b][i] = ids[i]
        for i in range(p + L, P):
            if c[i] > td:
                x[b][i] = ids[i]
        ks.append(K)
    return ks, x


def test_accept_matches_brute_force():
    for seed, L in [(0, 16), (1, 32), (2, 5), (3, 1)]:
        d = syn.accept_inputs(seed, 6, 32, 300, 299)
        z = syn.bf16_to_f32(d["logits_bf16"])
        cfg = decode.DecodeConfig(tau_commit=0.7, tau_draft=0.9, max_window=L, gen_len=32)
        K, x_out, ids, p1, p2 = accept.accept(z, d["committed"], d["x"], cfg, L)
        kb, xb = _brute(z, d["committed"], d["x"], L, 0.7, 0.9)
        assert list(K) == kb
        assert x_out.tolist() == xb
        # the generator's planted top index is the argmax; realised p1 is near its target
        for b in range(6):
            for i in range(int(d["committed"][b]), 32):
                assert ids[b, i] == d["top_index"][b, i]
                assert abs(p1[b, i] - d["target_p1"][b, i]) < 0.05
                assert p2[b, i] <= p1[b, i]


def test_accept_fully_committed_row_is_noop():
    d = syn.accept_inputs(5, 4, 8, 50, 49)
    d["committed"][:] = 8
    z = syn.bf16_to_f32(d["logits_bf16"])
    cfg = decode.DecodeConfig(max_window=4, gen_len=8)
    K, x_out, *_ = accept.accept(z, d["committed"], d["x"], cfg, 4)
    assert (K == 0).all() and (x_out == d["x"]).all()
