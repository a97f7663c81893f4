"""Pins of the decoding oracle (Eq. compute_k, Eq. draft_update, Eq. remasking, Algorithm 1).

Each test checks the oracle against something other than itself: hand-derived
trajectories (tests/golden/dcv_scripted.json), brute force, invariants the paper
states in prose, and special cases that reduce to textbook decoders.
"""
import json
import os

import numpy as np
import pytest

from oracle import decode, model
import synthetic as syn


# ---------------------------------------------------------------- Eq. compute_k

def _first_failure(c, tau):
    """Brute force: the largest k such that every c[0..k) exceeds tau (float32 compare)."""
    best = 0
    for k in range(len(c) + 1):
        if all(np.float32(c[j]) > np.float32(tau) for j in range(k)):
            best = k
    return best


def test_window_length_equals_first_failure_brute_force():
    rng = np.random.default_rng(7)
    for _ in range(3000):
        L = int(rng.integers(0, 40))
        tau = float(rng.choice([0.0, 0.3, 0.7, 0.7, 0.95, 1.0]))
        c = rng.random(L)
        # plant exact ties with tau (strict > must reject them)
        c[rng.random(L) < 0.15] = tau
        assert decode.window_length(c, tau) == _first_failure(c, tau)


def test_window_length_bounds_and_closed_forms():
    rng = np.random.default_rng(1)
    for _ in range(2000):
        L = int(rng.integers(1, 64))
        c = rng.random(L) * 0.999 + 1e-6
        K = decode.window_length(c, 0.7)
        assert 0 <= K <= L                                  # 0 <= K <= L (Sec. 3.2)
        assert decode.window_length(c, 0.0) == L            # every c > 0
        assert decode.window_length(c, 1.0) == 0            # no c > 1
    assert decode.window_length([], 0.5) == 0
    # the strict inequality of Eq. compute_k: c == tau does not pass
    assert decode.window_length([0.7, 0.9], 0.7) == 0
    assert decode.window_length([0.70001, 0.7], 0.7) == 1


# ------------------------------------------------------- scripted trajectories

def _scripted(case):
    script = case["script"]
    state = {"i": 0}

    def predict(tokens):
        s = script[state["i"]]
        state["i"] += 1
        ids = np.array(s["ids"], dtype=np.int32)
        c = np.array(s["c"], dtype=np.float64)
        return ids, c, c * 0.0
    return predict


def test_golden_scripted_trajectories(golden_dir):
    with open(os.path.join(golden_dir, "dcv_scripted.json")) as f:
        cases = json.load(f)["cases"]
    for case in cases:
        cfg = decode.DecodeConfig(tau_commit=case["tau_commit"], tau_draft=case["tau_draft"],
                                  max_window=case["window"], gen_len=case["gen_len"],
                                  min_commit=case["min_commit"],
                                  contiguous_drafts=case["contiguous_drafts"])
        out = decode.generate(_scripted(case), np.array([case["prompt"]]), cfg, case["mask_id"])
        assert out["done"]
        assert [list(map(int, a[0])) for a in out["inputs"]] == case["expect_inputs"], case["name"]
        assert list(map(int, out["k"][:, 0])) == case["expect_k"], case["name"]
        assert list(map(int, out["x"][0])) == case["expect_after"][-1], case["name"]


def test_golden_after_states_step_by_step(golden_dir):
    """Replays each golden step with commit_and_draft alone (no generate loop)."""
    with open(os.path.join(golden_dir, "dcv_scripted.json")) as f:
        cases = json.load(f)["cases"]
    for case in cases:
        N = len(case["prompt"])
        cfg = decode.DecodeConfig(tau_commit=case["tau_commit"], tau_draft=case["tau_draft"],
                                  max_window=case["window"], gen_len=case["gen_len"],
                                  contiguous_drafts=case["contiguous_drafts"])
        p = N
        for step, s in enumerate(case["script"]):
            x = np.array(case["expect_inputs"][step], dtype=np.int32)
            ids = np.zeros(x.shape[0], np.int32)
            c = np.zeros(x.shape[0])
            ids[N:], c[N:] = s["ids"], s["c"]
            K = decode.commit_and_draft(x, p, ids, c, cfg, case["window"])
            assert K == case["expect_k"][step]
            assert list(map(int, x)) == case["expect_after"][step], (case["name"], step)
            p += K


# -------------------------------------------------- tiny transformer decoders

MICRO = syn.ModelShape(n_layers=1, d_model=32, n_heads=2, n_kv_heads=2, head_dim=16,
                       ffn_dim=64, vocab=64, mask_id=63, rope_theta=10000.0)


def _micro_predict(seed, shape=MICRO, lm_scale=40.0):
    w = syn.model_weights(shape, seed, lm_head_scale=lm_scale, norm_gain_std=0.1)

    def make(N):
        def predict(tokens):
            ids, p1, p2 = model.predict(shape, w, tokens)
            return ids[N:], p1[N:], p2[N:]
        return predict
    return w, make


def _run(seed, N, M, tau_c, tau_d, window, B=2, contiguous=False, shape=MICRO):
    _, make = _micro_predict(seed, shape)
    prompt = syn.prompt_ids(seed + 100, B, N, shape.mask_id)
    cfg = decode.DecodeConfig(tau_commit=tau_c, tau_draft=tau_d, max_window=window, gen_len=M,
                              contiguous_drafts=contiguous)
    return decode.generate(make(N), prompt, cfg, shape.mask_id), prompt, cfg


@pytest.mark.parametrize("seed", [0, 1, 2])
@pytest.mark.parametrize("tau_c,tau_d,window", [(0.7, 0.98, 6), (0.5, 0.8, 3), (0.9, 0.6, 12),
                                                (0.3, 0.3, 1)])
def test_run_invariants(seed, tau_c, tau_d, window):
    N, M = 4, 12
    out, prompt, cfg = _run(seed, N, M, tau_c, tau_d, window)
    T = N + M
    mask = MICRO.mask_id
    B = prompt.shape[0]
    p = np.full(B, N)
    committed = [dict() for _ in range(B)]
    for s, (xin, k) in enumerate(zip(out["inputs"], out["k"])):
        for b in range(B):
            if p[b] >= T:
                assert k[b] == 0
                continue
            # prompt never changes; committed tokens never revert (contiguous prefix [N, p))
            assert (xin[b, :N] == prompt[b]).all()
            for pos, tok in committed[b].items():
                assert xin[b, pos] == tok
            # no draft inside the window at forward time (Eq. remasking)
            assert (xin[b, p[b]:min(p[b] + window, T)] == mask).all()
            assert 1 <= k[b] <= min(window, T - p[b])
            # the committed run is the model's top-1 prediction of this step
            ids = out["preds"][s][0, b].astype(np.int64)
            c1 = out["preds"][s][1, b]
            for j in range(p[b], p[b] + k[b]):
                committed[b][j] = ids[j - N]
            # K is the longest confident prefix (or the forced single token)
            assert k[b] == max(1, decode.window_length(c1[p[b] - N:p[b] - N + min(window, T - p[b])],
                                                     tau_c))
            p[b] += k[b]
    assert out["done"] and (out["p"] == T).all()
    for b in range(B):
        for pos, tok in committed[b].items():
            assert out["x"][b, pos] == tok


@pytest.mark.parametrize("seed", [0, 3])
def test_tau_commit_one_is_one_token_per_step(seed):
    N, M = 4, 12
    out, _, _ = _run(seed, N, M, 1.0, 0.9, 6)
    assert out["n_iter"] == M
    assert (out["k"] == 1).all()


@pytest.mark.parametrize("seed", [0, 3])
def test_tau_commit_zero_fills_whole_windows(seed):
    N, M, W = 4, 12, 5
    out, _, _ = _run(seed, N, M, 0.0, 0.98, W)
    assert out["n_iter"] == -(-M // W)
    expect = [min(W, M - W * i) for i in range(out["n_iter"])]
    assert list(out["k"][:, 0]) == expect


@pytest.mark.parametrize("seed", [0, 5])
def test_tau_draft_above_one_never_drafts(seed):
    N, M, W = 4, 12, 3
    out, _, _ = _run(seed, N, M, 0.6, 1.01, W)
    p = np.full(2, N)
    for xin, k in zip(out["inputs"], out["k"]):
        for b in range(2):
            if p[b] < N + M:
                assert (xin[b, p[b]:] == MICRO.mask_id).all()
            p[b] += k[b]


@pytest.mark.parametrize("seed", [0, 1])
def test_window_one_equals_tau_commit_one(seed):
    a, _, _ = _run(seed, 4, 12, 0.7, 0.9, 1)
    b, _, _ = _run(seed, 4, 12, 1.0, 0.9, 1)
    assert (a["x"] == b["x"]).all()
    assert a["n_iter"] == b["n_iter"] == 12


@pytest.mark.parametrize("seed", [0, 2, 4])
def test_sequential_chain_special_case(seed):
    """tau_commit = 1 with no drafts is the one-token-per-forward left-to-right decoder
    of Eq. sequential_chain; this loop is written independently of the oracle's."""
    N, M = 4, 10
    w, _ = _micro_predict(seed)
    prompt = syn.prompt_ids(seed + 100, 1, N, MICRO.mask_id)[0]
    seq = np.concatenate([prompt, np.full(M, MICRO.mask_id, np.int32)])
    for t in range(N, N + M):
        z = model.logits(w, model.forward_hidden(MICRO, w, seq))
        seq[t] = int(np.argmax(z[t]))
    cfg = decode.DecodeConfig(tau_commit=1.0, tau_draft=2.0, max_window=5, gen_len=M)

    def predict(tokens):
        ids, p1, p2 = model.predict(MICRO, w, tokens)
        return ids[N:], p1[N:], p2[N:]
    out = decode.generate(predict, prompt[None], cfg, MICRO.mask_id)
    assert (out["x"][0] == seq).all()


def _brute_alg1(predict, prompt, M, mask, L, tau_c, tau_d):
    """Algorithm 1 written out directly with Python loops (no numpy decisions shared)."""
    x = list(prompt) + [mask] * M
    N, T = len(prompt), len(prompt) + M
    p = N
    ks = []
    while p < T:
        for i in range(p, min(p + L, T)):
            x[i] = mask
        ids, c, _ = predict(np.array(x, dtype=np.int32))
        c = [float(np.float32(v)) for v in c]
        tc, td = float(np.float32(tau_c)), float(np.float32(tau_d))
        K = 0
        while K < min(L, T - p) and c[p + K - N] > tc:
            K += 1
        K = max(K, 1)
        for i in range(p, p + K):
            x[i] = int(ids[i - N])
        for i in range(p + L, T):
            if c[i - N] > td:
                x[i] = int(ids[i - N])
        p += K
        ks.append(K)
    return x, ks


def test_brute_force_tiny_vocabulary():
    shape = syn.ModelShape(1, 16, 2, 2, 8, 32, 8, 7, 10000.0)
    N, M = 2, 4
    w = syn.model_weights(shape, 11, lm_head_scale=60.0, norm_gain_std=0.1)
    prompt = np.array([3, 1], dtype=np.int32)

    def predict(tokens):
        ids, p1, p2 = model.predict(shape, w, tokens)
        return ids[N:], p1[N:], p2[N:]
    for L in range(1, M + 1):
        for tau_c in (0.0, 0.2, 0.35, 0.5, 0.7, 0.9, 1.0):
            for tau_d in (0.0, 0.3, 0.6, 0.98, 1.5):
                cfg = decode.DecodeConfig(tau_commit=tau_c, tau_draft=tau_d, max_window=L, gen_len=M)
                out = decode.generate(predict, prompt[None], cfg, shape.mask_id)
                x, ks = _brute_alg1(predict, prompt, M, shape.mask_id, L, tau_c, tau_d)
                assert list(out["x"][0]) == x
                assert list(out["k"][:, 0]) == ks


def test_contiguous_drafts_subset_of_default():
    """App. E drafts are a subset of the default drafts at the same state."""
    rng = np.random.default_rng(3)
    for _ in range(500):
        T, p, L = 40, int(rng.integers(0, 30)), int(rng.integers(1, 12))
        x0 = rng.integers(0, 50, T).astype(np.int32)
        ids = rng.integers(0, 50, T).astype(np.int32)
        c = rng.random(T)
        cfg_a = decode.DecodeConfig(tau_commit=0.5, tau_draft=0.6, gen_len=T, max_window=L)
        cfg_b = decode.DecodeConfig(tau_commit=0.5, tau_draft=0.6, gen_len=T, max_window=L,
                                    contiguous_drafts=True)
        xa, xb = x0.copy(), x0.copy()
        decode.commit_and_draft(xa, p, ids, c, cfg_a, L)
        decode.commit_and_draft(xb, p, ids, c, cfg_b, L)
        changed_b = xb != x0
        assert (xa[changed_b] == xb[changed_b]).all()


def test_remask_sets_exactly_the_clipped_window():
    """Eq. remasking: positions [p, p + L) become MASK, clipped to the sequence end; nothing
    else changes (checked against a per-position rule on every p and L of a short row)."""
    T, mask = 12, 99
    base = np.arange(T, dtype=np.int32)
    for p in range(T + 1):
        for L in range(1, T + 3):
            x = base.copy()
            decode.remask(x, p, L, mask)
            for i in range(T):
                assert x[i] == (mask if p <= i < p + L else base[i])


def test_prefix_end_is_the_start_of_the_current_block():
    """N + Bk floor((p - N) / Bk): the largest block boundary (counted from N) not above p."""
    for N in (0, 3, 32):
        for Bk in (1, 4, 32):
            for p in range(N, N + 5 * Bk + 3):
                pe = decode.prefix_end(p, N, Bk)
                assert N <= pe <= p < pe + Bk
                assert (pe - N) % Bk == 0


def test_decision_confidence_modes():
    p1 = np.array([0.9, 0.5, 0.2])
    H = np.array([0.0, np.log(2.0), np.log(5.0)])
    np.testing.assert_array_equal(decode.decision_confidence(p1, None, decode.DecodeConfig(gen_len=3)), p1)
    c = decode.decision_confidence(p1, H, decode.DecodeConfig(gen_len=3, confidence=1))
    np.testing.assert_allclose(c, [1.0, 0.5, 0.2], rtol=1e-15)  # exp(-ln k) = 1/k
    with pytest.raises(ValueError):
        decode.decision_confidence(p1, None, decode.DecodeConfig(gen_len=3, confidence=1))
    with pytest.raises(ValueError):
        decode.decision_confidence(p1, H, decode.DecodeConfig(gen_len=3, confidence=2))
