"""Pins of the oracle's approximate prefix cache (``kv_cache = 1``): it reduces to the
full forward where nothing is stale, hides exactly the prefix tokens changed since the
last refresh, and with block length 1 (a refresh at every step) reproduces the uncached
Algorithm 1 token for token."""
import numpy as np
import pytest

import synthetic as syn
from oracle import decode, model

TINY = syn.SHAPES["tiny"]
N, M = 32, 64
T = N + M


@pytest.fixture(scope="module")
def weights():
    return syn.model_weights(TINY, 0, lm_head_scale=40.0, norm_gain_std=0.1)


def _tokens(seed):
    rng = np.random.default_rng(seed)
    return rng.integers(0, TINY.vocab, T).astype(np.int32)


@pytest.mark.parametrize("bf16", [False, True])
def test_all_rows_equal_full_forward(weights, bf16):
    x = _tokens(1)
    kv = model.new_kv_store(TINY, T)
    got = model.forward_rows(TINY, weights, x, np.arange(T), kv, bf16)
    ref = model.forward_hidden(TINY, weights, x, bf16)
    assert np.array_equal(got, ref)


@pytest.mark.parametrize("pe", [N, N + 32, T - 1])
def test_suffix_with_fresh_store_equals_full_forward(weights, pe):
    """Keys / values stored by a full pass over the same tokens are not stale: the suffix
    rows then equal the full forward (up to summation order)."""
    x = _tokens(2)
    kv = model.new_kv_store(TINY, T)
    model.forward_rows(TINY, weights, x, np.arange(T), kv)
    got = model.forward_rows(TINY, weights, x, np.arange(pe, T), kv)
    ref = model.forward_hidden(TINY, weights, x)[pe:]
    assert np.abs(got - ref).max() <= 1e-10 * np.abs(ref).max()


def test_store_hides_prefix_changes_only(weights):
    """After a refresh, changing prefix tokens leaves the suffix rows unchanged (the
    prefix is seen through its stored keys / values); changing a suffix token does not."""
    pe = N + 16
    x = _tokens(3)
    kv = model.new_kv_store(TINY, T)
    model.forward_rows(TINY, weights, x, np.arange(T), kv)
    base = model.forward_rows(TINY, weights, x, np.arange(pe, T), [[k.copy(), v.copy()] for k, v in kv])
    y = x.copy()
    y[:pe] = (y[:pe] + 7) % TINY.vocab
    hid = model.forward_rows(TINY, weights, y, np.arange(pe, T), [[k.copy(), v.copy()] for k, v in kv])
    assert np.abs(hid - base).max() <= 1e-10 * np.abs(base).max()
    z = x.copy()
    z[T - 1] = (z[T - 1] + 7) % TINY.vocab
    hid = model.forward_rows(TINY, weights, z, np.arange(pe, T), [[k.copy(), v.copy()] for k, v in kv])
    assert np.abs(hid[0] - base[0]).max() > 1e-6  # bidirectional: row pe sees position T-1


def _cached_fn(weights):
    return lambda tok, start, state: model.predict_from(TINY, weights, tok, start, state, N)


def _full_fn(weights):
    return lambda tok: model.predict(TINY, weights, tok, rows=slice(N, T))


@pytest.mark.parametrize("seed,tau_c,L", [(0, 0.7, 32), (1, 0.4, 16)])
def test_block_length_one_is_full_recompute(weights, seed, tau_c, L):
    """Bk = 1: the prefix end moves at every step, so every step refreshes."""
    prompt = syn.prompt_ids(seed, 2, N, TINY.mask_id)
    full = decode.generate(_full_fn(weights), prompt,
                           decode.DecodeConfig(tau_commit=tau_c, max_window=L, gen_len=M), TINY.mask_id)
    cached = decode.generate(_cached_fn(weights), prompt,
                             decode.DecodeConfig(tau_commit=tau_c, max_window=L, gen_len=M, block_len=1,
                                                 kv_cache=1), TINY.mask_id)
    assert np.array_equal(full["x"], cached["x"])
    assert np.array_equal(full["k"], cached["k"])
    assert ((cached["start"] == 0) | (cached["start"] == -1)).all()


def test_refresh_exactly_at_block_changes(weights):
    prompt = syn.prompt_ids(5, 2, N, TINY.mask_id)
    cfg = decode.DecodeConfig(tau_commit=0.6, max_window=32, gen_len=M, block_len=16, kv_cache=1)
    out = decode.generate(_cached_fn(weights), prompt, cfg, TINY.mask_id)
    assert out["done"]
    for b in range(2):
        p = N
        pe_prev = None
        for k, s in zip(out["k"][:, b], out["start"][:, b]):
            if p >= T:
                assert s == -1 and k == 0
                continue
            pe = N + 16 * ((p - N) // 16)
            assert s == (0 if pe != pe_prev else pe)
            pe_prev = pe
            assert 1 <= k <= min(32, T - p)
            p += k
        assert p == T
    # the committed region is a contiguous run and nothing is MASK at the end
    assert (out["x"][:, N:] != TINY.mask_id).all()


# ---------------------------------------------------------------- the dual cache (kv_cache = 2)
def _predict(weights, with_entropy=False):
    def fn(tokens, start, state, end=None):
        return model.predict_from(TINY, weights, tokens, start, state, N, with_entropy=with_entropy, end=end)
    return fn


def _run(weights, seed, kv_cache, block_len, tau_c=0.5, tau_d=0.9, L=16):
    prompt = np.random.default_rng(seed).integers(0, TINY.vocab - 1, (1, N)).astype(np.int32)
    cfg = decode.DecodeConfig(tau_commit=tau_c, tau_draft=tau_d, max_window=L, block_len=block_len, gen_len=M,
                              kv_cache=kv_cache)
    if kv_cache:
        return decode.generate(_predict(weights), prompt, cfg, TINY.mask_id)
    fn = _predict(weights)
    return decode.generate(lambda toks: fn(toks, 0, {}), prompt, cfg, TINY.mask_id)


@pytest.mark.parametrize("seed,tau_c", [(5, 0.5), (6, 0.3)])
def test_dual_with_one_block_equals_the_prefix_cache(weights, seed, tau_c):
    """A block as long as the generation: every step after the first computes [N, T) with
    fresh predictions at every generation position and the block end is T, so the dual
    cache is the prefix cache, token for token and step for step."""
    a = _run(weights, seed, 2, M, tau_c)
    b = _run(weights, seed, 1, M, tau_c)
    assert np.array_equal(a["x"], b["x"]) and np.array_equal(a["k"], b["k"])
    assert np.array_equal(a["start"], b["start"]) and (a["end"] == T).all()


def test_dual_with_block_one_equals_the_uncached_loop(weights):
    """Block length 1: the prefix end is p itself and moves at every step (K >= 1), so
    every step refreshes (a full forward over fresh keys / values): the uncached
    Algorithm 1."""
    a = _run(weights, 7, 2, 1)
    b = _run(weights, 7, 0, 1)
    assert np.array_equal(a["x"], b["x"]) and np.array_equal(a["k"], b["k"])
    assert (a["start"] == 0).all() and (a["end"] == T).all()


@pytest.mark.parametrize("seed,tau_c,bk", [(10, 0.5, 8), (10, 0.7, 16), (8, 0.9, 32), (16, 0.7, 8)])
def test_dual_steps_between_refreshes_stay_in_the_block(weights, seed, tau_c, bk):
    """Between refreshes a dual step computes exactly the current block [b0, b0 + Bk)
    (clipped to T), commits only inside it, and the predictions it uses outside the block
    are those of the last step that computed them (the refresh); every generation ends
    with the whole sequence committed."""
    r = _run(weights, seed, 2, bk, tau_c)
    assert r["done"]
    p = N
    last = None
    n_between = 0
    for s, (k, st, en, pr) in enumerate(zip(r["k"][:, 0], r["start"][:, 0], r["end"][:, 0], r["preds"])):
        b0 = N + bk * ((p - N) // bk)
        if st == 0:
            assert en == T
            last = pr[:, 0].copy()
        else:
            n_between += 1
            assert st == b0 and en == min(b0 + bk, T)
            assert 1 <= k <= en - p
            out = np.r_[0:st - N, en - N:M]
            assert np.array_equal(pr[:3, 0][:, out], last[:3][:, out])
            last[:, st - N:en - N] = pr[:, 0][:, st - N:en - N]
        p += int(k)
    assert p == T and n_between > 0


def test_dual_cap_binds_where_the_window_runs_past_the_block(weights):
    """The cap is what keeps commits inside the block: on the same trajectory, some step
    between refreshes would have committed past the block end had K not been capped (its
    confident run, by Eq. compute_k over the whole window, reaches beyond the block)."""
    r = _run(weights, 16, 2, 8, 0.7)
    p, capped = N, 0
    for k, st, en, pr in zip(r["k"][:, 0], r["start"][:, 0], r["end"][:, 0], r["preds"]):
        if st > 0:
            c = np.zeros(T)
            c[N:] = pr[1, 0]
            w_eff = min(16, T - p)
            k_free = max(decode.window_length(c[p:p + w_eff], 0.7), 1)
            if k_free > en - p:
                capped += 1
                assert k == en - p
        p += int(k)
    assert capped > 0
