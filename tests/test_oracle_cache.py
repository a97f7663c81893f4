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
