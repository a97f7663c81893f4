"""Pins of the entropy confidence and of Eq. entropy_bound in the oracle.

The marginal entropy H = -sum_v P(v) ln P(v) of the Eq. 2 distribution is checked
against closed forms (uniform, two-level distributions), an independent library
routine (scipy.stats.entropy on probabilities), its invariances and bounds; the bound
function against the total correlation of brute-force joint distributions (the KL
divergence that Eq. entropy_bound bounds); the decoder with ``confidence = 1`` against
its special cases and against the top-1 decoder it can never out-accept.
"""
import numpy as np
import pytest
import scipy.stats

from oracle import decode, model
import synthetic as syn


# ----------------------------------------------------------- marginal entropy

@pytest.mark.parametrize("V", [2, 3, 8, 4096, 126464])
def test_entropy_uniform_is_log_v(V):
    for z0 in (0.0, -3.5, 17.0):
        assert model.entropy(np.full(V, z0))[0] == pytest.approx(np.log(V), rel=1e-12)


def test_entropy_two_level_closed_form():
    # one logit a, the other V-1 logits 0: P(top) = e^a / (e^a + V - 1)
    for V in (2, 3, 50):
        for a in (0.0, 0.3, 2.0, 9.0, 40.0):
            z = np.zeros(V)
            z[V // 2] = a
            q = np.exp(a) / (np.exp(a) + V - 1)
            r = (1 - q) / (V - 1)
            H = -q * np.log(q) - ((V - 1) * r * np.log(r) if r > 0 else 0.0)
            assert model.entropy(z)[0] == pytest.approx(H, rel=1e-10, abs=1e-14)


def test_entropy_matches_scipy_on_random_rows():
    rng = np.random.default_rng(3)
    for scale in (0.1, 1.0, 5.0, 30.0):
        z = rng.normal(size=(16, 1000)) * scale
        p = np.exp(z - z.max(axis=1, keepdims=True))
        ref = scipy.stats.entropy(p, axis=1)  # normalises p itself
        np.testing.assert_allclose(model.entropy(z), ref, rtol=1e-11, atol=1e-13)


def test_entropy_shift_invariance_bounds_and_order():
    rng = np.random.default_rng(5)
    z = rng.normal(size=(64, 300)) * rng.uniform(0.1, 20.0, size=(64, 1))
    H = model.entropy(z)
    np.testing.assert_allclose(model.entropy(z + 123.0), H, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(model.entropy(z[:, ::-1]), H, rtol=1e-12, atol=1e-14)
    assert (H >= 0).all() and (H <= np.log(300) + 1e-12).all()
    # exp(-H) <= sum_v P(v)^2 <= p1 (Jensen on ln, then sum P^2 <= max P)
    p = model.softmax(z)
    _, p1, _ = model.confidence(z)
    c = decode.entropy_confidence(H)
    assert (c <= (p * p).sum(axis=1) * (1 + 1e-12)).all()
    assert (c <= p1 * (1 + 1e-12)).all()
    assert (c >= 1.0 / 300 * (1 - 1e-12)).all()


def test_entropy_of_an_underflowed_distribution():
    # probabilities that underflow to 0 contribute their limit 0 (no NaN)
    z = np.array([[0.0, -800.0, -900.0], [1000.0, 0.0, 0.0]])
    H = model.entropy(z)
    assert np.isfinite(H).all()
    assert H[0] == 0.0 and H[1] == 0.0


# ------------------------------------------------------------ Eq. entropy_bound

def test_jpde_bound_special_cases():
    assert decode.jpde_bound([]) == 0.0
    assert decode.jpde_bound([2.5]) == 0.0
    assert decode.jpde_bound([0.4] * 5) == pytest.approx(4 * 0.4)
    rng = np.random.default_rng(2)
    for _ in range(200):
        h = rng.random(int(rng.integers(2, 20))) * 3
        b = decode.jpde_bound(h)
        assert b == pytest.approx(decode.jpde_bound(rng.permutation(h)))
        assert b >= 0
        assert b == pytest.approx(sum(sorted(h)[:-1]))  # all but the largest


def test_jpde_bound_dominates_the_kl_of_brute_force_joints():
    """D_KL(P || prod_i P_i) = sum_i H_i - H(P) <= sum_i H_i - max_j H_j (Eq. entropy_bound)."""
    rng = np.random.default_rng(11)
    for n_var, V in ((2, 2), (2, 5), (3, 3), (4, 2)):
        for _ in range(100):
            P = rng.dirichlet(np.full(V ** n_var, rng.choice([0.1, 1.0, 5.0]))).reshape((V,) * n_var)
            marg = [P.sum(axis=tuple(a for a in range(n_var) if a != i)) for i in range(n_var)]
            Q = marg[0]
            for m in marg[1:]:
                Q = np.multiply.outer(Q, m)
            nz = P > 0
            kl = float((P[nz] * np.log(P[nz] / Q[nz])).sum())
            H = [float(-(m[m > 0] * np.log(m[m > 0])).sum()) for m in marg]
            assert kl <= decode.jpde_bound(H) + 1e-12
            # a product distribution has zero KL; the bound stays >= 0
            assert kl >= -1e-12


# ------------------------------------------------------ decoding with exp(-H)

MICRO = syn.ModelShape(n_layers=1, d_model=32, n_heads=2, n_kv_heads=2, head_dim=16,
                       ffn_dim=64, vocab=64, mask_id=63, rope_theta=10000.0)


def _gen(seed, tau_c, tau_d, window, confidence, N=4, M=12, B=2):
    w = syn.model_weights(MICRO, seed, lm_head_scale=40.0, norm_gain_std=0.1)

    def predict(tokens):
        ids, p1, p2, H = model.predict(MICRO, w, tokens, with_entropy=True)
        return ids[N:], p1[N:], p2[N:], H[N:]
    prompt = syn.prompt_ids(seed + 100, B, N, MICRO.mask_id)
    cfg = decode.DecodeConfig(tau_commit=tau_c, tau_draft=tau_d, max_window=window, gen_len=M,
                              confidence=confidence)
    return decode.generate(predict, prompt, cfg, MICRO.mask_id), cfg


@pytest.mark.parametrize("seed", [0, 1])
def test_entropy_decoder_special_cases(seed):
    M = 12
    out, _ = _gen(seed, 1.0, 2.0, 6, 1, M=M)  # exp(-H) < 1 never passes tau_c = 1
    assert out["done"] and (out["k"] == 1).all() and out["n_iter"] == M
    assert np.nanmax(out["jpde"]) == 0.0     # single tokens: no joint error
    out, _ = _gen(seed, 0.0, 2.0, 5, 1, M=M)  # exp(-H) > 0 always passes tau_c = 0
    assert out["n_iter"] == -(-M // 5)
    assert list(out["k"][:, 0]) == [5, 5, 2]


@pytest.mark.parametrize("seed", [0, 1, 2])
@pytest.mark.parametrize("tau_c,window", [(0.3, 6), (0.5, 12), (0.2, 3)])
def test_entropy_decoder_never_accepts_more_than_top1(seed, tau_c, window):
    """Same state, same predictions: exp(-H) <= p1 gives K_entropy <= K_top1 (Eq. compute_k)."""
    out, cfg = _gen(seed, tau_c, 2.0, window, 1)
    N = 4
    p = np.full(2, N)
    for step, (xin, pr) in enumerate(zip(out["inputs"], out["preds"])):
        for b in range(2):
            if p[b] >= xin.shape[1]:
                continue
            ids, p1, _, H = pr[:, b]
            w_eff = min(window, xin.shape[1] - p[b])
            k_top1 = max(decode.window_length(p1[p[b] - N:p[b] - N + w_eff], tau_c), 1)
            k_ent = max(decode.window_length(np.exp(-H[p[b] - N:p[b] - N + w_eff]), tau_c), 1)
            assert int(out["k"][step, b]) == min(k_ent, w_eff)
            assert k_ent <= max(k_top1, 1)
            # the recorded bound is Eq. entropy_bound on the committed set [p, p + K)
            K = int(out["k"][step, b])
            Hs = H[p[b] - N:p[b] - N + K]
            assert out["jpde"][step, b] == pytest.approx(Hs.sum() - Hs.max() if K > 1 else 0.0)
            p[b] += K
    assert out["done"]


def test_top1_decoder_is_unchanged_by_entropy_outputs():
    """confidence = 0 ignores H: the trajectory equals the one from (ids, p1, p2) alone."""
    w = syn.model_weights(MICRO, 4, lm_head_scale=40.0, norm_gain_std=0.1)
    N, M = 4, 12
    prompt = syn.prompt_ids(104, 2, N, MICRO.mask_id)
    cfg = decode.DecodeConfig(tau_commit=0.5, tau_draft=0.9, max_window=6, gen_len=M)
    a = decode.generate(lambda t: tuple(v[N:] for v in model.predict(MICRO, w, t)), prompt, cfg, MICRO.mask_id)
    b = decode.generate(lambda t: tuple(v[N:] for v in model.predict(MICRO, w, t, with_entropy=True)), prompt,
                        cfg, MICRO.mask_id)
    assert (a["x"] == b["x"]).all() and (a["k"] == b["k"]).all()
    active = a["start"] >= 0  # finished rows commit nothing and record 0
    assert np.isnan(a["jpde"][active]).all() and (a["jpde"][~active] == 0).all()
    assert np.isfinite(b["jpde"]).all()


def test_entropy_confidence_requires_entropies():
    cfg = decode.DecodeConfig(gen_len=4, confidence=1)
    with pytest.raises(ValueError):
        decode.generate(lambda t: (np.zeros(4, np.int32), np.ones(4), np.zeros(4)), np.zeros((1, 2), np.int32),
                        cfg, 63)
