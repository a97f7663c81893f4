"""The shared input generators: published SplitMix64 outputs, the weight
distribution, bf16 rounding, and the acceptance-input recipe."""
import numpy as np

import synthetic as syn


def test_splitmix64_published_outputs():
    # successive outputs of SplitMix64 seeded with 1234567 (Vigna's reference implementation)
    z = np.uint64(1234567)
    gamma = np.uint64(0x9E3779B97F4A7C15)
    got = []
    with np.errstate(over="ignore"):
        for _ in range(3):
            got.append(int(syn.splitmix64(z)))
            z = z + gamma
    assert got == [6457827717110365317, 3203168211198807973, 9817491932198370423]


def test_weight_generator_statistics_and_determinism():
    v = syn.weight_values(1, syn.tensor_id(syn.TensorKind.WQ, 3), 0, 1 << 20, 0.02)
    assert abs(float(v.mean())) < 2e-4
    assert abs(float(v.std()) - 0.02) < 2e-4
    assert np.abs(v).max() <= 0.02 * 3.47                  # Irwin-Hall(4) is bounded at +-sqrt(12)
    w = syn.weight_values(1, syn.tensor_id(syn.TensorKind.WQ, 3), 1000, 10, 0.02)
    assert (w == v[1000:1010]).all()
    assert (syn.round_bf16(v) == v).all()                   # values are bf16-exact
    g = syn.weight_values(1, syn.tensor_id(syn.TensorKind.ATTN_NORM, 0), 0, 4096, 0.0, 1.0)
    assert (g == 1.0).all()


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -8 + 2 ** -20, -2.5], np.float32)
    got = syn.round_bf16(x)
    assert list(got) == [1.0, 1.0, 1.0 + 2 ** -6, 1.0 + 2 ** -7, -2.5]
    b = syn.bf16_bits(np.array([1.0], np.float32))
    assert b[0] == 0x3F80


def test_accept_inputs_recipe():
    d = syn.accept_inputs(0, 8, 32, 1000, 999)
    assert d["logits_bf16"].shape == (8, 32, 1000)
    assert ((d["committed"] >= 0) & (d["committed"] <= 32)).all()
    q = d["target_p1"]
    frac_mid = ((q > 0.65) & (q < 0.9)).mean()
    assert 0.3 < frac_mid < 0.7
    z = syn.bf16_to_f32(d["logits_bf16"]).astype(np.float64)
    top = np.argmax(z, axis=2)
    assert (top == d["top_index"]).all()


def test_weight_values_chunked_threaded_equals_definition():
    """The generator runs in threaded, cache-sized chunks; it must equal the definition in
    its docstring evaluated in one pass (a sub-range straddling thread boundaries)."""
    seed, tid, start, count, std, mean = 3, syn.tensor_id(syn.TensorKind.W_UP, 7), 12_345, 5_000_003, 0.3, -0.5
    idx = np.arange(start, start + count, dtype=np.uint64)
    key = (np.uint64(seed) << np.uint64(48)) | (np.uint64(tid) << np.uint64(32)) | idx
    h = syn.splitmix64(key)
    m16 = np.uint64(0xFFFF)
    s = ((h & m16) + ((h >> np.uint64(16)) & m16) + ((h >> np.uint64(32)) & m16)
         + (h >> np.uint64(48))).astype(np.int64)
    w = (s - 131070).astype(np.float32) * np.float32(float(np.float32(std)) / syn.GEN_SIGMA4)
    w = syn.round_bf16(w + np.float32(mean))
    got = syn.weight_values(seed, tid, start, count, std, mean)
    assert np.array_equal(got.view(np.uint32), w.view(np.uint32))
