"""The seeded input generators: determinism, distributions, padding."""
import numpy as np
import pytest

from synth import generators as G
from synth import workloads as W


def test_splitmix64_reference_values():
    # First outputs of SplitMix64 seeded with 0 (state advanced by the golden
    # gamma before mixing), as published with the algorithm.
    z = np.array([0, 0x9E3779B97F4A7C15, 2 * 0x9E3779B97F4A7C15 & (2**64 - 1)], np.uint64)
    assert [int(v) for v in G.mix(z)] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_normal_moments_and_support():
    e = G.element_hash(G.key(1, 1, 0, 0), np.arange(1 << 20))
    z = G.normal(e, 0).astype(np.float64)
    assert abs(z.mean()) < 5 / 1024 and abs(z.var() - 1) < 0.01
    assert z.min() >= -6 and z.max() <= 6
    assert abs(np.mean(z ** 4) - 3 + 1.2 / 12) < 0.05     # Irwin-Hall(12) kurtosis 3 - 0.1


def test_gradient_kinds():
    idx = np.arange(1 << 18)
    lay = W.layout([1 << 18])
    n = G.grad_values("normal", 5, 0, 3, idx, 0.01)
    assert n.dtype == np.float32 and abs(n.std() - 0.01) < 2e-4
    t3 = G.grad_values("student_t3", 5, 0, 3, idx, 1.0)
    assert abs(np.median(np.abs(t3)) - 0.765) < 0.02 and np.isfinite(t3).all()
    o = G.grad_values("normal_outliers", 5, 0, 3, idx, 1e-3)
    frac = np.mean(np.abs(o) > 0.0065)
    assert 0.008 < frac < 0.012
    w = {"grad_kind": "normal", "grad_sigma": 1.0, "grad_dtype": "bf16"}
    b = G.grads(w, lay, 5, 0, 3, idx)
    assert np.array_equal(G.round_bf16(b), b)
    assert not np.array_equal(b, G.grad_values("normal", 5, 0, 3, idx, 1.0))


def test_bf16_round_to_nearest_even():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -9, -2.5], np.float32)
    np.testing.assert_array_equal(G.round_bf16(x), np.array([1.0, 1.0, 1.015625, 1.0, -2.5],
                                                            np.float32))


def test_determinism_and_independence():
    idx = np.arange(4096)
    a = G.grad_values("normal", 9, 1, 2, idx, 1.0)
    assert np.array_equal(a, G.grad_values("normal", 9, 1, 2, idx, 1.0))
    assert np.array_equal(a[100:200], G.grad_values("normal", 9, 1, 2, idx[100:200], 1.0))
    for other in (G.grad_values("normal", 9, 0, 2, idx, 1.0), G.grad_values("normal", 9, 1, 3, idx, 1.0),
                  G.grad_values("normal", 10, 1, 2, idx, 1.0)):
        assert abs(np.corrcoef(a, other)[0, 1]) < 0.06


def test_padding_is_zero():
    shapes = [5, 3, 17]
    lay = W.layout(shapes)
    w = {"grad_kind": "normal", "grad_sigma": 1.0, "grad_dtype": "f32", "init_sigma": 0.02}
    idx = np.arange(lay["n_padded"])
    g = G.grads(w, lay, 1, 0, 0, idx)
    x = G.init_params(w, lay, 2, idx)
    inside = np.zeros(lay["n_padded"], bool)
    for off, num in zip(lay["offsets"], lay["numels"]):
        inside[off:off + num] = True
    assert np.all(g[~inside] == 0) and np.all(x[~inside] == 0)
    assert np.all(g[inside] != 0)


def _rosenbrock(x):
    a, b = x[0::2], x[1::2]
    return float(np.sum((1.0 - a) ** 2 + 100.0 * (b - a * a) ** 2))


def _central_diff(f, x, h=1e-6):
    g = np.empty_like(x)
    for i in range(x.size):
        e = np.zeros_like(x)
        e[i] = h
        g[i] = (f(x + e) - f(x - e)) / (2 * h)
    return g


def test_toy_gradients_match_their_objectives():
    """Without noise the toy gradients are the derivatives of the two
    objectives (quadratic sum lam x^2 / 2 of Figure 2, Rosenbrock pairs of
    Figure 1), checked against central differences of the objectives
    themselves; the Rosenbrock minimum (1, 1) has zero gradient."""
    rng = np.random.default_rng(7)
    x = rng.uniform(-1.5, 1.5, size=(3, 12))
    lam = rng.uniform(0.1, 10.0, size=12)
    gq = G.toy_grad("quadratic", x, 1, 0, 0.0, lam=lam)
    gr = G.toy_grad("rosenbrock", x, 1, 0, 0.0)
    for m in range(3):
        fq = lambda v: float(np.sum(lam * v * v) / 2)
        np.testing.assert_allclose(gq[m], _central_diff(fq, x[m]), rtol=1e-6, atol=1e-6)
        np.testing.assert_allclose(gr[m], _central_diff(_rosenbrock, x[m]), rtol=1e-6, atol=1e-4)
    assert np.all(G.toy_grad("rosenbrock", np.ones((2, 6)), 1, 0, 0.0) == 0.0)


def test_toy_gradient_noise():
    """sigma scales standard normal noise that depends on the worker, the
    step and the index, and not on x."""
    x = np.zeros((2, 1 << 16))
    g = G.toy_grad("quadratic", x, 5, 3, 0.5, lam=np.ones(1 << 16))
    assert abs(g.mean()) < 0.01 and abs(g.std() - 0.5) < 0.01
    assert not np.array_equal(g[0], g[1])
    g_next = G.toy_grad("quadratic", x, 5, 4, 0.5, lam=np.ones(1 << 16))
    assert not np.array_equal(g, g_next)
    x2 = np.full((2, 1 << 16), 3.0)
    g2 = G.toy_grad("quadratic", x2, 5, 3, 0.5, lam=np.ones(1 << 16))
    np.testing.assert_allclose(g2 - 3.0, g, atol=1e-12)


@pytest.mark.parametrize("name, d, ffn, blocks, total", [
    ("gpt2_small", 768, 3072, 12, 123_570_432),
    ("decoder_350m", 1024, 4096, 24, 353_553_408),
    ("decoder_1b", 2048, 8192, 24, 1_311_086_592),
])
def test_decoder_lists_count_the_architecture(name, d, ffn, blocks, total):
    """The named parameter lists hold V*d + L*(4 d^2 + 2 d F + 4 d) + 2 d
    values (embedding; per block qkv, projection, two FFN matrices and two
    layer norms; final layer norm) in 1 + 8 L + 2 tensors, all multiples of
    8, so the padded layout adds nothing before the slab's last tail."""
    shapes = W.WORKLOADS[name]["shapes"]
    assert len(shapes) == 1 + 8 * blocks + 2
    assert sum(shapes) == W.VOCAB * d + blocks * (4 * d * d + 2 * d * ffn + 4 * d) + 2 * d == total
    assert all(s % 8 == 0 for s in shapes)
    assert W.layout(shapes)["n_padded"] == -(-total // 256) * 256
