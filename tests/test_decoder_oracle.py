"""Pins of the reference decoder layer (oracle/decoder.py) against closed forms and invariants."""
import math

import numpy as np
import pytest

import oracle
from oracle import decoder
from paper_2506_01374_gb300 import inputs


def test_bf16_round_is_nearest_even():
    rng = np.random.default_rng(0)
    x = rng.standard_normal(20000).astype(np.float32)
    got = decoder.bf16_round(x.astype(np.float64))
    u = x.view(np.uint32)
    lo = (u & 0xFFFF0000).view(np.float32).astype(np.float64)          # truncation (toward zero)
    hi = ((u & 0xFFFF0000) + 0x10000).view(np.float32).astype(np.float64)  # next bf16 away from zero
    xd = x.astype(np.float64)
    dl, dh = np.abs(xd - lo), np.abs(hi - xd)
    even_lo = ((u >> 16) & 1) == 0
    want = np.where(dl < dh, lo, np.where(dh < dl, hi, np.where(even_lo, lo, hi)))
    np.testing.assert_array_equal(got, want)
    # exact ties: 1 + 2^-8 lies halfway between 1 and 1 + 2^-7 and goes to the even 1
    assert decoder.bf16_round(np.array([1 + 2.0 ** -8]))[0] == 1.0
    assert decoder.bf16_round(np.array([1 + 3 * 2.0 ** -8]))[0] == 1 + 2.0 ** -6


def test_rmsnorm_closed_forms():
    g = np.linspace(0.5, 1.5, 8)
    # a constant row c has mean square c^2: output g * c / sqrt(c^2 + eps)
    c = 3.0
    np.testing.assert_allclose(decoder.rmsnorm(np.full((1, 8), c), g, 1e-5)[0], g * c / math.sqrt(c * c + 1e-5))
    # scale invariance for eps = 0, and unit mean square of the normalised row
    rng = np.random.default_rng(1)
    x = rng.standard_normal((5, 8))
    np.testing.assert_allclose(decoder.rmsnorm(7.0 * x, g, 0.0), decoder.rmsnorm(x, g, 0.0), rtol=1e-12)
    n = decoder.rmsnorm(x, np.ones(8), 0.0)
    np.testing.assert_allclose(np.mean(n * n, axis=1), 1.0, rtol=1e-12)


def test_rope_closed_form_identity_and_relative_position():
    # D = 4, theta = 10000: pair 0 turns by p, pair 1 by p * 10000^(-1/2) = p / 100
    x = np.array([[[1.0, 2.0, 3.0, 4.0]]])
    got = decoder.rope(x, [1], 10000.0)[0, 0]
    a0, a1 = 1.0, 0.01
    want = [1 * math.cos(a0) - 3 * math.sin(a0), 2 * math.cos(a1) - 4 * math.sin(a1),
            3 * math.cos(a0) + 1 * math.sin(a0), 4 * math.cos(a1) + 2 * math.sin(a1)]
    np.testing.assert_allclose(got, want, rtol=1e-14)
    rng = np.random.default_rng(2)
    q = rng.standard_normal((6, 3, 128))
    k = rng.standard_normal((6, 3, 128))
    np.testing.assert_allclose(decoder.rope(q[:1], [0], 5e5), q[:1], rtol=0, atol=0)  # position 0: identity
    rq = decoder.rope(q, np.arange(6), 5e5)
    # each rotated pair keeps its length
    np.testing.assert_allclose(rq[..., :64] ** 2 + rq[..., 64:] ** 2, q[..., :64] ** 2 + q[..., 64:] ** 2, rtol=1e-12)
    # scores depend on the position difference only
    d1 = np.sum(decoder.rope(q, [3] * 6, 5e5) * decoder.rope(k, [1] * 6, 5e5), axis=-1)
    d2 = np.sum(decoder.rope(q, [10] * 6, 5e5) * decoder.rope(k, [8] * 6, 5e5), axis=-1)
    np.testing.assert_allclose(d1, d2, rtol=1e-9, atol=1e-9)


@pytest.fixture(scope="module")
def small():
    return inputs.decoder_layer(48, 256, 4, 2, 384, seed=9)


def test_layer_with_zero_output_projections_is_the_identity(small):
    x, g1, Wqkv, Wo, g2, W1, W2 = small
    zero_o, zero_2 = np.zeros_like(Wo), np.zeros_like(W2)
    y = decoder.decoder_layer_bf16(x, g1, Wqkv, zero_o, g2, W1, zero_2, 4, 2)
    np.testing.assert_array_equal(y, inputs.bf16_bits_to_f64(x))


def test_layer_without_attention_is_residual_plus_mlp(small):
    x, g1, Wqkv, Wo, g2, W1, W2 = small
    y = decoder.decoder_layer_bf16(x, g1, Wqkv, np.zeros_like(Wo), g2, W1, W2, 4, 2)
    X = inputs.bf16_bits_to_f64(x)
    b = decoder.bf16_bits(decoder.rmsnorm(X, inputs.bf16_bits_to_f64(g2), 1e-5))
    np.testing.assert_allclose(y, X + oracle.mlp_bf16(b, W1, W2), rtol=1e-12, atol=1e-12)


def test_layer_first_token_attends_to_itself_only(small):
    # with W2 = 0, row 0 of the layer is x0 + (v0 of every head's KV group) Wo^T: the only visible key
    x, g1, Wqkv, Wo, g2, W1, W2 = small
    y0 = decoder.decoder_layer_bf16(x, g1, Wqkv, Wo, g2, W1, np.zeros_like(W2), 4, 2, rows=[0])[0]
    X = inputs.bf16_bits_to_f64(x)
    a = decoder.bf16_round(decoder.rmsnorm(X[:1], inputs.bf16_bits_to_f64(g1), 1e-5))
    v = decoder.bf16_round((a @ inputs.bf16_bits_to_f64(Wqkv).T)[0, 6 * 128:].reshape(2, 128))
    o = np.concatenate([v[h // 2] for h in range(4)])
    want = decoder.bf16_round(X[0] + o @ inputs.bf16_bits_to_f64(Wo).T)
    np.testing.assert_allclose(y0, want, rtol=1e-12, atol=1e-12)


def test_row_sampling_matches_full_layer(small):
    x, g1, Wqkv, Wo, g2, W1, W2 = small
    full = decoder.decoder_layer_bf16(x, g1, Wqkv, Wo, g2, W1, W2, 4, 2)
    rows = [0, 5, 17, 47]
    np.testing.assert_allclose(decoder.decoder_layer_bf16(x, g1, Wqkv, Wo, g2, W1, W2, 4, 2, rows=rows), full[rows],
                               rtol=1e-12, atol=1e-12)
