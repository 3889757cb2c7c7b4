"""Pins of the oracle's building blocks against closed forms and textbook values."""
import math

import numpy as np
import pytest

from oracle import decoder as od


def test_gelu_is_the_erf_form():
    # GELU(x) = x * Phi(x); Phi(1) = 0.8413447460685429 (standard normal CDF table);
    # the tanh approximation would give 0.8411920.
    assert od.gelu(np.array(1.0)) == pytest.approx(0.8413447460685429, abs=1e-15)
    x = np.linspace(-6, 6, 97)
    np.testing.assert_allclose(od.gelu(x) - od.gelu(-x), x, atol=1e-14)   # Phi(x)+Phi(-x)=1
    assert od.gelu(np.array(0.0)) == 0.0


def test_layer_norm_moments_and_affine():
    rng = np.random.default_rng(0)
    x = rng.normal(3.0, 2.0, size=(5, 64))
    y = od.layer_norm(x, np.ones(64), np.zeros(64), 0.0)
    np.testing.assert_allclose(y.mean(-1), 0.0, atol=1e-13)
    np.testing.assert_allclose((y ** 2).mean(-1), 1.0, atol=1e-12)  # population variance
    g, b = rng.normal(size=64), rng.normal(size=64)
    np.testing.assert_allclose(od.layer_norm(x, g, b, 0.0), y * g + b, atol=1e-12)
    # eps enters under the square root: a constant row maps to the bias
    np.testing.assert_allclose(od.layer_norm(np.full((1, 8), 7.0), np.ones(8), b[:8], 1e-5), b[None, :8])


def test_linear_orientation_is_out_by_in():
    w = np.arange(6.0).reshape(2, 3)        # [out=2, in=3]
    y = od.linear(np.array([[1.0, 0.0, 0.0]]), w, np.array([10.0, 20.0]))
    np.testing.assert_array_equal(y, [[10.0, 23.0]])   # picks column 0 of each output row


def test_attention_closed_forms():
    rng = np.random.default_rng(1)
    dh, nh = 4, 2
    d = dh * nh
    q = rng.normal(size=(3, d))
    # head 0: all keys identical -> output is the mean of its values
    k = rng.normal(size=(5, d))
    k[:, :dh] = k[0, :dh]
    v = rng.normal(size=(5, d))
    out = od.multi_head_attention(q, k, v, nh)
    np.testing.assert_allclose(out[:, :dh], np.broadcast_to(v[:, :dh].mean(0), (3, dh)), atol=1e-13)
    # one key -> that key's value, for every head
    out1 = od.multi_head_attention(q, k[:1], v[:1], nh)
    np.testing.assert_allclose(out1, np.broadcast_to(v[0], (3, d)), atol=1e-13)
    # two keys whose dot products with q differ by delta: weight = logistic(delta / sqrt(dh))
    qq = np.zeros((1, dh)); qq[0, 0] = 1.0
    kk = np.zeros((2, dh)); kk[0, 0] = 3.0; kk[1, 0] = 1.0   # delta = 2
    vv = np.array([[1.0, 0, 0, 0], [0.0, 1, 0, 0]])
    o = od.multi_head_attention(qq, kk, vv, 1)
    w0 = 1.0 / (1.0 + math.exp(-2.0 / 2.0))                  # sqrt(4) = 2
    np.testing.assert_allclose(o[0, :2], [w0, 1 - w0], atol=1e-15)


def test_attention_mask_hides_keys():
    rng = np.random.default_rng(2)
    q, k, v = rng.normal(size=(2, 8)), rng.normal(size=(4, 8)), rng.normal(size=(4, 8))
    vis = np.array([[1, 1, 0, 0], [1, 1, 1, 1]], bool)
    a = od.multi_head_attention(q, k, v, 2, vis)
    v2 = v.copy(); v2[2:] = 1e6
    k2 = k.copy(); k2[2:] = -1e3
    b = od.multi_head_attention(q, k2, v2, 2, vis)
    np.testing.assert_allclose(a[0], b[0], atol=1e-12)
    assert not np.allclose(a[1], b[1])


def test_rope_rotation_convention():
    # one pair (dh=2): position p rotates (x1, x2) by +p radians (base^0 = 1)
    x = np.array([[1.0, 0.0]])
    y = od.rope(x, [1], 1, 10000.0)
    np.testing.assert_allclose(y, [[math.cos(1.0), math.sin(1.0)]], atol=1e-7)
    # dh=4: dim 0 pairs with dim 2 (half split), dim 1 with dim 3 at angle p*base^(-1/2)
    e0 = np.array([[1.0, 0, 0, 0]])
    y = od.rope(e0, [2], 1, 100.0)
    np.testing.assert_allclose(y, [[math.cos(2.0), 0, math.sin(2.0), 0]], atol=1e-6)
    e1 = np.array([[0, 1.0, 0, 0]])
    y = od.rope(e1, [2], 1, 100.0)
    np.testing.assert_allclose(y, [[0, math.cos(0.2), 0, math.sin(0.2)]], atol=1e-6)
    # position 0 is the identity
    z = np.random.default_rng(0).normal(size=(3, 128))
    np.testing.assert_allclose(od.rope(z, [0, 0, 0], 2, 1e4), z, atol=0)


def test_rope_depends_only_on_position_difference():
    rng = np.random.default_rng(3)
    q = rng.normal(size=(1, 64))
    k = rng.normal(size=(1, 64))
    s0 = (od.rope(q, [17], 1, 1e4) @ od.rope(k, [5], 1, 1e4).T).item()
    s1 = (od.rope(q, [117], 1, 1e4) @ od.rope(k, [105], 1, 1e4).T).item()
    assert s0 == pytest.approx(s1, abs=2e-4)        # FP32 phases: rounding-level change
    n = np.linalg.norm(od.rope(q, [300], 1, 1e4))
    assert n == pytest.approx(np.linalg.norm(q), rel=1e-12)
