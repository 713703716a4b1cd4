"""Pins of the float64 decoder-layer oracle (oracle/layer.py) against closed
forms and invariants: the rotary embedding's pairing, sign and frequencies,
its relative-position property, RMSNorm's unit mean square, SiLU's values,
and the residual structure of the layer."""
import math

import numpy as np
import pytest

from oracle import layer as L

THETA = 1.0e6


def test_rope_position_zero_is_identity():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((3, 2, 128))
    np.testing.assert_allclose(L.rope(x, [0, 0, 0], THETA), x, atol=0, rtol=0)


def test_rope_pairing_sign_and_frequency_closed_form():
    # unit vector at element f: its pair (f, f + 64) turns by pos * theta^(-f/64),
    # the first element to cos, the second to +sin (rotate-half convention)
    for f, pos in [(0, 5), (1, 7), (33, 1000), (63, 32767)]:
        x = np.zeros((1, 1, 128))
        x[0, 0, f] = 1.0
        y = L.rope(x, [pos], THETA)[0, 0]
        a = pos * THETA ** (-f / 64)
        assert y[f] == pytest.approx(math.cos(a), abs=1e-12)
        assert y[f + 64] == pytest.approx(math.sin(a), abs=1e-12)
        assert np.count_nonzero(np.abs(y) > 1e-15) <= 2
        # and the second element of the pair goes to (-sin, cos)
        x = np.zeros((1, 1, 128))
        x[0, 0, f + 64] = 1.0
        y = L.rope(x, [pos], THETA)[0, 0]
        assert y[f] == pytest.approx(-math.sin(a), abs=1e-12)
        assert y[f + 64] == pytest.approx(math.cos(a), abs=1e-12)


def test_rope_relative_positions():
    # <rope(q, a), rope(k, b)> depends only on a - b, and each pair keeps its norm
    rng = np.random.default_rng(1)
    q = rng.standard_normal((1, 1, 128))
    k = rng.standard_normal((1, 1, 128))
    dots = []
    for a, b in [(10, 3), (1017, 1010), (30007, 30000)]:
        ra, rb = L.rope(q, [a], THETA), L.rope(k, [b], THETA)
        dots.append(float(np.sum(ra * rb)))
        n0 = q[0, 0, :64] ** 2 + q[0, 0, 64:] ** 2
        n1 = ra[0, 0, :64] ** 2 + ra[0, 0, 64:] ** 2
        np.testing.assert_allclose(n1, n0, rtol=1e-12)
    assert dots[0] == pytest.approx(dots[1], rel=1e-9)
    assert dots[0] == pytest.approx(dots[2], rel=1e-8)


def test_rms_norm_unit_mean_square_and_scale_invariance():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((4, 256)) * 3.0
    y = L.rms_norm(x, np.ones(256), 0.0)
    np.testing.assert_allclose(np.mean(y * y, axis=1), 1.0, rtol=1e-12)
    np.testing.assert_allclose(L.rms_norm(7.5 * x, np.ones(256), 0.0), y, rtol=1e-12)
    w = rng.standard_normal(256)
    np.testing.assert_allclose(L.rms_norm(x, w, 0.0), y * w, rtol=1e-12)


def test_silu_values():
    gu = np.array([[0.0, 1.0, -1.0, 2.0, 1.0, 1.0]])
    y = L.silu_mul(gu, 3)
    # gate (0, 1, -1), up (2, 1, 1)
    np.testing.assert_allclose(y[0], [0.0, 1.0 / (1.0 + math.exp(-1.0)) * 1.0,
                                      -1.0 / (1.0 + math.exp(1.0)) * 1.0], rtol=1e-15)
    assert y[0, 2] == pytest.approx(-0.2689414213699951, rel=1e-15)
    assert y[0, 1] == pytest.approx(0.7310585786300049, rel=1e-15)


def test_bf16_round_trip():
    u = np.array([0x3F80, 0xBF80, 0x0000, 0x4049, 0x7F7F], dtype=np.uint16)
    np.testing.assert_array_equal(L.f64_to_bf16(L.bf16_to_f64(u)), u)
    assert L.bf16_to_f64(np.uint16(0x3F80)) == 1.0
    # round to nearest even: 1 + 2^-8 is halfway between 1 and 1 + 2^-7
    assert L.f64_to_bf16(1.0 + 2.0 ** -8) == 0x3F80
    assert L.f64_to_bf16(1.0 + 3 * 2.0 ** -8) == 0x3F82


def _weights(rng, d, f, hq, hkv, zero=False):
    z = (lambda *s: np.zeros(s)) if zero else (lambda *s: rng.standard_normal(s) * 0.05)
    return {"norm_in": 1 + 0.1 * rng.standard_normal(d), "w_qkv": z(d, (hq + 2 * hkv) * 128),
            "q_norm": 1 + 0.1 * rng.standard_normal(128), "k_norm": 1 + 0.1 * rng.standard_normal(128),
            "w_o": z(hq * 128, d), "norm_post": 1 + 0.1 * rng.standard_normal(d),
            "w_gate_up": z(d, 2 * f), "w_down": z(f, d)}


def test_layer_with_zero_projections_is_the_identity():
    rng = np.random.default_rng(3)
    d, f, hq, hkv, n = 64, 96, 2, 1, 5
    x = rng.standard_normal((n, d))
    w = _weights(rng, d, f, hq, hkv, zero=True)
    att = lambda q, k, v: rng.standard_normal((n, hq, 128))
    y = L.decoder_layer(x, w, att, np.arange(n), hq, hkv, THETA, 1e-6, rounded=False)
    np.testing.assert_allclose(y, x, atol=0, rtol=0)


def test_layer_residual_structure():
    # with W_o = 0 the attention does not reach x; with W_down = 0 the MLP does not
    rng = np.random.default_rng(4)
    d, f, hq, hkv, n = 64, 96, 2, 1, 5
    x = rng.standard_normal((n, d))
    w = _weights(rng, d, f, hq, hkv)
    out = rng.standard_normal((n, hq, 128))
    w_no_mlp = dict(w, w_down=np.zeros_like(w["w_down"]))
    y = L.decoder_layer(x, w_no_mlp, lambda q, k, v: out, np.arange(n), hq, hkv, THETA, 1e-6, rounded=False)
    np.testing.assert_allclose(y, x + out.reshape(n, -1) @ w["w_o"], rtol=1e-12)
    w_no_att = dict(w, w_o=np.zeros_like(w["w_o"]))
    y = L.decoder_layer(x, w_no_att, lambda q, k, v: out, np.arange(n), hq, hkv, THETA, 1e-6, rounded=False)
    h = L.rms_norm(x, w["norm_post"], 1e-6)
    np.testing.assert_allclose(y, x + L.silu_mul(h @ w["w_gate_up"], f) @ w["w_down"], rtol=1e-12)
