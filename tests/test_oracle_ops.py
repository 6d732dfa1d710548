"""Oracle pins for the dense ops, the merge / Euler update (Alg. 1 step 3)
and the dynamic-voxel count (Sec. 4.1 Eq. 1)."""
import math

import numpy as np
import pytest
from scipy.special import softmax

from paper_2511_22533_gb300 import synth


def test_linear_matches_library_matmul(orc):
    rng = np.random.default_rng(0)
    x = rng.standard_normal((37, 70)).astype(np.float32)
    w = rng.standard_normal((23, 70)).astype(np.float32)
    b = rng.standard_normal(23).astype(np.float32)
    y = orc.linear(x, w, b)
    ref = x.astype(np.float64) @ w.astype(np.float64).T + b
    np.testing.assert_allclose(y, ref, rtol=1e-6, atol=1e-5)
    y0 = orc.linear(x, w)
    np.testing.assert_allclose(y0, x.astype(np.float64) @ w.astype(np.float64).T, rtol=1e-6, atol=1e-5)


def test_layernorm_moments(orc):
    rng = np.random.default_rng(1)
    x = (3.0 + 5.0 * rng.standard_normal((16, 1024))).astype(np.float32)
    y = orc.layernorm(x).astype(np.float64)
    np.testing.assert_allclose(y.mean(1), 0.0, atol=1e-6)
    np.testing.assert_allclose(y.var(1), 1.0, rtol=1e-5)
    # a constant row normalises to exactly zero
    z = orc.layernorm(np.full((2, 64), 7.0, np.float32))
    assert np.all(z == 0.0)


def test_attention_single_key_returns_its_value(orc):
    rng = np.random.default_rng(2)
    q = rng.standard_normal((5, 64)).astype(np.float32)
    k = rng.standard_normal((1, 64)).astype(np.float32)
    v = rng.standard_normal((1, 64)).astype(np.float32)
    out = orc.attention(q, k, v, heads=2)
    np.testing.assert_allclose(out, np.repeat(v, 5, 0), rtol=1e-6, atol=1e-6)


def test_attention_probabilities_match_softmax(orc):
    # values = one-hot rows, so each output row IS the attention distribution
    rng = np.random.default_rng(3)
    H, dh, nk = 2, 16, 16
    q = rng.standard_normal((7, H * dh)).astype(np.float32)
    k = rng.standard_normal((nk, H * dh)).astype(np.float32)
    v = np.zeros((nk, H * dh), np.float32)
    for h in range(H):
        v[:, h * dh:(h + 1) * dh] = np.eye(nk, dh)
    out = orc.attention(q, k, v, heads=H)
    for h in range(H):
        logits = q[:, h * dh:(h + 1) * dh].astype(np.float64) @ k[:, h * dh:(h + 1) * dh].T.astype(np.float64)
        p = softmax(logits / math.sqrt(dh), axis=1)
        np.testing.assert_allclose(out[:, h * dh:(h + 1) * dh], p, rtol=1e-5, atol=1e-7)
        np.testing.assert_allclose(out[:, h * dh:(h + 1) * dh].sum(1), 1.0, rtol=1e-6)


def test_attention_identical_keys_average_values(orc):
    rng = np.random.default_rng(4)
    q = rng.standard_normal((3, 32)).astype(np.float32)
    k = np.repeat(rng.standard_normal((1, 32)).astype(np.float32), 9, 0)
    v = rng.standard_normal((9, 32)).astype(np.float32)
    out = orc.attention(q, k, v, heads=1)
    np.testing.assert_allclose(out, np.repeat(v.mean(0, keepdims=True), 3, 0), rtol=1e-5, atol=1e-6)


def test_gelu_against_erf_form(orc):
    # the tanh form stays within 1e-3 of the exact erf GELU
    for x in np.linspace(-6, 6, 121):
        exact = 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0)))
        assert abs(orc.gelu(float(x)) - exact) < 1e-3
    assert orc.gelu(0.0) == 0.0
    assert abs(orc.gelu(10.0) - 10.0) < 1e-6 and abs(orc.gelu(-10.0)) < 1e-6


def test_pos_embed_coordinates(orc):
    W, g = 128, 8
    F = W // 6
    # token (d, h, w) = (3, 5, 6)
    i = (3 * g + 5) * g + 6
    pe = orc.pos_embed(g, W, i)
    for a, coord in enumerate((3, 5, 6)):
        for f in (0, 1, F - 1):
            w = 10000.0 ** (-f / F)
            assert pe[a * 2 * F + f] == pytest.approx(math.sin(coord * w), abs=1e-6)
            assert pe[a * 2 * F + F + f] == pytest.approx(math.cos(coord * w), abs=1e-6)
    assert np.all(pe[6 * F:] == 0.0)


def test_merge_euler_semantics(orc):
    rng = np.random.default_rng(5)
    N, C = 40, 8
    S = rng.standard_normal((N, C)).astype(np.float32)
    vc = synth.f32_to_bf16_bits(rng.standard_normal((N, C)))
    idx = np.array([3, 9, 21], np.int32)
    va = np.zeros((3, C), np.float32)
    va[0] = 2.0
    va[1] = 1.0 + 2.0 ** -8           # halfway between bf16 1 and 1 + 2^-7: ties to even (1.0)
    va[2] = 1.0 + 3 * 2.0 ** -9       # above halfway: rounds up to 1 + 2^-7
    S2, vt = orc.merge_euler(S, idx, va, vc, 0.5)
    cached = np.setdiff1d(np.arange(N), idx)
    # cached tokens carry their stored velocity bit for bit
    np.testing.assert_array_equal(vt[cached], vc[cached])
    f = synth.bf16_bits_to_f32(vt)
    assert np.all(f[3] == 2.0) and np.all(f[9] == 1.0) and np.all(f[21] == 1.0 + 2.0 ** -7)
    # S <- S - dt v in fp32: dt * 2 = 1 exactly
    np.testing.assert_array_equal(S2[3], (S[3] - np.float32(1.0)).astype(np.float32))
    np.testing.assert_array_equal(S2[cached], (S[cached] - np.float32(0.5) * f[cached]).astype(np.float32))


def test_merge_with_everything_cached_moves_by_stored_velocity(orc):
    rng = np.random.default_rng(6)
    S = rng.standard_normal((10, 8)).astype(np.float32)
    vc = synth.f32_to_bf16_bits(rng.standard_normal((10, 8)))
    S2, vt = orc.merge_euler(S, np.zeros(0, np.int32), np.zeros((0, 8), np.float32), vc, 0.25)
    np.testing.assert_array_equal(vt, vc)
    np.testing.assert_array_equal(S2, S - np.float32(0.25) * synth.bf16_bits_to_f32(vc))


def test_dynamic_voxels_invariants(orc):
    rng = np.random.default_rng(7)
    S = rng.standard_normal((64, 8)).astype(np.float32)
    dec = synth.f32_to_bf16_bits(rng.standard_normal((8, 64)))
    o = orc.occupancy(S, dec)
    assert orc.dynamic_voxels(o, o) == 0
    # negating the latent negates every logit: every nonzero logit flips
    on = orc.occupancy(-S, dec)
    logits = S.astype(np.float64) @ synth.bf16_bits_to_f32(dec).reshape(8, 64).astype(np.float64)
    assert orc.dynamic_voxels(o, on) == int(np.count_nonzero(logits))
    # occupancy agrees with the fp64 logit sign wherever the logit is not tiny
    sure = np.abs(logits) > 1e-4
    np.testing.assert_array_equal(o[sure], (logits > 0)[sure])


def test_dynamic_voxels_brute_force(orc):
    rng = np.random.default_rng(8)
    a = rng.integers(0, 2, 1000).astype(np.uint8)
    b = rng.integers(0, 2, 1000).astype(np.uint8)
    assert orc.dynamic_voxels(a, b) == sum(int(x != y) for x, y in zip(a, b))
