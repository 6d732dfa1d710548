"""Oracle pins for the convolutional stand-in decoder of Eq. 1's grids
(3x3x3 convolutions with zero padding and ReLU, C -> 16 at D^3, nearest 2x
upsampling, 16 -> 8 at (2D)^3, 2x, 8 -> 1 at (4D)^3; occupied iff logit > 0),
checked against closed forms on hand-set weights."""
import numpy as np

from paper_2511_22533_gb300 import synth

TINY = synth.SHAPES["tiny"]
D = TINY.grid
CENTER = 13  # tap (0, 0, 0): 9 (dz + 1) + 3 (dy + 1) + (dx + 1)


def _blob_with(**conv):
    blob = synth.weights_blob(TINY, 0)
    for name in ("dc1_w", "dc1_b", "dc2_w", "dc2_b", "dc3_w", "dc3_b"):
        synth.set_weight(blob, TINY, name, -1, conv.get(name, 0.0))
    return blob


def _pass_through(c_in, c_out, tap=CENTER, channels=None):
    """[c_out, c_in * 27] weights with w[c, c * 27 + tap] = 1 for c < min(c_in, c_out)."""
    w = np.zeros((c_out, c_in * 27), np.float32)
    for c in range(min(c_in, c_out) if channels is None else channels):
        w[c, c * 27 + tap] = 1.0
    return w


def _grid4(S):
    """Token values on the (4D)^3 grid by nearest upsampling, index (z, y, x)."""
    g = S.reshape(D, D, D, -1)
    return g.repeat(4, 0).repeat(4, 1).repeat(4, 2)


def test_constant_logit(orc):
    S = synth.latents(TINY, 1, 0)[0]
    for b, want in ((0.5, 1), (-0.5, 0)):
        m = orc.Model(TINY, _blob_with(dc3_b=b))
        occ = m.decode_conv(S)
        assert occ.shape == (64 * D ** 3,) and np.all(occ == want)


def test_pointwise_path_is_relu_of_the_latent_upsampled(orc):
    # centre taps pass channel c through every layer: the logit at sub-voxel
    # (z, y, x) is ReLU(S_0) of token (z/4, y/4, x/4) minus 0.25
    S = synth.latents(TINY, 1, 1)[0]
    w3 = np.zeros((1, 8 * 27), np.float32)
    w3[0, CENTER] = 1.0
    m = orc.Model(TINY, _blob_with(dc1_w=_pass_through(8, 16), dc2_w=_pass_through(16, 8), dc3_w=w3, dc3_b=-0.25))
    occ = m.decode_conv(S).reshape(4 * D, 4 * D, 4 * D)
    want = (np.maximum(_grid4(S)[..., 0], 0) - np.float32(0.25) > 0)
    np.testing.assert_array_equal(occ, want.astype(np.uint8))
    assert 0.05 < occ.mean() < 0.6


def test_off_centre_tap_shifts_the_grid(orc):
    # the last layer reads tap (dz, dy, dx) = (0, 0, +1): the logit at x is the
    # input at x + 1, and 0 beyond the far face (zero padding)
    S = synth.latents(TINY, 1, 2)[0]
    w3 = np.zeros((1, 8 * 27), np.float32)
    w3[0, 9 * 1 + 3 * 1 + 2] = 1.0
    m = orc.Model(TINY, _blob_with(dc1_w=_pass_through(8, 16), dc2_w=_pass_through(16, 8), dc3_w=w3, dc3_b=-0.25))
    occ = m.decode_conv(S).reshape(4 * D, 4 * D, 4 * D)
    g = np.maximum(_grid4(S)[..., 0], 0)
    shifted = np.zeros_like(g)
    shifted[:, :, :-1] = g[:, :, 1:]
    np.testing.assert_array_equal(occ, (shifted - np.float32(0.25) > 0).astype(np.uint8))
    assert not occ[:, :, -1].any()


def test_relu_clips_negative_channels(orc):
    # a negated pass-through in layer 1 leaves ReLU(-S): layer 3 with weight +1
    # and bias -0.25 then marks where S_0 < -0.25
    S = synth.latents(TINY, 1, 3)[0]
    w1 = -_pass_through(8, 16)
    w3 = np.zeros((1, 8 * 27), np.float32)
    w3[0, CENTER] = 1.0
    m = orc.Model(TINY, _blob_with(dc1_w=w1, dc2_w=_pass_through(16, 8), dc3_w=w3, dc3_b=-0.25))
    occ = m.decode_conv(S).reshape(4 * D, 4 * D, 4 * D)
    np.testing.assert_array_equal(occ, (np.maximum(-_grid4(S)[..., 0], 0) - np.float32(0.25) > 0).astype(np.uint8))


def test_sampler_measures_sigma_with_the_conv_decoder(orc):
    blob = synth.weights_blob(TINY, 0)
    m = orc.Model(TINY, blob)
    S = synth.latents(TINY, 1, 0)
    cond = synth.cond_tokens(TINY, 1, 0)
    out = m.sample(S, cond, T=TINY.steps, decoder=1)
    lin = m.sample(S, cond, T=TINY.steps, decoder=0)
    assert 0 < out["sigma"][0] < 64 * D ** 3 and out["sigma"][0] != lin["sigma"][0]
