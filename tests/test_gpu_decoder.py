"""The convolutional stand-in decoder on the GPU (Eq. 1 at the anchor step):
given the same latent grids, the dynamic-voxel count is exact -- the
decoder sums every output in one fixed fp32 order on both sides, so the
occupancy bits agree bit for bit."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_clean, dev_f32, dev_i32, dev_u16, handle_for
from paper_2511_22533_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("shape", [synth.SHAPES["tiny"], synth.ModelShape(16, 8, 128, 1, 4, 4, 64, 128, 8, 64)],
                         ids=["grid8", "grid16"])
def test_anchor_step_dynamic_voxels_exact(orc, shape):
    B = 2
    h, blob, _ = handle_for(shape, max_batch=B, decoder=1)
    m = orc.Model(shape, blob)
    cond = synth.cond_tokens(shape, B, 2)
    S = synth.latents(shape, B, 2)
    h.set_cond(dev_u16(cond), B)
    hist = synth.velocity_history(shape.grid, 8, B, seed=7)
    N = shape.tokens
    k = 3
    ring = np.zeros((3, B, N, 8), np.uint16)
    ring[(k - 1) % 3], ring[(k - 2) % 3] = hist[2], hist[1]
    S_d = dev_f32(S)
    dyn = torch.zeros(B, dtype=torch.int64, device="cuda")
    h.step(k, B, S_d, dev_u16(ring), dev_i32(np.array([N // 2, 0], np.int32)), dyn_voxels=dyn)
    torch.cuda.synchronize()
    assert_clean(h)
    S_after = S_d.cpu().numpy()
    got = dyn.cpu().numpy()
    for b in range(B):
        want = int(np.sum(m.decode_conv(S[b]) ^ m.decode_conv(S_after[b])))
        assert got[b] == want, (b, got[b], want)
        assert 0 < want < 64 * N
    h.close()


def test_sampler_sigma_with_conv_decoder(orc):
    # Algorithm 1 measuring sigma with the convolutional decoder: both sides
    # decode nearly the same latents at the anchor step
    shape = synth.SHAPES["tiny"]
    B = 2
    h, blob, _ = handle_for(shape, max_batch=B, decoder=1)
    m = orc.Model(shape, blob)
    cond = synth.cond_tokens(shape, B, 0)
    S = synth.latents(shape, B, 0)
    S_d = dev_f32(S)
    qlog, sigma = h.sample(S_d, dev_u16(cond), B)
    out = m.sample(S, cond, T=shape.steps, decoder=1)
    assert np.all(np.abs(sigma - out["sigma"]) <= 0.02 * np.maximum(out["sigma"], 50)), (sigma, out["sigma"])
    assert_clean(h)
    h.close()


@pytest.mark.parametrize("decoder", [0, 1])
def test_dynamic_voxel_curve_against_oracle(orc, decoder):
    # Eq. 1 at every step of an uncached run (the curve the PCSC slope is
    # fitted to): both sides decode nearly the same latents at every step
    shape = synth.SHAPES["tiny"]
    B = 2
    h, blob, _ = handle_for(shape, max_batch=B, decoder=decoder)
    m = orc.Model(shape, blob)
    cond = synth.cond_tokens(shape, B, 1)
    S = synth.latents(shape, B, 1)
    curve = h.dynamic_voxel_curve(dev_f32(S), dev_u16(cond), B)
    T = shape.steps
    out = m.sample(S, cond, T=T, quota_schedule=np.zeros((T, B), np.int32), tau=0, decoder=decoder, want_curve=True)
    ref = out["dyn"]
    assert curve.shape == (T, B) and np.all(curve >= 0)
    assert np.all(np.abs(curve - ref) <= 0.02 * np.maximum(ref, 50)), (curve, ref)
    assert_clean(h)
    h.close()
