"""SSC with three predictions on the GPU: the acceleration term is the second
difference of the velocity over the history ring's three slots (v(t-3) sits
in the slot the step overwrites).  Selection is compared exactly (the set of
recomputed tokens), fresh velocities within the step tolerance."""
import numpy as np
import pytest
import torch

from gpu_helpers import (VEL_REL_L2, assert_clean, dev_f32, dev_i32, dev_u16, handle_for, host_u16,
                         rel_l2, stored_vel_excess)
from paper_2511_22533_gb300 import synth

pytestmark = pytest.mark.gpu

TINY = synth.SHAPES["tiny"]


def _step3(orc, shape, B, k, quotas, seed, sample_rows=None):
    h, blob, _ = handle_for(shape, max_batch=B, seed=seed, ssc_accel=1)
    m = orc.Model(shape, blob)
    cond = synth.cond_tokens(shape, B, seed)
    S = synth.latents(shape, B, seed)
    h.set_cond(dev_u16(cond), B)
    hist = synth.velocity_history(shape.grid, 8, B, seed=seed + 1)
    N = shape.tokens
    ring = np.zeros((3, B, N, 8), np.uint16)
    ring[(k - 1) % 3], ring[(k - 2) % 3], ring[k % 3] = hist[2], hist[1], hist[0]
    ring_d = dev_u16(ring)
    S_d = dev_f32(S)
    h.step(k, B, S_d, ring_d, dev_i32(quotas))
    torch.cuda.synchronize()
    assert_clean(h)
    vt = host_u16(ring_d)[k % 3]
    t = orc.time_schedule(shape.steps, 3.0)
    for b in range(B):
        sc = orc.ssc_score3(hist[2, b], hist[1, b], hist[0, b], 0.7)
        cached, idx = orc.select(sc, int(quotas[b]))
        cm = cached.astype(bool)
        np.testing.assert_array_equal(vt[b][cm], hist[2, b][cm])
        fresh = np.any(vt[b] != hist[2, b], axis=1)
        assert not fresh[cm].any() and fresh[~cm].sum() >= (~cm).sum() - 2
        # the first-difference score would have chosen another set
        _, idx1 = orc.select(orc.ssc_score(hist[2, b], hist[1, b], 0.7), int(quotas[b]))
        assert not np.array_equal(idx, idx1)
        rows = idx if sample_rows is None else idx[::sample_rows]
        kv = m.cond_kv(cond[b])
        va = m.forward(S[b], idx, float(t[k - 1]), kv)
        sel = np.searchsorted(idx, rows)
        got = synth.bf16_bits_to_f32(vt[b][rows])
        ref = synth.bf16_bits_to_f32(orc.merge_euler(S[b], idx, va, hist[2, b], float(t[k - 1] - t[k]))[1][rows])
        assert stored_vel_excess(got, ref) < 0, (b, np.max(np.abs(got - ref)))
        assert rel_l2(got, ref) < VEL_REL_L2
    h.close()


def test_ssc3_step_tiny(orc):
    _step3(orc, TINY, 2, 5, np.array([256, 400], np.int32), seed=3)


def test_ssc3_step_32cubed_grid(orc):
    # 32768 tokens: tokens beyond each thread's first four take the
    # selection kernel's re-read path
    shape = synth.ModelShape(32, 8, 128, 1, 4, 4, 64, 128, 8, 64)
    _step3(orc, shape, 1, 6, np.array([32768 - 3000], np.int32), seed=5, sample_rows=7)


def test_ssc3_sampler_tiny(orc):
    B = 2
    h, blob, _ = handle_for(TINY, max_batch=B, tau=0, ssc_accel=1)
    m = orc.Model(TINY, blob)
    cond = synth.cond_tokens(TINY, B, 0)
    S = synth.latents(TINY, B, 0)
    T = TINY.steps
    qs = np.zeros((T, B), np.int32)
    qs[2:] = 256
    S_d = dev_f32(S)
    qlog, _ = h.sample(S_d, dev_u16(cond), B, quota_schedule=qs)
    out = m.sample(S, cond, T=T, quota_schedule=qs, tau=0, ssc_accel=1)
    np.testing.assert_array_equal(qlog, out["quota"])
    offs, _ = synth.weight_offsets(TINY)
    off, dims = offs[("dec_w", -1)]
    dec = blob[off:off + dims[0] * dims[1]]
    S_gpu = S_d.cpu().numpy()
    for b in range(B):
        assert float(np.mean(orc.occupancy(S_gpu[b], dec) == orc.occupancy(out["S"][b], dec))) >= 0.995
    assert_clean(h)
    h.close()
