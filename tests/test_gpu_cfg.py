"""Classifier-free guidance on the GPU against the oracle: a guided step runs
every sample with its condition and with the zero condition on the same
active tokens (one batch of 2B samples) and stores v = v_u + s (v_c - v_u)
for the steps whose t_k lies in the CFG interval (Supp. Sec. D).

Tolerance: each prediction is within the step tolerance of the oracle's, so
the guided one is within |1 - s| e + s e = (2s - 1) e for s >= 1 (e the
per-prediction bound), plus one bf16 unit where both sides store it."""
import dataclasses

import numpy as np
import pytest
import torch

from gpu_helpers import (VEL_MAX_ABS, VEL_REL_L2, assert_clean, bf16_ulp, dev_f32, dev_i32, dev_u16, handle_for,
                         host_u16, max_abs)
from paper_2511_22533_gb300 import synth

pytestmark = pytest.mark.gpu

TINY = synth.SHAPES["tiny"]


def _step(h, c_S, k, quotas, hist):
    B, N = c_S.shape[0], c_S.shape[1]
    ring = np.zeros((3, B, N, 8), np.uint16)
    ring[(k - 1) % 3] = hist[2]
    ring[(k - 2) % 3] = hist[1]
    ring_d = dev_u16(ring)
    S_d = dev_f32(c_S)
    h.step(k, B, S_d, ring_d, dev_i32(quotas))
    torch.cuda.synchronize()
    assert_clean(h)
    return host_u16(ring_d)[k % 3], S_d.cpu().numpy()


def _oracle_step(orc, m, S, k, quota, hist_b, kv_c, kv_u, s, T):
    t = orc.time_schedule(T, 3.0)
    sc = orc.ssc_score(hist_b[2], hist_b[1], 0.7)
    cached, idx = orc.select(sc, int(quota))
    if len(idx):
        vc = m.forward(S, idx, float(t[k - 1]), kv_c)
        vu = m.forward(S, idx, float(t[k - 1]), kv_u)
        va = orc.cfg_combine(vc, vu, s)
    else:
        vc = vu = va = np.zeros((0, 8), np.float32)
    S_o, vt_o = orc.merge_euler(S, idx, va, hist_b[2], float(t[k - 1] - t[k]))
    return cached, idx, vc, vu, S_o, vt_o


def _guided_bound(vc, vu, s):
    e = (abs(1.0 - s) + s)
    return e * VEL_MAX_ABS, e * VEL_REL_L2 * max(np.linalg.norm(vc), np.linalg.norm(vu))


@pytest.mark.parametrize("s", [2.0, 5.0])
def test_cfg_step_teacher_forced_tiny(orc, s):
    B = 2
    h, blob, _ = handle_for(TINY, max_batch=B, cfg_strength=s, cfg_t_lo=0.0)
    m = orc.Model(TINY, blob)
    cond = synth.cond_tokens(TINY, B, 0)
    S = synth.latents(TINY, B, 0)
    h.set_cond(dev_u16(cond), B)
    kv_u = m.cond_kv(np.zeros_like(cond[0]))
    hist = synth.velocity_history(8, 8, B, seed=9)
    quotas = np.array([256, 0], np.int32)
    k = 4
    vt_gpu, S_gpu = _step(h, S, k, quotas, hist)
    for b in range(B):
        cached, idx, vc, vu, S_o, vt_o = _oracle_step(orc, m, S[b], k, quotas[b], hist[:, b], m.cond_kv(cond[b]),
                                                       kv_u, s, TINY.steps)
        cm = cached.astype(bool)
        np.testing.assert_array_equal(vt_gpu[b][cm], hist[2, b][cm])   # cached: bit for bit
        np.testing.assert_array_equal(S_gpu[b][cm], S_o[cm])
        got = synth.bf16_bits_to_f32(vt_gpu[b][idx])
        ref = synth.bf16_bits_to_f32(vt_o[idx])
        amax, l2 = _guided_bound(vc, vu, s)
        assert np.all(np.abs(got - ref) <= amax + bf16_ulp(np.maximum(np.abs(got), np.abs(ref)))), (b, max_abs(got, ref))
        assert np.linalg.norm(got.astype(np.float64) - ref) <= l2 + np.sqrt(got.size) * 2.0 ** -8 * np.abs(ref).max()
        # guidance moved the fresh velocities away from the conditional ones
        assert max_abs(ref, vc) > 1e-3
    h.close()


def test_cfg_zero_condition_and_empty_interval_are_unguided(orc):
    # with the zero condition both predictions coincide, so a guided step stores
    # exactly what an unguided one does; so does a step outside the interval
    B = 2
    hg, blob, _ = handle_for(TINY, max_batch=B, cfg_strength=5.0, cfg_t_lo=0.0)
    hn, _, _ = handle_for(TINY, max_batch=B)
    he, _, _ = handle_for(TINY, max_batch=B, cfg_strength=5.0, cfg_t_lo=1.5)
    S = synth.latents(TINY, B, 1)
    hist = synth.velocity_history(8, 8, B, seed=3)
    quotas = np.array([300, 100], np.int32)
    zero = np.zeros_like(synth.cond_tokens(TINY, B, 1))
    cond = synth.cond_tokens(TINY, B, 1)
    for h in (hg, hn):
        h.set_cond(dev_u16(zero), B)
    vg, Sg = _step(hg, S, 5, quotas, hist)
    vn, Sn = _step(hn, S, 5, quotas, hist)
    np.testing.assert_array_equal(vg, vn)
    np.testing.assert_array_equal(Sg, Sn)
    hn.set_cond(dev_u16(cond), B)
    he.set_cond(dev_u16(cond), B)
    ve, Se = _step(he, S, 5, quotas, hist)
    vn, Sn = _step(hn, S, 5, quotas, hist)
    np.testing.assert_array_equal(ve, vn)
    np.testing.assert_array_equal(Se, Sn)
    for h in (hg, hn, he):
        h.close()


def test_cfg_sample_tiny_against_oracle(orc):
    # Algorithm 1 with guidance over [0.5, 1]: both sides take the same
    # quotas; the free-running latents agree on the decoded occupancy
    B = 2
    s = 3.0
    h, blob, _ = handle_for(TINY, max_batch=B, cfg_strength=s, cfg_t_lo=0.5, tau=0)
    m = orc.Model(TINY, blob)
    cond = synth.cond_tokens(TINY, B, 0)
    S = synth.latents(TINY, B, 0)
    T = TINY.steps
    qs = np.zeros((T, B), np.int32)
    qs[2:] = 256
    S_d = dev_f32(S)
    qlog, _ = h.sample(S_d, dev_u16(cond), B, quota_schedule=qs)
    out = m.sample(S, cond, T=T, quota_schedule=qs, tau=0, cfg=s, cfg_t_lo=0.5)
    np.testing.assert_array_equal(qlog, out["quota"])
    plain = m.sample(S, cond, T=T, quota_schedule=qs, tau=0)
    offs, _ = synth.weight_offsets(TINY)
    off, dims = offs[("dec_w", -1)]
    dec = blob[off:off + dims[0] * dims[1]]
    S_gpu = S_d.cpu().numpy()
    for b in range(B):
        og, oo = orc.occupancy(S_gpu[b], dec), orc.occupancy(out["S"][b], dec)
        assert float(np.mean(og == oo)) >= 0.99
        # and the guidance changed the sample
        assert not np.array_equal(oo, orc.occupancy(plain["S"][b], dec))
    assert_clean(h)
    h.close()


def test_cfg_trellis_width_step(orc):
    # TRELLIS-L width (1024, 16 heads, 1374 condition tokens) with two blocks:
    # one guided step at 1229 active tokens
    shape = dataclasses.replace(synth.SHAPES["trellis_l"], blocks=2)
    s = 2.0
    h, blob, _ = handle_for(shape, max_batch=1, cfg_strength=s, cfg_t_lo=0.0)
    m = orc.Model(shape, blob)
    cond = synth.cond_tokens(shape, 1, 0)
    S = synth.latents(shape, 1, 0)
    h.set_cond(dev_u16(cond), 1)
    hist = synth.velocity_history(shape.grid, 8, 1, seed=4)
    q = np.array([shape.tokens - 1229], np.int32)
    k = 8
    vt_gpu, S_gpu = _step(h, S, k, q, hist)
    cached, idx, vc, vu, S_o, vt_o = _oracle_step(orc, m, S[0], k, q[0], hist[:, 0], m.cond_kv(cond[0]),
                                                   m.cond_kv(np.zeros_like(cond[0])), s, shape.steps)
    cm = cached.astype(bool)
    np.testing.assert_array_equal(vt_gpu[0][cm], hist[2, 0][cm])
    got = synth.bf16_bits_to_f32(vt_gpu[0][idx])
    ref = synth.bf16_bits_to_f32(vt_o[idx])
    amax, l2 = _guided_bound(vc, vu, s)
    assert np.all(np.abs(got - ref) <= amax + bf16_ulp(np.maximum(np.abs(got), np.abs(ref)))), max_abs(got, ref)
    h.close()
