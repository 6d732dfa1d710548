"""Parity of the whole cached step on the GPU against the oracle:
the flow transformer on active subsets (Sec. 4.2; Supp. Sec. F), one
teacher-forced cached step (Algorithm 1 steps 2-3: exact selection, cached
tokens bit for bit, fresh velocities within the bf16 tolerance), the
free-running sampler (final occupancy agreement >= 99.5% of voxels) and
full-size properties at the benchmark's TRELLIS-L configuration."""
import numpy as np
import pytest
import torch

from gpu_helpers import (VEL_MAX_ABS, VEL_REL_L2, assert_clean, dev_f32, dev_i32, dev_u16, handle_for, host_u16,
                         max_abs, rel_l2, stored_vel_excess)
from paper_2511_22533_gb300 import synth

pytestmark = pytest.mark.gpu

TINY = synth.SHAPES["tiny"]


def _dec_w(blob, shape):
    offs, _ = synth.weight_offsets(shape)
    off, dims = offs[("dec_w", -1)]
    return blob[off:off + dims[0] * dims[1]]


def _forward_gpu(h, t, S, lists):
    B, N = S.shape[0], S.shape[1]
    idx = np.zeros((B, N), np.int32)
    for b, l in enumerate(lists):
        idx[b, :len(l)] = l
    na = np.array([len(l) for l in lists], np.int32)
    v = torch.zeros((B, N, 8), dtype=torch.float32, device="cuda")
    h.forward(t, B, dev_f32(S), dev_i32(idx), dev_i32(na), v)
    torch.cuda.synchronize()
    out = v.cpu().numpy()
    return [out[b, :na[b]] for b in range(B)]


def _assert_vel(got, ref, what=""):
    """Computed (fp32) velocities against the oracle's."""
    assert np.isfinite(got).all(), what
    assert max_abs(got, ref) < VEL_MAX_ABS, (what, max_abs(got, ref))
    assert rel_l2(got, ref) < VEL_REL_L2, (what, rel_l2(got, ref))


def _assert_stored_vel(got, ref, what=""):
    """Velocities as both sides store them (bf16): the max-abs bound holds for
    the computed values, so the stored ones may differ by one more bf16 unit."""
    assert np.isfinite(got).all(), what
    assert stored_vel_excess(got, ref) < 0, (what, max_abs(got, ref), stored_vel_excess(got, ref))
    assert rel_l2(got, ref) < VEL_REL_L2, (what, rel_l2(got, ref))


class Ctx:
    def __init__(self, orc, shape, B, seed=0, **hyper):
        self.shape = shape
        self.h, self.blob, self.cfg = handle_for(shape, max_batch=B, seed=seed, **hyper)
        self.m = orc.Model(shape, self.blob)
        self.cond = synth.cond_tokens(shape, B, seed)
        self.S = synth.latents(shape, B, seed)
        self.kv = [self.m.cond_kv(self.cond[b]) for b in range(B)]
        self.h.set_cond(dev_u16(self.cond), B)


@pytest.fixture(scope="module")
def tiny(orc):
    c = Ctx(orc, TINY, 2)
    yield c
    c.h.close()


def test_forward_tiny_all_tokens(tiny):
    lists = [np.arange(512), np.arange(512)]
    got = _forward_gpu(tiny.h, 0.9, tiny.S, lists)
    for b in range(2):
        _assert_vel(got[b], tiny.m.forward(tiny.S[b], lists[b], 0.9, tiny.kv[b]), f"sample {b}")
    assert_clean(tiny.h)


def test_forward_tiny_ragged_subsets(tiny):
    g = np.random.default_rng(3)
    lists = [np.sort(g.choice(512, 200, replace=False)), np.sort(g.choice(512, 77, replace=False))]
    got = _forward_gpu(tiny.h, 0.6, tiny.S, lists)
    for b in range(2):
        _assert_vel(got[b], tiny.m.forward(tiny.S[b], lists[b], 0.6, tiny.kv[b]), f"sample {b}")


def test_forward_single_token_and_empty(tiny):
    lists = [np.array([511]), np.array([], np.int64)]
    got = _forward_gpu(tiny.h, 0.3, tiny.S, lists)
    _assert_vel(got[0], tiny.m.forward(tiny.S[0], lists[0], 0.3, tiny.kv[0]))
    assert got[1].shape == (0, 8)
    assert_clean(tiny.h)


def test_forward_deep_narrow(orc):
    # TRELLIS-L depth (24 blocks) at the tiny width: error accumulation over depth
    shape = synth.ModelShape(8, 8, 128, 24, 4, 4, 64, 128, 8, 64)
    c = Ctx(orc, shape, 1, seed=2)
    lists = [np.arange(512)]
    got = _forward_gpu(c.h, 0.7, c.S, lists)
    _assert_vel(got[0], c.m.forward(c.S[0], lists[0], 0.7, c.kv[0]))
    c.h.close()


def test_forward_trellis_width_two_blocks(orc):
    # TRELLIS-L width / heads / condition (W 1024, 16 heads, 1374 x 1024) with 2 blocks
    shape = synth.ModelShape(16, 8, 1024, 2, 16, 4, 1374, 1024, 25, 64)
    c = Ctx(orc, shape, 2, seed=4)
    g = np.random.default_rng(4)
    lists = [np.sort(g.choice(4096, 1229, replace=False)), np.arange(4096)]
    got = _forward_gpu(c.h, 0.85, c.S, lists)
    _assert_vel(got[0], c.m.forward(c.S[0], lists[0], 0.85, c.kv[0]), "1229 active")
    rows = np.arange(0, 4096, 16)
    ref1 = c.m.forward(c.S[1], lists[1], 0.85, c.kv[1])
    _assert_vel(got[1][rows], ref1[rows], "4096 active")
    assert_clean(c.h)
    c.h.close()


def test_forward_trellis_width_few_active(orc):
    # 300 and 77 active tokens at TRELLIS width: every projection (QKV with the
    # QK norm, out, cross-Q, cross-out, fc1 + GELU, fc2) runs few, narrow tiles
    shape = synth.ModelShape(16, 8, 1024, 1, 16, 4, 1374, 1024, 25, 64)
    c = Ctx(orc, shape, 2, seed=8)
    g = np.random.default_rng(8)
    lists = [np.sort(g.choice(4096, 300, replace=False)), np.sort(g.choice(4096, 77, replace=False))]
    got = _forward_gpu(c.h, 0.7, c.S, lists)
    for b in range(2):
        _assert_vel(got[b], c.m.forward(c.S[b], lists[b], 0.7, c.kv[b]), f"sample {b}")
    assert_clean(c.h)
    c.h.close()


def test_forward_ragged_batch8(orc):
    # batch 8 with ragged active counts in [400, 4096] (TRELLIS width, 1 block);
    # three samples are checked against the oracle, all eight run packed
    shape = synth.ModelShape(16, 8, 1024, 1, 16, 4, 1374, 1024, 25, 64)
    c = Ctx(orc, shape, 8, seed=5)
    counts = synth.ragged_active_targets(8, 4096, 400, 4096, seed=0)
    g = np.random.default_rng(5)
    lists = [np.sort(g.choice(4096, int(a), replace=False)) for a in counts]
    got = _forward_gpu(c.h, 0.5, c.S, lists)
    for b in (0, int(np.argmin(counts)), 7):
        _assert_vel(got[b], c.m.forward(c.S[b], lists[b], 0.5, c.kv[b]), f"sample {b} a={counts[b]}")
    assert_clean(c.h)
    c.h.close()


def test_forward_scaled_grid_subset(orc):
    # the 32^3 grid (32768 tokens): positions and gathers over the large grid
    shape = synth.ModelShape(32, 8, 128, 2, 4, 4, 64, 128, 50, 64)
    c = Ctx(orc, shape, 1, seed=6)
    g = np.random.default_rng(6)
    lists = [np.sort(g.choice(32768, 3000, replace=False))]
    got = _forward_gpu(c.h, 0.4, c.S, lists)
    _assert_vel(got[0], c.m.forward(c.S[0], lists[0], 0.4, c.kv[0]))
    c.h.close()


def _teacher_forced_step(orc, c, k, quotas, hist):
    """Runs f3dc_step k on (S, v^(k-1), v^(k-2)) = (c.S, hist[2], hist[1]) and
    the oracle on the same inputs; returns both sides."""
    B, N = c.S.shape[0], c.S.shape[1]
    ring = np.zeros((3, B, N, 8), np.uint16)
    ring[(k - 1) % 3] = hist[2]
    ring[(k - 2) % 3] = hist[1]
    ring_d = dev_u16(ring)
    S_d = dev_f32(c.S)
    c.h.step(k, B, S_d, ring_d, dev_i32(quotas))
    torch.cuda.synchronize()
    assert_clean(c.h)
    vt_gpu = host_u16(ring_d)[k % 3]
    S_gpu = S_d.cpu().numpy()
    t = orc.time_schedule(c.shape.steps, 3.0)
    res = []
    for b in range(B):
        s = orc.ssc_score(hist[2, b], hist[1, b], 0.7)
        cached, idx = orc.select(s, int(quotas[b]))
        va = c.m.forward(c.S[b], idx, float(t[k - 1]), c.kv[b]) if len(idx) else np.zeros((0, 8), np.float32)
        S_o, vt_o = orc.merge_euler(c.S[b], idx, va, hist[2, b], float(t[k - 1] - t[k]))
        res.append((cached, idx, S_o, vt_o))
    return vt_gpu, S_gpu, res


def test_step_teacher_forced_tiny(orc, tiny):
    hist = synth.velocity_history(8, 8, 2, seed=9)
    quotas = np.array([256, 300], np.int32)
    vt_gpu, S_gpu, res = _teacher_forced_step(orc, tiny, 4, quotas, hist)
    for b, (cached, idx, S_o, vt_o) in enumerate(res):
        cm = cached.astype(bool)
        # cached tokens reuse the stored velocity bit for bit, and their Euler
        # update is bit-exact with the oracle
        np.testing.assert_array_equal(vt_gpu[b][cm], hist[2, b][cm])
        np.testing.assert_array_equal(S_gpu[b][cm], S_o[cm])
        # exactly the selected tokens were recomputed
        fresh = np.any(vt_gpu[b] != hist[2, b], axis=1)
        assert not fresh[cm].any() and fresh[~cm].sum() >= (~cm).sum() - 2
        _assert_stored_vel(synth.bf16_bits_to_f32(vt_gpu[b][~cm]), synth.bf16_bits_to_f32(vt_o[~cm]), f"sample {b}")
        assert max_abs(S_gpu[b], S_o) < VEL_MAX_ABS


def test_step_quota_extremes(orc, tiny):
    hist = synth.velocity_history(8, 8, 2, seed=10)
    quotas = np.array([512, 0], np.int32)   # everything cached / nothing cached
    vt_gpu, S_gpu, res = _teacher_forced_step(orc, tiny, 6, quotas, hist)
    np.testing.assert_array_equal(vt_gpu[0], hist[2, 0])
    np.testing.assert_array_equal(S_gpu[0], res[0][2])
    _assert_stored_vel(synth.bf16_bits_to_f32(vt_gpu[1]), synth.bf16_bits_to_f32(res[1][3]))


def test_sample_tiny_free_running(orc):
    # tiny workload: T = 8, quota 50% (256 cached) from step 3, full before
    c = Ctx(orc, TINY, 2, tau=0)
    T = TINY.steps
    qs = np.zeros((T, 2), np.int32)
    qs[2:] = 256
    S_d = dev_f32(c.S)
    qlog, _ = c.h.sample(S_d, dev_u16(c.cond), 2, quota_schedule=qs)
    S_gpu = S_d.cpu().numpy()
    out = c.m.sample(c.S, c.cond, T=T, quota_schedule=qs, tau=0)
    np.testing.assert_array_equal(qlog, out["quota"])
    dec = _dec_w(c.blob, TINY)
    for b in range(2):
        og, oo = orc.occupancy(S_gpu[b], dec), orc.occupancy(out["S"][b], dec)
        agree = float(np.mean(og == oo))
        assert agree >= 0.995, agree
        # free-running, a near-tie in the score can cache a different token on
        # each side, so the latents drift apart a little beyond the per-step
        # velocity tolerance; the occupancy agreement above is the criterion
        assert rel_l2(S_gpu[b], out["S"][b]) < 5e-2
    assert_clean(c.h)
    c.h.close()


def test_sample_tiny_pcsc(orc):
    # Algorithm 1 with the PCSC budget; sigma fixed so both sides forecast the
    # same quotas, the measured dynamic voxels (Eq. 1) are reported and close
    c = Ctx(orc, TINY, 2)
    T = TINY.steps
    sig = np.array([6400.0, 12800.0])
    S_d = dev_f32(c.S)
    qlog, sigma = c.h.sample(S_d, dev_u16(c.cond), 2, sigma_override=sig)
    out = c.m.sample(c.S, c.cond, T=T, sigma_override=sig)
    np.testing.assert_array_equal(qlog, out["quota"])
    assert np.all(np.abs(sigma - out["sigma"]) <= 0.02 * np.maximum(out["sigma"], 50))
    dec = _dec_w(c.blob, TINY)
    S_gpu = S_d.cpu().numpy()
    for b in range(2):
        assert np.mean(orc.occupancy(S_gpu[b], dec) == orc.occupancy(out["S"][b], dec)) >= 0.995
    # measured-sigma path (host reads sigma back at the anchor step)
    S_d = dev_f32(c.S)
    qlog2, sigma2 = c.h.sample(S_d, dev_u16(c.cond), 2)
    out2 = c.m.sample(c.S, c.cond, T=T)
    assert np.all(np.abs(sigma2 - out2["sigma"]) <= 0.02 * np.maximum(out2["sigma"], 50))
    assert_clean(c.h)
    c.h.close()


@pytest.fixture(scope="module")
def trellis(orc):
    shape = synth.SHAPES["trellis_l"]
    h, blob, cfg = handle_for(shape, max_batch=1, seed=0)
    cond = synth.cond_tokens(shape, 1, 0)
    S = synth.latents(shape, 1, 0)
    h.set_cond(dev_u16(cond), 1)
    yield dict(h=h, blob=blob, S=S, cond=cond, shape=shape)
    h.close()


def test_full_size_step_properties(orc, trellis):
    # the benchmark's configuration (TRELLIS-L, 24 blocks, batch 1): one cached
    # step at the first Phase-2 quota of the benchmark's sigma (3141 cached)
    h, S = trellis["h"], trellis["S"]
    N, k = 4096, 6
    hist = synth.velocity_history(16, 8, 1, seed=12)
    ring = np.zeros((3, 1, N, 8), np.uint16)
    ring[(k - 1) % 3] = hist[2]
    ring[(k - 2) % 3] = hist[1]
    ring_d, S_d = dev_u16(ring), dev_f32(S)
    h.step(k, 1, S_d, ring_d, dev_i32([3141]))
    torch.cuda.synchronize()
    vt = host_u16(ring_d)[k % 3][0]
    S_gpu = S_d.cpu().numpy()[0]
    s = orc.ssc_score(hist[2, 0], hist[1, 0], 0.7)
    cached, idx = orc.select(s, 3141)
    cm = cached.astype(bool)
    np.testing.assert_array_equal(vt[cm], hist[2, 0][cm])
    # the fused step computes exactly what the separate forward computes
    t = orc.time_schedule(25, 3.0)
    vf = _forward_gpu(h, float(t[k - 1]), S, [idx])[0]
    vb = synth.f32_to_bf16_bits(vf)
    np.testing.assert_array_equal(vt[idx], vb)
    # and its Euler update is bit-exact with the oracle's given that velocity
    S_o, vt_o = orc.merge_euler(S[0], idx, synth.bf16_bits_to_f32(vb), hist[2, 0], float(t[k - 1] - t[k]))
    np.testing.assert_array_equal(vt, vt_o)
    np.testing.assert_array_equal(S_gpu, S_o)
    assert np.isfinite(vf).all() and 0.05 < np.std(vf) < 50
    assert_clean(h)


def test_full_size_sample_runs_and_logs(orc, trellis):
    # Algorithm 1 end to end at the benchmark's configuration with sigma 65536
    h, S, cond = trellis["h"], trellis["S"], trellis["cond"]
    S_d = dev_f32(S)
    qlog, sigma = h.sample(S_d, dev_u16(cond), 1, sigma_override=np.array([65536.0]))
    rows = [int(r) for r in open_golden_column()]
    assert qlog[:, 0].tolist() == rows
    assert np.isfinite(S_d.cpu().numpy()).all()
    assert sigma[0] >= 0
    assert_clean(h)


def open_golden_column():
    import os
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "phase_table_T25.txt")
    out = []
    for line in open(path):
        line = line.strip()
        if line and not line.startswith("#"):
            out.append(line.split()[3])
    return out


def test_sample_graph_replay_matches_eager(orc):
    # the sampler's CUDA-graph segments compute exactly what eager launches do,
    # on the first (capturing) call and on later replays
    c = Ctx(orc, TINY, 2)
    sig = np.array([6400.0, 9000.0])
    outs = []
    for graphs in (False, True, True):
        c.h.set_graphs(graphs)
        S_d = dev_f32(c.S)
        qlog, sigma = c.h.sample(S_d, dev_u16(c.cond), 2, sigma_override=sig)
        outs.append((S_d.cpu().numpy(), qlog, sigma))
    for S_g, q_g, s_g in outs[1:]:
        np.testing.assert_array_equal(S_g, outs[0][0])
        np.testing.assert_array_equal(q_g, outs[0][1])
        np.testing.assert_array_equal(s_g, outs[0][2])
    # the measured-sigma path splits the run at the anchor step
    res = []
    for graphs in (False, True):
        c.h.set_graphs(graphs)
        S_d = dev_f32(c.S)
        res.append((S_d,) + c.h.sample(S_d, dev_u16(c.cond), 2))
    np.testing.assert_array_equal(res[0][0].cpu().numpy(), res[1][0].cpu().numpy())
    np.testing.assert_array_equal(res[0][1], res[1][1])
    assert_clean(c.h)
    c.h.close()


def test_step_batch64_32cubed_merge(orc):
    # the largest step workload of the merge / Euler kernel: 64 samples of the
    # 32^3 grid (32768 tokens each, half cached), a one-block width-128 model;
    # selection, cached velocities and the Euler update of every token are
    # bit-exact with the oracle given the velocities the step stored
    shape = synth.ModelShape(32, 8, 128, 1, 4, 4, 64, 128, 50, 64)
    B, N, k = 64, shape.tokens, 8
    h, blob, _ = handle_for(shape, max_batch=B, seed=9)
    cond = synth.cond_tokens(shape, 1, 9)
    h.set_cond(dev_u16(np.ascontiguousarray(np.broadcast_to(cond, (B,) + cond.shape[1:]))), B)
    hist = synth.velocity_history(32, 8, B, seed=33)
    ring = np.zeros((3, B, N, 8), np.uint16)
    ring[(k - 1) % 3], ring[(k - 2) % 3] = hist[2], hist[1]
    S = synth.latents(shape, B, 9)
    quotas = np.full(B, N // 2, np.int32)
    ring_d, S_d = dev_u16(ring), dev_f32(S)
    h.step(k, B, S_d, ring_d, dev_i32(quotas))
    torch.cuda.synchronize()
    assert_clean(h)
    vt = host_u16(ring_d)[k % 3]
    S_gpu = S_d.cpu().numpy()
    t = orc.time_schedule(shape.steps, 3.0)
    for b in (0, 17, 63):
        cached, idx = orc.select(orc.ssc_score(hist[2, b], hist[1, b], 0.7), N // 2)
        cm = cached.astype(bool)
        np.testing.assert_array_equal(vt[b][cm], hist[2, b][cm])
        S_o, vt_o = orc.merge_euler(S[b], idx, synth.bf16_bits_to_f32(vt[b][idx]), hist[2, b],
                                    float(t[k - 1] - t[k]))
        np.testing.assert_array_equal(vt[b], vt_o)
        np.testing.assert_array_equal(S_gpu[b], S_o)
        assert np.isfinite(synth.bf16_bits_to_f32(vt[b])).all()
    h.close()
