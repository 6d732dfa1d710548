"""Oracle pins for classifier-free guidance (CFG) in the sampler: the CFG
interval t in [t_lo, 1] of the flow sampler (Supp. Sec. D; Phase 3 of
Algorithm 1 is the CFG-free stage) and the guided velocity
v = v_u + s (v_c - v_u), with the unconditional prediction made for the
all-zero condition on the same active tokens (a reading)."""
import os

import numpy as np
import pytest

from paper_2511_22533_gb300 import synth

TINY = synth.SHAPES["tiny"]
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "schedule_turning_points.txt")


def _turning_points():
    rows = []
    for line in open(GOLDEN):
        if line.strip() and not line.startswith("#"):
            T, eta, k0 = line.split()
            rows.append((int(T), float(eta), int(k0)))
    return rows


def test_cfg_interval_matches_the_printed_turning_points(orc):
    # Supp. Sec. D: CFG acts for t in [0.5, 1]; the first 0-based step k0 with
    # t < 0.5 is printed for eta = 1, 2 (and follows for 3): 1-based steps
    # 1..k0 are guided, k0 + 1..T are not
    for T, eta, k0 in _turning_points():
        on = [orc.cfg_on(T, eta, 0.5, k) for k in range(1, T + 1)]
        assert on == [k <= k0 for k in range(1, T + 1)], (T, eta)


def test_cfg_interval_edges(orc):
    assert all(orc.cfg_on(25, 3.0, 0.0, k) for k in range(1, 26))      # t in [0, 1]: every step
    assert not any(orc.cfg_on(25, 3.0, 1.5, k) for k in range(1, 26))  # empty interval
    assert orc.cfg_on(25, 3.0, 1.0, 1) and not orc.cfg_on(25, 3.0, 1.0, 2)  # t_1 = 1 exactly


def test_cfg_combine_endpoints_and_affinity(orc):
    # s = 0 is the unconditional prediction exactly, s = 1 the conditional one
    # (to one rounding of the difference), and the result is affine in s
    rng = np.random.default_rng(0)
    vc = rng.standard_normal(4096).astype(np.float32)
    vu = rng.standard_normal(4096).astype(np.float32)
    np.testing.assert_array_equal(orc.cfg_combine(vc, vu, 0.0), vu)
    v1 = orc.cfg_combine(vc, vu, 1.0)
    ulp = np.spacing(np.maximum(np.abs(vc), np.abs(vu)).astype(np.float32)) * 2
    assert np.all(np.abs(v1 - vc) <= ulp)
    s = np.array([0.5, 2.0, 3.0, 7.5])
    vs = np.stack([orc.cfg_combine(vc, vu, x) for x in s])
    slope = (vs - vu) / s[:, None]
    assert np.allclose(slope, (vc - vu)[None, :], rtol=1e-5, atol=1e-5)
    # guidance pushes past the conditional prediction for s > 1
    d = vc - vu
    big = np.abs(d) > 1e-2
    assert np.all(np.sign(vs[1][big] - vc[big]) == np.sign(d[big]))


@pytest.fixture(scope="module")
def tiny(orc):
    blob = synth.weights_blob(TINY, 0)
    m = orc.Model(TINY, blob)
    cond = synth.cond_tokens(TINY, 1, 0)
    S = synth.latents(TINY, 1, 0)
    return dict(model=m, cond=cond, S=S)


def _quotas(T):
    q = np.zeros((T, 1), np.int32)
    q[2:] = 256
    return q


def test_cfg_strength_zero_is_the_unconditional_sampler(tiny):
    # s = 0 guides every step onto the zero-condition prediction: the sampler
    # is then bit for bit the unguided sampler run with the zero condition
    m, S, cond = tiny["model"], tiny["S"], tiny["cond"]
    T, q = TINY.steps, _quotas(TINY.steps)
    g = m.sample(S, cond, T=T, quota_schedule=q, tau=0, cfg=0.0, cfg_t_lo=0.0)
    u = m.sample(S, np.zeros_like(cond), T=T, quota_schedule=q, tau=0)
    np.testing.assert_array_equal(g["S"], u["S"])
    np.testing.assert_array_equal(g["v_hist"], u["v_hist"])


def test_cfg_with_zero_condition_is_unguided(tiny):
    # when the condition is the zero condition both predictions agree bit for
    # bit, so any strength leaves the sampler unchanged
    m, S, cond = tiny["model"], tiny["S"], tiny["cond"]
    T, q = TINY.steps, _quotas(TINY.steps)
    z = np.zeros_like(cond)
    g = m.sample(S, z, T=T, quota_schedule=q, tau=0, cfg=5.0, cfg_t_lo=0.0)
    u = m.sample(S, z, T=T, quota_schedule=q, tau=0)
    np.testing.assert_array_equal(g["S"], u["S"])


def test_cfg_outside_the_interval_and_strength_one(tiny):
    # an empty interval is the unguided sampler bit for bit; s = 1 tracks the
    # conditional sampler up to the rounding of v_u + (v_c - v_u); a real
    # strength changes the result
    m, S, cond = tiny["model"], tiny["S"], tiny["cond"]
    T, q = TINY.steps, _quotas(TINY.steps)
    base = m.sample(S, cond, T=T, quota_schedule=q, tau=0)
    none = m.sample(S, cond, T=T, quota_schedule=q, tau=0, cfg=5.0, cfg_t_lo=1.5)
    np.testing.assert_array_equal(none["S"], base["S"])
    one = m.sample(S, cond, T=T, quota_schedule=q, tau=0, cfg=1.0, cfg_t_lo=0.0)
    assert np.max(np.abs(one["S"] - base["S"])) < 0.05 * np.max(np.abs(base["S"]))
    five = m.sample(S, cond, T=T, quota_schedule=q, tau=0, cfg=5.0, cfg_t_lo=0.0)
    assert np.max(np.abs(five["S"] - base["S"])) > 1e-3
    # guiding only the steps in [0.5, 1] sits between the two
    half = m.sample(S, cond, T=T, quota_schedule=q, tau=0, cfg=5.0, cfg_t_lo=0.5)
    assert not np.array_equal(half["S"], base["S"]) and not np.array_equal(half["S"], five["S"])
