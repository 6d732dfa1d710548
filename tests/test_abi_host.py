"""libf3dc.so loads without a GPU, exports every symbol include/f3dc.h
declares, and its host-only schedule logic (Supp. Sec. D; Sec. 4.2 PCSC;
Algorithm 1 phases and tau rule) agrees exactly with the oracle."""
import ctypes as C

import numpy as np
import pytest

from paper_2511_22533_gb300 import f3dc, synth


@pytest.fixture(scope="module")
def L():
    return f3dc.lib()


def test_exports_every_declared_symbol(L):
    names = f3dc.declared_symbols()
    assert len(names) >= 15
    for n in names:
        assert hasattr(L, n), n


def test_weights_elems_matches_layout():
    for name, shape in synth.SHAPES.items():
        cfg = f3dc.config_for(shape)
        _, total = synth.weight_offsets(shape)
        assert f3dc.weights_elems(cfg) == total, name


def test_time_schedule_matches_oracle(orc):
    for eta, T in [(3.0, 25), (2.0, 25), (1.0, 8), (3.0, 50)]:
        cfg = f3dc.config_for(synth.SHAPES["trellis_l"], steps=T, eta=eta)
        np.testing.assert_array_equal(f3dc.time_schedule(cfg), orc.time_schedule(T, eta))


@pytest.mark.parametrize("tau,mode", [(3, 0), (5, 0), (8, 0), (1, 0), (0, 0), (3, 1)])
def test_pcsc_quota_matches_oracle(orc, tau, mode):
    rng = np.random.default_rng(tau * 10 + mode)
    shape = synth.SHAPES["trellis_l"]
    for sigma in [0.0, 1.0, 6400.0, 65536.0, 2.6e5, 1e9] + list(rng.uniform(0, 3e5, 6)):
        cfg = f3dc.config_for(shape, tau=tau, refresh_mode=mode)
        consec = np.zeros(1, np.int32)
        gate = orc.TauGate(tau, mode)
        for k in range(1, 26):
            q, ph = f3dc.pcsc_quota(cfg, sigma, k, consec)
            oq, oph = orc.phase_quota(4096, 25, 0.2, 0.75, -0.07, 0.7, 3, 64, sigma, k)
            assert (q, ph) == (gate(oq), oph), (sigma, k)


def test_pcsc_quota_other_hyperparameters(orc):
    shape = synth.SHAPES["scaled"]
    for mu, xi, fc in [(-0.169, 0.8, 2), (-0.7, 0.9, 0), (-0.007, 0.7, 1)]:
        cfg = f3dc.config_for(shape, mu=mu, xi=xi, f_corr=fc)
        for k in range(1, 51):
            q, ph = f3dc.pcsc_quota(cfg, 3.0e6, k)
            assert (q, ph) == orc.phase_quota(32768, 50, 0.2, 0.75, mu, xi, fc, 64, 3.0e6, k)


def test_invalid_arguments_are_reported(L):
    cfg = f3dc.config_for(synth.SHAPES["trellis_l"])
    with pytest.raises(f3dc.F3dcError) as e:
        f3dc.pcsc_quota(cfg, 10.0, 0)
    assert e.value.status == 1
    with pytest.raises(f3dc.F3dcError) as e:
        f3dc.pcsc_quota(cfg, float("nan"), 3)
    assert e.value.status == 6
    bad = f3dc.config_for(synth.SHAPES["trellis_l"], heads=7)
    assert f3dc.weights_elems(bad) == 0
    with pytest.raises(f3dc.F3dcError):
        f3dc.time_schedule(bad)
    bad = f3dc.config_for(synth.SHAPES["trellis_l"], channels=4)
    assert f3dc.weights_elems(bad) == 0
    # create rejects a bad config before touching any device
    h = C.c_void_p()
    st = L.f3dc_create(C.byref(bad), None, None, C.byref(h))
    assert st == 1 and not h
    assert b"channels" in L.f3dc_last_error(None)


def test_fit_mu_matches_oracle(orc):
    # the library's data-driven slope fit (host only) and the oracle's, on
    # log-linear curves with noise, gross outliers, zero counts and hopeless
    # instances
    rng = np.random.default_rng(3)
    T = 25
    k = np.arange(1, T + 1, dtype=np.float64)
    curves = []
    for i in range(40):
        slope = rng.uniform(-0.3, -0.01)
        y = rng.uniform(6, 11) + slope * (k - 8) + rng.normal(0, rng.choice([0.005, 0.05, 1.0]), T)
        d = np.exp(y)
        for _ in range(rng.integers(0, 3)):
            d[rng.integers(7, 18)] *= np.exp(rng.choice([-3.0, 2.5]))
        if i % 7 == 0:
            d[rng.integers(7, 18)] = 0.0
        curves.append(np.round(d))
    curves = np.stack(curves)
    for tol, frac in ((0.1, 0.6), (0.05, 0.8), (0.3, 0.5)):
        mu_l, sl_l, kept_l = f3dc.fit_mu(curves, tol=tol, min_frac=frac)
        mu_o, sl_o, kept_o = orc.fit_mu(curves, tol=tol, min_frac=frac)
        np.testing.assert_array_equal(kept_l, kept_o)
        np.testing.assert_allclose(sl_l, sl_o, rtol=0, atol=1e-12)
        assert abs(mu_l - mu_o) < 1e-12
        assert 0 < kept_l.sum() < len(curves)


@pytest.mark.parametrize("field,value,needle", [
    ("cfg_strength", -1.0, b"cfg_strength"),
    ("cfg_strength", float("inf"), b"cfg_strength"),
    ("ssc_accel", 2, b"ssc_accel"),
    ("decoder", 3, b"decoder"),
    ("width", 384, b"width"),
])
def test_new_config_fields_are_validated(L, field, value, needle):
    bad = f3dc.config_for(synth.SHAPES["tiny"], **{field: value})
    assert f3dc.weights_elems(bad) == 0
    h = C.c_void_p()
    assert L.f3dc_create(C.byref(bad), None, None, C.byref(h)) == 1 and not h
    assert needle in L.f3dc_last_error(None)


def test_guidance_and_decoder_constraints(L):
    # guidance runs 2B samples in one plan (B <= 32); the convolutional
    # decoder yields 64 sub-voxels per token
    ok = f3dc.config_for(synth.SHAPES["tiny"], 32, cfg_strength=2.0)
    assert f3dc.weights_elems(ok) > 0
    bad = f3dc.config_for(synth.SHAPES["tiny"], 33, cfg_strength=2.0)
    assert f3dc.weights_elems(bad) == 0
    bad = f3dc.config_for(synth.ModelShape(8, 8, 128, 2, 4, 4, 64, 128, 8, 8), decoder=1)
    assert f3dc.weights_elems(bad) == 0
    d = f3dc.default_config()
    assert d.cfg_strength == 0.0 and d.cfg_t_lo == 0.5 and d.ssc_accel == 0 and d.decoder == 0


def test_fit_mu_rejects_bad_arguments(L):
    with pytest.raises(f3dc.F3dcError):
        f3dc.fit_mu(np.ones((2, 25)), k_lo=10, k_hi=5)
    with pytest.raises(f3dc.F3dcError):
        f3dc.fit_mu(np.ones((2, 25)), min_frac=1.5)


def test_fault_injection_argument_checks():
    # host only: out-of-range settings are refused, valid ones and "off" accepted
    for bad in [dict(fail_alloc_at=-2), dict(gemm_missing_arrivals=-1), dict(gemm_missing_arrivals=5000),
                dict(gemm_wait_ns=-1), dict(attn_missing_kv=2)]:
        with pytest.raises(f3dc.F3dcError) as e:
            f3dc.set_fault_injection(**bad)
        assert e.value.status == 1
    f3dc.set_fault_injection(fail_alloc_at=3, gemm_missing_arrivals=1, gemm_wait_ns=1000, attn_missing_kv=1)
    f3dc.set_fault_injection()
    assert f3dc.lib().f3dc_set_fault_injection(None) == 0
