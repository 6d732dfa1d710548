"""Oracle pins for the data-driven PCSC slope (Supp. "Data-driven Parameter
Selection"): RANSAC fits of ln(dS_k) against the step index over steps
8..18, poor fits filtered out, mu = the median of the remaining slopes."""
import math

import numpy as np


def _curve(T, slope, level=9.0, k_lo=8, k_hi=18, noise=None, outliers=()):
    k = np.arange(1, T + 1, dtype=np.float64)
    y = level + slope * (k - 8)
    if noise is not None:
        y = y + noise
    d = np.exp(y)
    for kk, factor in outliers:
        d[kk - 1] *= factor
    return d


def test_exact_log_linear_curves_give_their_slopes(orc):
    slopes = [-0.07, -0.183, -0.02, -0.3]
    curves = np.stack([_curve(25, s) for s in slopes])
    mu, got, kept = orc.fit_mu(curves)
    assert kept.all()
    np.testing.assert_allclose(got, slopes, rtol=0, atol=1e-12)
    assert abs(mu - 0.5 * (-0.07 + -0.183)) < 1e-12          # median of four: mean of the middle two


def test_gross_outliers_do_not_move_the_fit(orc):
    # two steps of the window off by factors e^2 and e^-3: RANSAC keeps the
    # line, while a plain least-squares fit over all points would not
    d = _curve(25, -0.1, outliers=((10, math.e ** 2), (15, math.e ** -3)))
    mu, got, kept = orc.fit_mu(d[None, :])
    assert kept[0] and abs(got[0] + 0.1) < 1e-12 and abs(mu + 0.1) < 1e-12
    k = np.arange(8, 19, dtype=np.float64)
    ls = np.polyfit(k, np.log(d[7:18]), 1)[0]
    assert abs(ls + 0.1) > 0.02


def test_window_edges_and_zero_counts(orc):
    # points outside 8..18 are ignored; a zero count carries no point
    d = _curve(25, -0.05)
    d[:7] = 1.0                       # steps 1..7: anything
    d[18:] = 1e9                      # steps 19..: anything
    d[11] = 0.0                       # step 12: no point
    mu, got, kept = orc.fit_mu(d[None, :])
    assert kept[0] and abs(got[0] + 0.05) < 1e-12


def test_noisy_instances_are_filtered_and_median_taken(orc):
    rng = np.random.default_rng(0)
    good = [_curve(25, s, noise=rng.normal(0, 0.01, 25)) for s in (-0.06, -0.07, -0.08)]
    bad = _curve(25, -0.07, noise=rng.normal(0, 1.5, 25))   # no line fits most points
    few = np.zeros(25)
    few[9] = few[10] = 5.0                                   # two points only
    mu, got, kept = orc.fit_mu(np.stack(good + [bad, few]))
    assert list(kept) == [True, True, True, False, False]
    assert abs(mu - np.median(got[:3])) < 1e-15 and abs(mu + 0.07) < 0.01
    mu_none, _, kept_none = orc.fit_mu(np.stack([bad, few]))
    assert not kept_none.any() and math.isnan(mu_none)


def test_sampler_curve_contains_the_anchor_measurement(orc):
    # the per-step curve of Eq. 1 holds the anchor step's sigma at k_a
    from paper_2511_22533_gb300 import synth
    shape = synth.SHAPES["tiny"]
    m = orc.Model(shape, synth.weights_blob(shape, 0))
    S = synth.latents(shape, 1, 0)
    cond = synth.cond_tokens(shape, 1, 0)
    T = shape.steps
    out = m.sample(S, cond, T=T, quota_schedule=np.zeros((T, 1), np.int32), tau=0, want_curve=True)
    ka = math.ceil(T * 0.2)
    assert out["dyn"][ka - 1, 0] == out["sigma"][0]
    assert np.all(out["dyn"] >= 0) and np.all(out["dyn"] <= 64 * shape.tokens) and out["dyn"].sum() > 0
