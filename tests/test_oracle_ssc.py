"""Oracle pins: SSC score (Sec. 4.1-4.2) and lowest-c selection (Alg. 1)."""
import itertools

import numpy as np
import pytest

from conftest import read_golden
from paper_2511_22533_gb300 import synth


def _bits(a):
    return synth.f32_to_bf16_bits(np.asarray(a, np.float32))


def _worked():
    rows = read_golden("ssc_worked_example.txt")
    v1 = np.zeros((len(rows), 8), np.float32)
    v2 = np.zeros((len(rows), 8), np.float32)
    exp = []
    for r, row in enumerate(rows):
        v1[r, :2] = [float(row[1]), float(row[2])]
        v2[r, :2] = [float(row[3]), float(row[4])]
        exp.append(float(row[5]))
    return v1, v2, np.array(exp)


def test_ssc_worked_example(orc):
    v1, v2, exp = _worked()
    s = orc.ssc_score(_bits(v1), _bits(v2), 0.7)
    np.testing.assert_allclose(s, exp, rtol=0, atol=2e-7)
    for c, expect in [(1, {1}), (2, {1, 0}), (3, {1, 0, 3}), (4, {0, 1, 2, 3})]:
        cached, idx = orc.select(s, c)
        assert set(np.nonzero(cached)[0].tolist()) == expect
        assert sorted(set(range(4)) - expect) == idx.tolist()


def test_ssc_omega_extremes(orc):
    rng = np.random.default_rng(1)
    v1 = rng.standard_normal((300, 8)).astype(np.float32)
    v2 = rng.standard_normal((300, 8)).astype(np.float32)
    b1, b2 = _bits(v1), _bits(v2)
    f1, f2 = synth.bf16_bits_to_f32(b1), synth.bf16_bits_to_f32(b2)
    V = np.sqrt((f1.astype(np.float64) ** 2).sum(1))
    A = np.sqrt(((f1.astype(np.float64) - f2) ** 2).sum(1))
    s1 = orc.ssc_score(b1, b2, 1.0)   # acceleration only
    s0 = orc.ssc_score(b1, b2, 0.0)   # velocity only
    assert np.array_equal(np.argsort(s1, kind="stable"), np.argsort(A, kind="stable"))
    assert np.array_equal(np.argsort(s0, kind="stable"), np.argsort(V, kind="stable"))
    # the extremes of each statistic normalise to exactly 0 and 1
    assert s1[np.argmin(A)] == 0.0 and s1[np.argmax(A)] == 1.0
    assert s0[np.argmin(V)] == 0.0 and s0[np.argmax(V)] == 1.0


def test_ssc_range_and_scale_invariance(orc):
    rng = np.random.default_rng(2)
    v1 = _bits(rng.standard_normal((512, 8)))
    v2 = _bits(rng.standard_normal((512, 8)))
    s = orc.ssc_score(v1, v2, 0.7)
    assert s.min() >= 0.0 and s.max() <= 1.0
    # multiplying every velocity by 4 scales every norm by 4 exactly; the
    # min-max normalisation cancels it
    f1, f2 = synth.bf16_bits_to_f32(v1) * 4, synth.bf16_bits_to_f32(v2) * 4
    s4 = orc.ssc_score(_bits(f1), _bits(f2), 0.7)
    np.testing.assert_array_equal(s, s4)


def test_ssc_permutation_equivariant(orc):
    rng = np.random.default_rng(3)
    v1 = _bits(rng.standard_normal((200, 8)))
    v2 = _bits(rng.standard_normal((200, 8)))
    p = rng.permutation(200)
    s = orc.ssc_score(v1, v2, 0.7)
    sp = orc.ssc_score(v1[p], v2[p], 0.7)
    np.testing.assert_array_equal(s[p], sp)


def test_ssc_unchanged_velocity_has_zero_acceleration(orc):
    # v(t-1) == v(t-2) everywhere: A = 0 (degenerate range) so C = (1-w) norm(V)
    rng = np.random.default_rng(4)
    v = _bits(rng.standard_normal((100, 8)))
    s = orc.ssc_score(v, v, 0.7)
    s0 = orc.ssc_score(v, v, 0.0)
    f = synth.bf16_bits_to_f32(v).astype(np.float64)
    V = np.sqrt((f ** 2).sum(1))
    assert np.array_equal(np.argsort(s, kind="stable"), np.argsort(V, kind="stable"))
    np.testing.assert_allclose(s, np.float32(0.3) * s0, rtol=1e-6, atol=1e-7)


def test_ssc_constant_field_caches_lowest_indices(orc):
    h = synth.velocity_history(4, 8, 1, 0, "constant")
    s = orc.ssc_score(h[2, 0], h[1, 0], 0.7)
    assert np.all(s == 0.0)
    cached, idx = orc.select(s, 10)
    assert np.nonzero(cached)[0].tolist() == list(range(10))
    assert idx.tolist() == list(range(10, 64))


def test_ssc_nan_is_never_cached(orc):
    rng = np.random.default_rng(5)
    v1 = rng.standard_normal((50, 8)).astype(np.float32)
    v1[7, 3] = np.nan
    b1 = _bits(v1)
    b2 = _bits(rng.standard_normal((50, 8)))
    s = orc.ssc_score(b1, b2, 0.7)
    assert np.isnan(s[7]) and np.isfinite(np.delete(s, 7)).all()
    cached, idx = orc.select(s, 49)
    assert cached[7] == 0 and idx.tolist() == [7]


def _brute_force_cached(s, c):
    """cached iff fewer than c tokens precede it in the (score, index) order;
    NaN scores follow every number.  O(N^2), independent of any sort."""
    N = len(s)
    out = np.zeros(N, np.uint8)
    for i in range(N):
        rank = 0
        for j in range(N):
            if j == i:
                continue
            ni, nj = np.isnan(s[i]), np.isnan(s[j])
            if ni != nj:
                before = ni  # j is a number and i is NaN
            elif not ni and s[j] != s[i]:
                before = s[j] < s[i]
            else:
                before = j < i
            rank += before
        out[i] = rank < c
    return out


@pytest.mark.parametrize("grid,kind", list(itertools.product([2, 3, 4], ["drift", "ties"])))
def test_selection_brute_force_small_grids(orc, grid, kind):
    h = synth.velocity_history(grid, 8, 1, 11 + grid, kind)
    s = orc.ssc_score(h[2, 0], h[1, 0], 0.7)
    N = grid ** 3
    for c in range(0, N + 1):
        cached, idx = orc.select(s, c)
        np.testing.assert_array_equal(cached, _brute_force_cached(s, c))
        assert idx.tolist() == [i for i in range(N) if not cached[i]]
        assert len(idx) == N - c


def test_selection_clamps_quota(orc):
    s = np.linspace(0, 1, 10).astype(np.float32)
    cached, idx = orc.select(s, 25)
    assert cached.all() and len(idx) == 0
    cached, idx = orc.select(s, -3)
    assert not cached.any() and idx.tolist() == list(range(10))


def test_selection_signed_zero_ties_by_index(orc):
    s = np.array([0.0, -0.0, 0.0, -0.0], np.float32)
    cached, _ = orc.select(s, 2)
    assert cached.tolist() == [1, 1, 0, 0]


# ---- SSC with three predictions: the second difference of the velocity
def _bf16(a):
    return synth.f32_to_bf16_bits(np.asarray(a, np.float32))


def test_ssc3_linear_history_has_zero_acceleration(orc):
    # v(t-3), v(t-2), v(t-1) on a straight line (small integers: exact in
    # bf16) have a zero second difference everywhere, so the score is the
    # velocity term alone: (1 - w) norm(V)
    rng = np.random.default_rng(0)
    a = rng.integers(-8, 8, (64, 8)).astype(np.float32)
    d = rng.integers(-4, 4, (64, 8)).astype(np.float32)
    v3, v2, v1 = _bf16(a), _bf16(a + d), _bf16(a + 2 * d)
    s3 = orc.ssc_score3(v1, v2, v3, 0.7)
    nv = orc.ssc_score(v1, v2, 0.0)                 # w = 0: exactly norm(V)
    np.testing.assert_array_equal(s3, (np.float32(1.0) - np.float32(0.7)) * nv)


def test_ssc3_constant_previous_pair_is_the_first_difference(orc):
    # v(t-3) = v(t-2): the second difference is the first difference exactly
    v = synth.velocity_history(4, 8, 1, seed=2)
    v1, v2 = v[2, 0], v[1, 0]
    np.testing.assert_array_equal(orc.ssc_score3(v1, v2, v2, 0.7), orc.ssc_score(v1, v2, 0.7))


def test_ssc3_quadratic_history_orders_by_curvature(orc):
    # v = a + b t + c t^2 at t = 0, 1, 2: second difference 2c per token, so
    # with w = 1 the order is that of |c|
    rng = np.random.default_rng(1)
    n = 27
    a = rng.integers(-4, 4, (n, 8)).astype(np.float32)
    b = rng.integers(-2, 2, (n, 8)).astype(np.float32)
    c = np.zeros((n, 8), np.float32)
    mags = rng.permutation(n).astype(np.float32) + 1
    c[:, 0] = mags / 8.0                            # distinct |c|, exact in bf16
    v3, v2, v1 = _bf16(a), _bf16(a + b + c), _bf16(a + 2 * b + 4 * c)
    s = orc.ssc_score3(v1, v2, v3, 1.0)
    np.testing.assert_array_equal(np.argsort(s, kind="stable"), np.argsort(mags, kind="stable"))
    assert s[np.argmin(mags)] == 0.0 and s[np.argmax(mags)] == 1.0
