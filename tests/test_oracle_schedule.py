"""Oracle pins: time schedule (Supp. Sec. D), phases and PCSC (Sec. 4.2,
Algorithm 1 step 1) and the tau refresh rule (Sec. 4.3, Algorithm 1 SSC)."""

import numpy as np
import pytest

from conftest import read_golden

DEF = dict(rho_a=0.2, rho_off=0.75, mu=-0.07, xi=0.7, f_corr=3, gamma_up=64)


@pytest.mark.parametrize("row", read_golden("schedule_turning_points.txt"))
def test_schedule_worked_example(orc, row):
    T, eta, k0 = int(row[0]), float(row[1]), int(row[2])
    t = orc.time_schedule(T, eta)
    below = np.nonzero(t < 0.5)[0]
    assert below[0] == k0


def test_schedule_endpoints_and_monotone(orc):
    for eta in (1.0, 2.0, 3.0):
        t = orc.time_schedule(25, eta)
        assert t[0] == 1.0 and t[-1] == 0.0
        assert np.all(np.diff(t) < 0)


def test_schedule_eta1_is_uniform(orc):
    t = orc.time_schedule(25, 1.0)
    expect = (1.0 - np.arange(26) / 25.0).astype(np.float32)
    np.testing.assert_array_equal(t, expect)


def test_ceil_steps(orc):
    assert orc.ceil_steps(25, 0.2) == 5
    assert orc.ceil_steps(25, 0.75) == 19
    assert orc.ceil_steps(8, 0.2) == 2
    assert orc.ceil_steps(50, 0.2) == 10


def test_phase_table_T25(orc):
    gate = orc.TauGate(3, 0)
    for row in read_golden("phase_table_T25.txt"):
        k, phase, q_raw, q_tau = map(int, row)
        c, ph = orc.phase_quota(4096, 25, DEF["rho_a"], DEF["rho_off"], DEF["mu"], DEF["xi"],
                                DEF["f_corr"], DEF["gamma_up"], 65536.0, k)
        assert (c, ph) == (q_raw, phase), k
        assert gate(c) == q_tau, k


def test_pcsc_clamps(orc):
    # a huge anchor change forecasts more dynamic voxels than the grid has: no caching
    c, ph = orc.phase_quota(4096, 25, 0.2, 0.75, -0.07, 0.7, 3, 64, 1e12, 6)
    assert (c, ph) == (0, 2)
    # no measured change: everything may be cached (upper bound N)
    c, _ = orc.phase_quota(4096, 25, 0.2, 0.75, -0.07, 0.7, 3, 64, 0.0, 6)
    assert c == 4096
    # NaN sigma is treated as "cache nothing"
    c, _ = orc.phase_quota(4096, 25, 0.2, 0.75, -0.07, 0.7, 3, 64, float("nan"), 6)
    assert c == 0


def test_pcsc_monotone_in_k(orc):
    # mu < 0: the forecast decays, so the cached budget grows through Phase 2
    qs = [orc.phase_quota(4096, 25, 0.2, 0.75, -0.07, 0.7, 3, 64, 2.0e5, k)[0] for k in range(6, 19)]
    assert all(b >= a for a, b in zip(qs, qs[1:]))
    assert qs[-1] > qs[0]


def test_phase3_fcorr_variants(orc):
    # f_corr = 1: every Phase-3 step is a full step ("Full sampling")
    for k in range(19, 26):
        assert orc.phase_quota(4096, 25, 0.2, 0.75, -0.07, 0.7, 1, 64, 1.0, k)[0] == 0
    # f_corr = 0: never corrected (Table "f_corr = 0 (w.o. f_corr)")
    for k in range(19, 26):
        assert orc.phase_quota(4096, 25, 0.2, 0.75, -0.07, 0.7, 0, 64, 1.0, k)[0] == 2867
    # f_corr = 2: correction at k_r = 1, 3, 5
    got = [orc.phase_quota(4096, 25, 0.2, 0.75, -0.07, 0.7, 2, 64, 1.0, k)[0] for k in range(19, 26)]
    assert got == [2867, 0, 2867, 0, 2867, 0, 2867]


def test_tau_period_reading(orc):
    # tau = 1 in the period reading caches nothing at all (consistent with the
    # tau = 1 row running slower than vanilla, Table "muandtau")
    g = orc.TauGate(1, 0)
    assert [g(100) for _ in range(6)] == [0] * 6
    g = orc.TauGate(3, 0)
    assert [g(100) for _ in range(7)] == [100, 100, 0, 100, 100, 0, 100]
    g = orc.TauGate(0, 0)  # disabled
    assert [g(100) for _ in range(5)] == [100] * 5


def test_tau_literal_reading(orc):
    g = orc.TauGate(3, 1)
    assert [g(100) for _ in range(9)] == [100, 100, 100, 0, 100, 100, 100, 0, 100]
    g = orc.TauGate(1, 1)
    assert [g(100) for _ in range(4)] == [100, 0, 100, 0]


def test_tau_counter_resets_on_natural_full_step(orc):
    g = orc.TauGate(3, 0)
    assert [g(q) for q in (100, 0, 100, 100, 100)] == [100, 0, 100, 100, 0]


def test_phase_table_file_matches_its_generator():
    # the stored table is exactly what its committed generator writes (50-digit
    # decimal arithmetic, independent of the oracle), and every Phase-2 value
    # lies far from an integer compared with fp64 rounding (the closest,
    # step 8, by 0.038), so the floor is not decided by rounding
    import importlib.util
    import io
    import os
    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    spec = importlib.util.spec_from_file_location("make_phase_table_T25",
                                                  os.path.join(here, "make_phase_table_T25.py"))
    gen = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(gen)
    buf = io.StringIO()
    gen.main(buf)
    with open(os.path.join(here, "phase_table_T25.txt")) as f:
        assert f.read() == buf.getvalue()
    margins = [m for *_, m in gen.table() if m is not None]
    assert len(margins) == 13 and min(margins) > 0.03
