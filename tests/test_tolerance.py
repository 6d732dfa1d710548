"""The stored-velocity bound used by the step parity tests: VEL_MAX_ABS on
the computed velocities, plus one bf16 unit for the two sides' own storage
rounding (round to nearest even, half a unit each)."""
import numpy as np

from gpu_helpers import VEL_MAX_ABS, bf16_ulp, stored_vel_excess
from paper_2511_22533_gb300 import synth


def test_bf16_ulp_spacing():
    assert bf16_ulp(1.0) == 2.0 ** -7
    assert bf16_ulp(1.99) == 2.0 ** -7
    assert bf16_ulp(-2.0) == 2.0 ** -6
    assert bf16_ulp(4.4) == 2.0 ** -5
    # next bf16 value above x is x + ulp(x)
    for x in [1.0, 1.5, 3.0, 4.5, 100.0]:
        b = synth.f32_to_bf16_bits(np.array([x], np.float32))
        nxt = synth.bf16_bits_to_f32(b + np.uint16(1))[0]
        assert nxt - x == bf16_ulp(x)


def test_rounding_flip_is_within_bound():
    # two computed values 1e-3 apart on either side of a rounding boundary at
    # |v| in [4, 8) store one unit (2^-5) apart: allowed
    lo, hi = 4.0 + 2.0 ** -6 - 5e-4, 4.0 + 2.0 ** -6 + 5e-4
    g = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(np.array([lo], np.float32)))
    r = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(np.array([hi], np.float32)))
    assert abs(g[0] - r[0]) == 2.0 ** -5 > VEL_MAX_ABS
    assert stored_vel_excess(g, r) < 0


def test_real_differences_fail():
    # three units at |v| in [2, 4) (0.047) exceed 2e-2 + one unit (0.036)
    assert stored_vel_excess(np.array([2.0 + 3 * 2.0 ** -6]), np.array([2.0])) > 0
    # 0.03 at |v| < 1 exceeds 2e-2 + 2^-8
    assert stored_vel_excess(np.array([0.53]), np.array([0.5])) > 0
    assert stored_vel_excess(np.array([0.515]), np.array([0.5])) < 0
