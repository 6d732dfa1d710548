"""Writes phase_table_T25.txt: the three-phase cache budget of Algorithm 1
(step 1) with the PCSC forecast of Sec. 4.2 and the tau refresh rule of
Sec. 4.3, for T = 25 and the paper's default hyperparameters, evaluated in
50-digit decimal arithmetic (Python's decimal module).  It imports nothing
from the oracle or the library: the values it writes are what those two are
tested against.

    python tests/golden/make_phase_table_T25.py > tests/golden/phase_table_T25.txt
"""
from __future__ import annotations

import math
import sys
from decimal import Decimal, getcontext

getcontext().prec = 50

T = 25
N = 16 ** 3           # 16^3 latent tokens
GAMMA_UP = 64         # (64 / 16)^3 occupancy sub-voxels per token
SIGMA = 65536         # dynamic voxels measured at the anchor step
MU = Decimal("-0.07")
XI = Decimal("0.7")
RHO_A = Decimal("0.2")
RHO_OFF = Decimal("0.75")
F_CORR = 3
TAU = 3

HEADER = """\
# Three-phase cache budget for T = 25 with the paper's default hyperparameters
# (Supp. "More Ablation Study": mu=-0.07, omega=0.7, tau=3, xi=0.7, f_corr=3,
# rho_a=0.2, rho_CFG-OFF=0.75) on a 16^3 latent grid (N = 4096 tokens),
# gamma_up = 64 (64^3 occupancy grid over 16^3 tokens) and an anchor
# measurement sigma = 65536 dynamic voxels.
#
# Phase rule: Algorithm 1, step 1 -- k_a = ceil(25*0.2) = 5, k_off =
# ceil(25*0.75) = 19; Phase 1 (k <= 5) caches nothing; Phase 2 (5 < k < 19)
# caches c_k = N - sigma*exp(mu*(k - k_a))/gamma_up (Sec. 4.2, PCSC eqs.),
# floored; Phase 3 (k >= 19) caches floor(N*xi) = floor(2867.2) = 2867
# except the full-correction steps where (k - 19 + 1) mod 3 = 0, i.e. 21, 24.
# Phase-2 values are evaluated at 50 significant digits by
# make_phase_table_T25.py (Python decimal), not with the oracle; the closest
# to an integer is step 8 (0.038 away), far beyond the ~1e-12 error of an
# fp64 evaluation, so floor() is not decided by rounding.  Step 6 is the
# hand check
# floor(4096 - 1024*e^-0.07) = floor(4096 - 954.77) = 3141.
#
# The last column applies the tau = 3 refresh rule (Sec. 4.3 Phase 2,
# Algorithm 1 SSC) in the period reading: at most tau-1 = 2 consecutive
# cached steps, then a forced full step; the counter restarts on every
# full step, and the rule applies in every phase.
#
# k phase quota_before_tau quota_after_tau"""


def ceil_dec(x: Decimal) -> int:
    return int(x.to_integral_value(rounding="ROUND_CEILING"))


def table():
    """Rows (k, phase, quota before tau, quota after tau, phase-2 margin to the
    nearest integer or None)."""
    ka = ceil_dec(T * RHO_A)
    koff = ceil_dec(T * RHO_OFF)
    rows, consec = [], 0
    for k in range(1, T + 1):
        margin = None
        if k <= ka:
            phase, q = 1, 0
        elif k < koff:
            phase = 2
            exact = Decimal(N) - Decimal(SIGMA) * (MU * (k - ka)).exp() / GAMMA_UP
            q = max(0, min(N, math.floor(exact)))
            frac = exact - math.floor(exact)
            margin = min(frac, 1 - frac)
        else:
            phase = 3
            q = 0 if (k - koff + 1) % F_CORR == 0 else math.floor(Decimal(N) * XI)
        # period reading of the tau rule: at most tau - 1 consecutive cached steps
        after = q
        if after > 0 and consec >= TAU - 1:
            after = 0
        consec = consec + 1 if after > 0 else 0
        rows.append((k, phase, q, after, margin))
    return rows


def main(out=sys.stdout):
    print(HEADER, file=out)
    for k, phase, q, after, _ in table():
        print(f"{k} {phase} {q} {after}", file=out)


if __name__ == "__main__":
    main()
