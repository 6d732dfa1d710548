"""K1 parity: SSC score + lowest-c selection on the GPU is bit-exact with the
oracle (Sec. 4.1-4.2 Eq. ssc / Eq. normalize; Algorithm 1 SSC) on the
selection-only workload (16^3 tokens x 8 channels, batch 1-64, quotas
10-90%), on ties, constant fields, NaN / Inf, edge quotas and other grids."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_clean, dev_i32, dev_u16, handle_for
from paper_2511_22533_gb300 import synth

pytestmark = pytest.mark.gpu


def _shape(grid):
    return synth.ModelShape(grid, 8, 128, 1, 4, 4, 64, 128, 25, 64)


@pytest.fixture(scope="module")
def h16():
    h, _, _ = handle_for(_shape(16), max_batch=64)
    yield h
    h.close()


def _run(h, hist, quotas):
    B, N = hist.shape[1], hist.shape[2]
    v1, v2 = dev_u16(hist[2]), dev_u16(hist[1])
    q = dev_i32(quotas)
    idx = torch.full((B, N), -7, dtype=torch.int32, device="cuda")
    na = torch.zeros(B, dtype=torch.int32, device="cuda")
    mask = torch.full((B, N), 9, dtype=torch.uint8, device="cuda")
    h.ssc_select(v1, v2, B, q, idx, na, mask)
    torch.cuda.synchronize()
    assert_clean(h)
    return idx.cpu().numpy(), na.cpu().numpy(), mask.cpu().numpy()


def _check(orc, hist, quotas, idx, na, mask, omega=0.7):
    N = hist.shape[2]
    for b in range(hist.shape[1]):
        s = orc.ssc_score(hist[2, b], hist[1, b], omega)
        cached, aidx = orc.select(s, int(quotas[b]))
        assert na[b] == len(aidx) == N - min(max(int(quotas[b]), 0), N)
        np.testing.assert_array_equal(mask[b], cached, err_msg=f"sample {b}")
        np.testing.assert_array_equal(idx[b, :na[b]], aidx, err_msg=f"sample {b}")


@pytest.mark.parametrize("B", [1, 8, 64])
def test_selection_sweep_drift(orc, h16, B):
    hist = synth.velocity_history(16, 8, B, seed=B, kind="drift")
    N = 4096
    qs = np.array([int(np.floor(q * N)) for q in np.tile([0.1, 0.3, 0.5, 0.7, 0.9], 13)[:B]], np.int32)
    idx, na, mask = _run(h16, hist, qs)
    _check(orc, hist, qs, idx, na, mask)


@pytest.mark.parametrize("kind", ["ties", "constant"])
def test_selection_ties_and_constant(orc, h16, kind):
    hist = synth.velocity_history(16, 8, 6, seed=3, kind=kind)
    qs = np.array([1, 409, 2048, 2867, 4000, 4095], np.int32)
    idx, na, mask = _run(h16, hist, qs)
    _check(orc, hist, qs, idx, na, mask)


def test_selection_edge_quotas(orc, h16):
    hist = synth.velocity_history(16, 8, 6, seed=4)
    qs = np.array([0, 4096, -5, 9999, 1, 4095], np.int32)
    idx, na, mask = _run(h16, hist, qs)
    _check(orc, hist, qs, idx, na, mask)
    np.testing.assert_array_equal(idx[0], np.arange(4096))
    assert na.tolist() == [4096, 0, 4096, 0, 4095, 1]


def test_selection_nan_inf(orc, h16):
    hist = synth.velocity_history(16, 8, 2, seed=5)
    f = synth.bf16_bits_to_f32(hist).copy()
    f[2, 0, 17, 3] = np.nan          # NaN velocity: never cached
    f[2, 0, 99, 0] = np.inf          # an infinite magnitude
    f[1, 1, 5, :] = f[2, 1, 5, :]    # a token with zero acceleration
    hist = synth.f32_to_bf16_bits(f)
    qs = np.array([3000, 2000], np.int32)
    idx, na, mask = _run(h16, hist, qs)
    _check(orc, hist, qs, idx, na, mask)
    assert mask[0, 17] == 0


@pytest.mark.parametrize("omega", [0.0, 0.3, 1.0])
def test_selection_omega(orc, omega):
    h, _, _ = handle_for(_shape(16), max_batch=4, omega=omega)
    hist = synth.velocity_history(16, 8, 4, seed=6)
    qs = np.array([500, 1500, 2500, 3500], np.int32)
    idx, na, mask = _run(h, hist, qs)
    _check(orc, hist, qs, idx, na, mask, omega=omega)
    h.close()


@pytest.mark.parametrize("grid,B", [(8, 3), (32, 2)])
def test_selection_other_grids(orc, grid, B):
    h, _, _ = handle_for(_shape(grid), max_batch=B)
    hist = synth.velocity_history(grid, 8, B, seed=grid)
    N = grid ** 3
    qs = np.array([N // 2, int(0.7 * N), N // 10][:B], np.int32)
    idx, na, mask = _run(h, hist, qs)
    _check(orc, hist, qs, idx, na, mask)
    h.close()


def test_selection_batch64_32cubed(orc):
    # the largest selection workload: 64 samples of 32768 tokens (the 32^3
    # grid), quotas 10-90 %, bit-exact on every sample
    h, _, _ = handle_for(_shape(32), max_batch=64)
    hist = synth.velocity_history(32, 8, 64, seed=32)
    N = 32768
    qs = np.array([int(np.floor(q * N)) for q in np.tile([0.1, 0.3, 0.5, 0.7, 0.9], 13)[:64]], np.int32)
    idx, na, mask = _run(h, hist, qs)
    _check(orc, hist, qs, idx, na, mask)
    h.close()
