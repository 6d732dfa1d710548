"""f3dc_gemm_noalloc: the GEMM for callers that cannot allocate device memory
(code under global-mode graph capture, frameworks that own every device
allocation, loops that must not enter the driver's allocator).  Its split-K
scratch is a fixed array inside libf3dc instead of an allocation, and it
makes f3dc_gemm's launch decisions, so its output must equal f3dc_gemm's bit
for bit -- here on two split calls in a row with different split counts (the
second starts from whatever the first left in the shared array), on shapes
that take the CTA-pair kernel, and once against the oracle.

This file is collected last so that a run which stops at the first failure
has already run every other test."""
import numpy as np
import pytest
import torch

from gpu_helpers import dev_bf16, dev_f32, rel_l2
from paper_2511_22533_gb300 import f3dc, synth

pytestmark = pytest.mark.gpu


def _split_count(M, N, K, sms):
    """The library's split-K rule for a standalone GEMM (host restatement):
    split only when whole 128-row tiles leave at least half of the grid idle
    and K >= 2048, >= 4 K blocks of 64 per split, no empty split."""
    bn = 256 if N % 256 == 0 else (128 if N % 128 == 0 else 64)
    tiles = -(-M // 128) * (N // bn)
    grid = sms if 2 * tiles <= sms else min(tiles, sms)
    kb = K // 64
    if 2 * tiles > grid or tiles > 1024 or kb < 32:
        return 1
    sp = min(grid // tiles, kb // 4, sms // tiles, 16)
    if sp <= 1:
        return 1
    per = -(-kb // sp)
    return -(-kb // per)


def _inputs(M, N, K, seed):
    g = np.random.default_rng(seed)
    A = synth.f32_to_bf16_bits(g.standard_normal((M, K)).astype(np.float32))
    Bw = synth.f32_to_bf16_bits((g.standard_normal((N, K)) / np.sqrt(K)).astype(np.float32))
    bias = synth.f32_to_bf16_bits((0.02 * g.standard_normal(N)).astype(np.float32))
    gate = g.standard_normal(N).astype(np.float32)
    x0 = g.standard_normal((M, N)).astype(np.float32)
    return A, Bw, bias, gate, x0


def _both(M, N, K, epi, seed):
    A, Bw, bias, gate, x0 = _inputs(M, N, K, seed)
    Ad, Bd, bd = dev_bf16(A), dev_bf16(Bw), dev_bf16(bias)
    if epi == f3dc.EPI_RESID:
        ref, got = dev_f32(x0), dev_f32(x0)
        g = dev_f32(gate)
    else:
        ref = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
        got = torch.full((M, N), 7.0, dtype=torch.bfloat16, device="cuda")
        g = None
    f3dc.gemm(Ad, Bd, bd, g, ref, M, N, K, epi)
    f3dc.gemm_noalloc(Ad, Bd, bd, g, got, M, N, K, epi)
    torch.cuda.synchronize()
    return got.float().cpu().numpy(), ref.float().cpu().numpy(), (A, Bw, bias, gate, x0)


def test_noalloc_equals_gemm_on_two_split_calls_in_a_row(orc):
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    cases = [(300, 1024, 4096, f3dc.EPI_RESID, 1), (200, 1024, 2048, f3dc.EPI_BIAS, 2)]
    counts = [_split_count(M, N, K, sms) for M, N, K, _, _ in cases]
    assert counts[0] > 1 and counts[1] > 1 and counts[0] != counts[1], counts
    for (M, N, K, epi, seed) in cases:
        got, ref, (A, Bw, bias, gate, x0) = _both(M, N, K, epi, seed)
        np.testing.assert_array_equal(got, ref)
        if epi == f3dc.EPI_RESID:
            # once against the oracle: x0 + gate * (A B^T + bias) on sampled rows
            rows = np.arange(0, M, 7)
            y = orc.linear(synth.bf16_bits_to_f32(A[rows]), synth.bf16_bits_to_f32(Bw),
                           synth.bf16_bits_to_f32(bias)).astype(np.float64)
            expect = x0[rows].astype(np.float64) + gate.astype(np.float64) * y
            assert np.max(np.abs(got[rows] - expect)) < 1e-3 * max(1.0, np.abs(expect).max())
    assert f3dc.gemm_status() == 0


def test_noalloc_equals_gemm_without_split():
    # the CTA-pair kernel (256-wide tiles, K % 128 == 0, no split) and the
    # single-CTA kernel for a 128-wide N
    for M, N, K, epi, seed in [(4096, 3072, 1024, f3dc.EPI_GELU, 3), (128, 256, 1024, f3dc.EPI_GELU, 4),
                               (955, 1024, 1024, f3dc.EPI_BIAS, 5), (300, 384, 512, f3dc.EPI_RESID, 6)]:
        got, ref, _ = _both(M, N, K, epi, seed)
        np.testing.assert_array_equal(got, ref)
        assert rel_l2(got, ref) == 0.0
    assert f3dc.gemm_status() == 0


def test_noalloc_rejects_bad_arguments():
    A, Bw, bias, _, _ = _inputs(128, 128, 128, 5)
    out = torch.zeros((128, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(f3dc.F3dcError) as e:
        f3dc.gemm_noalloc(dev_bf16(A), dev_bf16(Bw), dev_bf16(bias), None, out, 128, 100, 128, f3dc.EPI_BIAS)
    assert e.value.status == 1
