"""f3dc_gemm_noalloc: the GEMM for callers that cannot allocate device memory
(code under global-mode graph capture, frameworks that own every device
allocation, loops that must not enter the driver's allocator).  Its split-K
scratch is a fixed array inside libf3dc instead of an allocation; its output
must match f3dc_gemm's on two calls in a row, the second of which starts from
whatever the first left in that shared array.

This file is collected last so that a run which stops at the first failure
has already run every other test."""
import numpy as np
import pytest
import torch

from gpu_helpers import dev_bf16, dev_f32, rel_l2
from paper_2511_22533_gb300 import f3dc, synth

pytestmark = pytest.mark.gpu


def _inputs(M, N, K, seed):
    g = np.random.default_rng(seed)
    A = dev_bf16(synth.f32_to_bf16_bits(g.standard_normal((M, K)).astype(np.float32)))
    Bw = dev_bf16(synth.f32_to_bf16_bits((g.standard_normal((N, K)) / np.sqrt(K)).astype(np.float32)))
    bias = dev_bf16(synth.f32_to_bf16_bits((0.02 * g.standard_normal(N)).astype(np.float32)))
    gate = dev_f32(g.standard_normal(N).astype(np.float32))
    x0 = g.standard_normal((M, N)).astype(np.float32)
    return A, Bw, bias, gate, x0


def _both(M, N, K, epi, seed):
    A, Bw, bias, gate, x0 = _inputs(M, N, K, seed)
    if epi == f3dc.EPI_RESID:
        ref, got = dev_f32(x0), dev_f32(x0)
        g = gate
    else:
        ref = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
        got = torch.full((M, N), 7.0, dtype=torch.bfloat16, device="cuda")
        g = None
    f3dc.gemm(A, Bw, bias, g, ref, M, N, K, epi)
    f3dc.gemm_noalloc(A, Bw, bias, g, got, M, N, K, epi)
    torch.cuda.synchronize()
    return got.float().cpu().numpy(), ref.float().cpu().numpy()


def _assert_close(got, ref, epi):
    # the tolerances of the GEMM parity tests
    if epi == f3dc.EPI_RESID:
        assert np.max(np.abs(got - ref)) < 1e-3 * max(1.0, np.abs(ref).max())
    else:
        assert rel_l2(got, ref) < 4e-3
        assert np.all(np.abs(got - ref) <= 2.0 ** -7 * np.abs(ref) + 1e-3)


def test_noalloc_matches_gemm_on_two_calls_in_a_row():
    # first call: few row tiles, so K is split and the static scratch is used;
    # second call: a different split count over the scratch the first one left
    for M, N, K, epi, seed in [(300, 1024, 4096, f3dc.EPI_RESID, 1), (955, 1024, 1024, f3dc.EPI_BIAS, 2)]:
        got, ref = _both(M, N, K, epi, seed)
        _assert_close(got, ref, epi)


def test_noalloc_without_split_and_with_gelu():
    for M, N, K, epi, seed in [(4096, 3072, 1024, f3dc.EPI_GELU, 3), (128, 256, 1024, f3dc.EPI_GELU, 4)]:
        got, ref = _both(M, N, K, epi, seed)
        _assert_close(got, ref, epi)


def test_noalloc_rejects_bad_arguments():
    A, Bw, bias, _, _ = _inputs(128, 128, 128, 5)
    out = torch.zeros((128, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(f3dc.F3dcError) as e:
        f3dc.gemm_noalloc(A, Bw, bias, None, out, 128, 100, 128, f3dc.EPI_BIAS)
    assert e.value.status == 1
