"""K4 parity: the tcgen05 GEMM with its fused epilogues against the oracle's
fp64-accumulated nn.Linear (Supp. Sec. F projections), on sampled output
rows at the transformer's shapes (active-token counts 1229 / 4096, widths
1024 / 3072 / 4096, K 1024 / 4096) and on ragged small cases."""
import numpy as np
import pytest
import torch

from gpu_helpers import dev_bf16, dev_f32, rel_l2
from paper_2511_22533_gb300 import f3dc, synth

pytestmark = pytest.mark.gpu

SHAPES = [(1229, 1024, 1024), (4096, 3072, 1024), (1000, 4096, 1024), (1229, 1024, 4096), (100, 256, 128),
          (1, 64, 64), (257, 384, 128), (300, 128, 256)]
# few row tiles: the kernel splits K over CTAs and reduces the partials in
# split order (workspace + per-tile arrival counters)
SPLIT_SHAPES = [(955, 1024, 1024), (300, 1024, 4096), (128, 256, 1024), (640, 3072, 1024), (413, 1024, 4096)]


def _inputs(M, N, K, seed):
    g = np.random.default_rng(seed)
    A = synth.f32_to_bf16_bits(g.standard_normal((M, K)).astype(np.float32))
    Bw = synth.f32_to_bf16_bits((g.standard_normal((N, K)) / np.sqrt(K)).astype(np.float32))
    bias = synth.f32_to_bf16_bits((0.02 * g.standard_normal(N)).astype(np.float32))
    gate = g.standard_normal(N).astype(np.float32)
    rows = np.unique(np.concatenate([[0, M - 1], g.integers(0, M, 64)]))
    return A, Bw, bias, gate, rows


def _ref(orc, A, Bw, bias, rows):
    a = synth.bf16_bits_to_f32(A[rows])
    w = synth.bf16_bits_to_f32(Bw)
    return orc.linear(a, w, synth.bf16_bits_to_f32(bias)).astype(np.float64)


@pytest.mark.parametrize("M,N,K", SHAPES + SPLIT_SHAPES)
def test_gemm_bias(orc, M, N, K):
    A, Bw, bias, _, rows = _inputs(M, N, K, M + N + K)
    out = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
    f3dc.gemm(dev_bf16(A), dev_bf16(Bw), dev_bf16(bias), None, out, M, N, K, f3dc.EPI_BIAS)
    torch.cuda.synchronize()
    got = out.float().cpu().numpy()[rows]
    ref = _ref(orc, A, Bw, bias, rows)
    assert rel_l2(got, ref) < 4e-3
    # bf16 output: within one rounding step of the fp64 result
    assert np.all(np.abs(got - ref) <= 2.0 ** -7 * np.abs(ref) + 1e-3)


@pytest.mark.parametrize("M,N,K", SHAPES[:4] + SPLIT_SHAPES[:2])
def test_gemm_gelu(orc, M, N, K):
    A, Bw, bias, _, rows = _inputs(M, N, K, 7 + M)
    out = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
    f3dc.gemm(dev_bf16(A), dev_bf16(Bw), dev_bf16(bias), None, out, M, N, K, f3dc.EPI_GELU)
    torch.cuda.synchronize()
    got = out.float().cpu().numpy()[rows]
    pre = _ref(orc, A, Bw, bias, rows)
    ref = np.vectorize(orc.gelu)(pre.astype(np.float32)).astype(np.float64)
    assert rel_l2(got, ref) < 5e-3
    assert np.max(np.abs(got - ref)) < 2e-2 * max(1.0, np.abs(ref).max())


@pytest.mark.parametrize("M,N,K", SHAPES[:4] + SHAPES[6:] + SPLIT_SHAPES)
@pytest.mark.parametrize("with_gate", [True, False])
def test_gemm_residual(orc, M, N, K, with_gate):
    A, Bw, bias, gate, rows = _inputs(M, N, K, 11 + N)
    x0 = np.random.default_rng(1).standard_normal((M, N)).astype(np.float32)
    x = dev_f32(x0)
    f3dc.gemm(dev_bf16(A), dev_bf16(Bw), dev_bf16(bias), dev_f32(gate) if with_gate else None, x, M, N, K,
              f3dc.EPI_RESID)
    torch.cuda.synchronize()
    got = x.cpu().numpy().astype(np.float64)
    y = _ref(orc, A, Bw, bias, rows)
    ref = x0[rows].astype(np.float64) + (gate[None, :] * y if with_gate else y)
    assert np.max(np.abs(got[rows] - ref)) < 1e-3 * max(1.0, np.abs(ref).max())
    # untouched rows beyond M do not exist; every row of x was updated exactly once
    others = np.setdiff1d(np.arange(M), rows)[:8]
    if len(others):
        y2 = _ref(orc, A, Bw, bias, others)
        r2 = x0[others] + (gate[None, :] * y2 if with_gate else y2)
        assert np.max(np.abs(got[others] - r2)) < 1e-3 * max(1.0, np.abs(r2).max())


def test_gemm_no_bias_and_repeat_is_deterministic(orc):
    M, N, K = 777, 1024, 1024
    A, Bw, _, _, rows = _inputs(M, N, K, 5)
    outs = []
    for _ in range(2):
        out = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
        f3dc.gemm(dev_bf16(A), dev_bf16(Bw), None, None, out, M, N, K, f3dc.EPI_BIAS)
        outs.append(out)
    torch.cuda.synchronize()
    assert torch.equal(outs[0], outs[1])
    ref = orc.linear(synth.bf16_bits_to_f32(A[rows]), synth.bf16_bits_to_f32(Bw))
    assert rel_l2(outs[0].float().cpu().numpy()[rows], ref) < 4e-3


def test_gemm_split_k_repeat_is_deterministic(orc):
    # the split partials are always summed in split order by whichever CTA
    # arrives last, so repeated launches agree bit for bit
    M, N, K = 300, 1024, 4096
    A, Bw, bias, gate, rows = _inputs(M, N, K, 21)
    outs = []
    for _ in range(3):
        x = torch.zeros((M, N), dtype=torch.float32, device="cuda")
        f3dc.gemm(dev_bf16(A), dev_bf16(Bw), dev_bf16(bias), dev_f32(gate), x, M, N, K, f3dc.EPI_RESID)
        outs.append(x)
    torch.cuda.synchronize()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])
