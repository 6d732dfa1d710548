"""K5 / K6 parity: the tcgen05 flash attention against the oracle's fp64
softmax attention (Supp. Sec. F self- and cross-attention) on sampled query
rows: active-token sequences (ragged, 1229, 4096), the 1374-token condition,
head dims 32 and 64, a single key and odd tails."""
import numpy as np
import pytest
import torch

from gpu_helpers import dev_bf16, rel_l2
from paper_2511_22533_gb300 import f3dc, synth

pytestmark = pytest.mark.gpu

CASES = [(300, 300, 4, 32), (1229, 1229, 16, 64), (4096, 4096, 16, 64), (1229, 1374, 16, 64), (5, 1, 2, 64),
         (130, 129, 2, 32), (128, 256, 1, 64), (700, 77, 4, 32), (256, 256, 1, 64), (128, 384, 1, 64),
         (1, 200, 1, 32), (128, 129, 1, 64)]


@pytest.mark.parametrize("nq,nk,H,dh", CASES)
def test_attention(orc, nq, nk, H, dh):
    g = np.random.default_rng(nq * 7 + nk)
    W = H * dh
    q = synth.f32_to_bf16_bits(g.standard_normal((nq, W)).astype(np.float32))
    kv = synth.f32_to_bf16_bits(g.standard_normal((nk, 2 * W)).astype(np.float32))
    out = torch.zeros((nq, W), dtype=torch.bfloat16, device="cuda")
    kvd = dev_bf16(kv)
    f3dc.attention(dev_bf16(q), W, kvd, kvd[:, W:], 2 * W, out, nq, nk, H, dh)
    torch.cuda.synchronize()
    rows = np.unique(np.concatenate([[0, nq - 1], g.integers(0, nq, 48)]))
    kf = synth.bf16_bits_to_f32(kv)
    ref = orc.attention(synth.bf16_bits_to_f32(q[rows]), kf[:, :W], kf[:, W:], H).astype(np.float64)
    got = out.float().cpu().numpy()[rows]
    assert np.isfinite(got).all()
    assert rel_l2(got, ref) < 1e-2
    assert np.max(np.abs(got - ref)) < 2e-2


def test_attention_rows_beyond_nq_untouched():
    nq, nk, H, dh = 100, 300, 2, 64
    g = np.random.default_rng(0)
    q = dev_bf16(synth.f32_to_bf16_bits(g.standard_normal((128, H * dh)).astype(np.float32)))
    kv = dev_bf16(synth.f32_to_bf16_bits(g.standard_normal((nk, H * dh)).astype(np.float32)))
    out = torch.full((128, H * dh), 3.0, dtype=torch.bfloat16, device="cuda")
    f3dc.attention(q, H * dh, kv, kv, H * dh, out, nq, nk, H, dh)
    torch.cuda.synchronize()
    assert torch.all(out[nq:] == 3.0)
    assert torch.isfinite(out[:nq].float()).all()
