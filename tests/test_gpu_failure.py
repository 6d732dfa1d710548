"""Failure paths on the GPU, made on the host (nothing faults, traps or hangs
a GPU): a split-K arrival wait that no CTA can satisfy runs out after a short
limit, the kernel returns and the timeout is reported in the status word,
and the context stays usable; an allocation that f3dc_create is told has
failed makes it free what it holds and return F3DC_ERR_OOM."""
import time

import numpy as np
import pytest
import torch

from gpu_helpers import assert_clean, dev_bf16, dev_f32, dev_i32, dev_u16, handle_for
from paper_2511_22533_gb300 import f3dc, synth

pytestmark = pytest.mark.gpu

TIMEOUT = 1  # F3DC_DEV_TIMEOUT


def _gemm_inputs(M, N, K, seed):
    g = np.random.default_rng(seed)
    A = dev_bf16(synth.f32_to_bf16_bits(g.standard_normal((M, K)).astype(np.float32)))
    Bw = dev_bf16(synth.f32_to_bf16_bits((g.standard_normal((N, K)) / np.sqrt(K)).astype(np.float32)))
    bias = dev_bf16(synth.f32_to_bf16_bits((0.02 * g.standard_normal(N)).astype(np.float32)))
    return A, Bw, bias


def _tiny_step_clean():
    # a fresh handle runs a cached step with a clean status word
    shape = synth.SHAPES["tiny"]
    h, blob, _ = handle_for(shape, max_batch=1, seed=0)
    h.set_cond(dev_u16(synth.cond_tokens(shape, 1, 0)), 1)
    hist = synth.velocity_history(8, 8, 1, seed=1)
    ring = np.zeros((3, 1, shape.tokens, 8), np.uint16)
    ring[2], ring[1] = hist[2], hist[1]
    S = dev_f32(synth.latents(shape, 1, 0))
    h.step(3, 1, S, dev_u16(ring), dev_i32([256]))
    torch.cuda.synchronize()
    assert torch.isfinite(S).all()
    assert_clean(h)
    h.close()


def test_split_k_wait_runs_out_and_is_reported():
    M, N, K = 300, 1024, 4096  # 12 tiles on 152 SMs: K is split
    A, Bw, bias = _gemm_inputs(M, N, K, 1)
    assert f3dc.gemm_status() == 0
    out = torch.zeros((M, N), dtype=torch.bfloat16, device="cuda")
    f3dc.set_fault_injection(gemm_missing_arrivals=1, gemm_wait_ns=2_000_000)
    try:
        t0 = time.perf_counter()
        f3dc.gemm(A, Bw, bias, None, out, M, N, K, f3dc.EPI_BIAS)
        st = f3dc.gemm_status()  # synchronizes: the kernel has returned
        elapsed = time.perf_counter() - t0
    finally:
        f3dc.set_fault_injection()
    assert st & TIMEOUT, st
    assert elapsed < 5.0
    # the context is usable: the same GEMM now completes, equals the
    # no-alloc variant bit for bit, and reports nothing
    ref = torch.zeros_like(out)
    f3dc.gemm(A, Bw, bias, None, out, M, N, K, f3dc.EPI_BIAS)
    f3dc.gemm_noalloc(A, Bw, bias, None, ref, M, N, K, f3dc.EPI_BIAS)
    torch.cuda.synchronize()
    assert torch.equal(out, ref) and torch.isfinite(out.float()).all()
    assert f3dc.gemm_status() == 0
    _tiny_step_clean()


@pytest.mark.parametrize("n", [0, 7, 20, 34])
def test_create_reports_oom_and_frees(n):
    shape = synth.SHAPES["tiny"]
    blob = dev_u16(synth.weights_blob(shape, 0))
    cfg = f3dc.config_for(shape, 1)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    f3dc.set_fault_injection(fail_alloc_at=n)
    try:
        for _ in range(3):
            with pytest.raises(f3dc.F3dcError) as e:
                f3dc.Handle(cfg, blob)
            assert e.value.status == 3, e.value
    finally:
        f3dc.set_fault_injection()
    torch.cuda.synchronize()
    # what the failed calls allocated was freed (driver granularity aside)
    assert free0 - torch.cuda.mem_get_info()[0] < 8 << 20
    _tiny_step_clean()


@pytest.mark.parametrize("nq,H", [(256, 2), (2600, 8)])
def test_attention_wait_runs_out_and_is_reported(orc, nq, H):
    # the attention kernel's first CTA is told to skip the load of its first
    # item's last key tile (the earlier tiles go through): the MMA issuer's
    # and then the softmax warps' bounded waits run out (1 s, the others
    # seeing the abort flag), every warp leaves its work loop, the kernel
    # returns and the timeout is reported; the next call computes the right
    # result.  256 queries x 2 heads run the one-tile kernel, 2600 x 8 (168
    # tile-head items on 152 SMs) the pair kernel.
    nk, dh = 512, 64
    W = H * dh
    g = np.random.default_rng(3)
    q = synth.f32_to_bf16_bits(g.standard_normal((nq, W)).astype(np.float32))
    kv = synth.f32_to_bf16_bits(g.standard_normal((nk, 2 * W)).astype(np.float32))
    qd, kvd = dev_bf16(q), dev_bf16(kv)
    out = torch.zeros((nq, W), dtype=torch.bfloat16, device="cuda")
    assert f3dc.gemm_status() == 0
    f3dc.set_fault_injection(attn_missing_kv=1)
    try:
        t0 = time.perf_counter()
        f3dc.attention(qd, W, kvd, kvd[:, W:], 2 * W, out, nq, nk, H, dh)
        st = f3dc.gemm_status()
        elapsed = time.perf_counter() - t0
    finally:
        f3dc.set_fault_injection()
    assert st & TIMEOUT, st
    assert elapsed < 10.0
    out.zero_()
    f3dc.attention(qd, W, kvd, kvd[:, W:], 2 * W, out, nq, nk, H, dh)
    assert f3dc.gemm_status() == 0
    kf = synth.bf16_bits_to_f32(kv)
    ref = orc.attention(synth.bf16_bits_to_f32(q), kf[:, :W], kf[:, W:], H).astype(np.float64)
    got = out.float().cpu().numpy()
    assert np.max(np.abs(got - ref)) < 2e-2
    _tiny_step_clean()
