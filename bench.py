"""Benchmark of the Fast3Dcache cached denoising step on GB300.

Workload (the configuration the headline metric is quoted on): a
TRELLIS-L-shaped sparse-structure flow transformer -- 16^3 x 8 latent (4096
tokens), width 1024, 24 blocks, 16 heads, MLP 4x, cross-attention to 1374
condition tokens of dim 1024, bf16 tensor-core arithmetic with fp32
accumulation, 25 Euler steps with the three-phase PCSC schedule and the
paper's default hyperparameters, batch 1 per GPU, random-init weights,
seeded N(0,1) latents and condition tokens.  The anchor measurement sigma is
fixed at 65536 dynamic voxels (25% of the 64^3 occupancy grid) so the active
counts follow a TRELLIS-like budget; the stand-in decoder's own dynamic-voxel
count is still computed at the anchor step in every sample.

One benchmark step = one full sample (all 25 denoising steps: selection,
transformer on the active tokens, merge + Euler, the anchor's voxel count).
value = denoising steps per second over all GPUs.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl f3dc|reference]

--impl reference times the CPU oracle (the plain C restatement of the
paper) on the host cores instead, on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2511_22533_gb300 import synth  # noqa: E402

METRIC = "cached denoise steps/s at PCSC quota (1 GB300); tensor-pipe % of bf16 peak"
UNIT = "steps/s"
WORKLOAD = "trellis_l"
CFG_STRENGTH = 5.0  # guidance strength of the secondary CFG measurement (the work does not depend on it)
SIGMA = 65536.0
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# DRAM traffic of the GEMM family, from one ncu capture of the six projections
# of a 1229-row cached-step block (profiles/k_gemm_pair_cached_step_1229rows.md):
# 68.9 MB over 6 launches against 67.1 MB of operand bytes.  Valid only for the
# kernel source it was taken on (sha256 of csrc/k_gemm.cu); null otherwise.
GEMM_TRAFFIC = {"dram_bytes_per_launch": 68.9e6 / 6, "algorithmic_bytes_per_launch": 67.1e6 / 6,
                "shape": "QKV, attention out, cross Q, cross out, fc1, fc2 at 1229 active rows, width 1024",
                "profile": "profiles/k_gemm_pair_cached_step_1229rows.md",
                "k_gemm_cu_sha256": "d080472e424c0a678d801a1a68e8872efd72620b4b902365757673d2778e0f3e"}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="f3dc", choices=["f3dc", "reference"])
    return p.parse_args()


def gemm_traffic(path=None):
    """The captured GEMM traffic per launch, or None once k_gemm.cu (or the
    file at `path`) differs from the source the counters were taken on."""
    import hashlib
    if path is None:
        path = os.path.join(ROOT, "paper_2511_22533_gb300", "csrc", "k_gemm.cu")
    try:
        with open(path, "rb") as f:
            sha = hashlib.sha256(f.read()).hexdigest()
    except OSError:
        return None
    return GEMM_TRAFFIC if sha == GEMM_TRAFFIC["k_gemm_cu_sha256"] else None


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    except Exception:
        return FALLBACK_PEAKS, "fallback"


# ------------------------------------------------------------------ work model

def block_matmul_flops(a: int, W: int, Nc: int) -> float:
    """Tensor-core FLOPs of one block on a active tokens (Supp. Sec. F terms
    that are matrix products): QKV 6aW^2, out 2aW^2, CA-Q 2aW^2, CA-out
    2aW^2, MLP 16aW^2, QK^T + PV 4a^2W, cross QK^T + PV 4aN_cW."""
    return 28.0 * a * W * W + 4.0 * a * a * W + 4.0 * a * Nc * W


def paper_block_flops(a: int, W: int, Nc: int, H: int, B: int = 1) -> float:
    """The paper's per-block FLOPs count (Supp. Sec. F), N_tok = a."""
    mod = 5 * B * W + 2 * B * W * 6 * W
    ln = 7 * B * a * W
    sa = 8 * B * a * W * W + 4 * B * a * a * W + 5 * B * H * a * a
    ca = 4 * B * a * W * W + 4 * B * Nc * W * W + 4 * B * a * Nc * W + 5 * B * H * a * Nc
    mlp = 16 * B * a * W * W + 20 * B * a * W
    return mod + 3 * ln + sa + ca + mlp


def sample_flops(quota_log, shape, guided=None):
    """Tensor-core and paper FLOPs of one call of the sampler: quota_log
    [T, B] holds each sample's cache quota per step (attention runs per
    sample, so its a_b^2 term is summed per sample); guided[k] marks the
    steps that run the transformer twice (classifier-free guidance)."""
    N, W, L, Nc, H = shape.tokens, shape.width, shape.blocks, shape.cond_tokens, shape.heads
    q = np.asarray(quota_log).reshape(len(quota_log), -1)
    mm = paper = 0.0
    for k in range(q.shape[0]):
        reps = 2 if guided is not None and guided[k] else 1
        for c in q[k]:
            a = N - int(c)
            if a > 0:
                mm += reps * L * block_matmul_flops(a, W, Nc)
                paper += reps * L * paper_block_flops(a, W, Nc, H)
    mm += q.shape[1] * L * 2.0 * Nc * (2 * W) * shape.cond_dim  # condition K / V, once per sample
    return mm, paper


# ------------------------------------------------------------------ ranks

def rank_seed(rank: int) -> int:
    """Each rank samples its own latents and condition (independent samples)."""
    return 100 + rank


def max_over_ranks(ms: float, world: int, device="cpu") -> float:
    """The slowest rank's elapsed time (the whole job ends with it)."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_throughput(steps_per_sample: int, samples_per_rank: int, world: int, max_ms: float) -> float:
    """Denoising steps per second over all ranks (weak scaling: every rank
    runs its own samples)."""
    return steps_per_sample * samples_per_rank * world / (max_ms / 1000.0)


# ------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons, n = [], [], set(), 0
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                n += 1
                for name, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(name)
        os.unlink(self.path)
        loaded = [s for s in sm if mx and s > 0.5 * max(mx)] or sm
        return {"sm_mhz": statistics.median(loaded) if loaded else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons), "samples": n}


# ------------------------------------------------------------------ oracle leg

def oracle_bounded_sample(orc, quota_log):
    """Times the CPU oracle on a bounded sample of the workload and
    extrapolates the whole 25-step sample: one transformer block (of 24) at
    1229 and at 4096 active tokens (the Phase-3 cached and the full steps), the SSC score + selection and the merge /
    Euler update at N = 4096, and the condition K / V of one block.  Block
    time is interpolated linearly in FLOPs between the two measurements."""
    shape = synth.SHAPES[WORKLOAD]
    one = synth.ModelShape(shape.grid, shape.channels, shape.width, 1, shape.heads, shape.mlp_ratio,
                           shape.cond_tokens, shape.cond_dim, shape.steps, shape.gamma_up)
    blob = synth.weights_blob(one, 0)
    m = orc.Model(one, blob)
    cond = synth.cond_tokens(one, 1, 0)
    S = synth.latents(one, 1, 0)[0]
    hist = synth.velocity_history(shape.grid, 8, 1, seed=1)
    t0 = time.perf_counter()
    kv = m.cond_kv(cond[0])
    t_kv = time.perf_counter() - t0
    pts = []
    for a in (1229, 4096):
        idx = np.arange(a, dtype=np.int32)
        t0 = time.perf_counter()
        m.forward(S, idx, 0.9, kv)
        pts.append((block_matmul_flops(a, shape.width, shape.cond_tokens), time.perf_counter() - t0))
    t0 = time.perf_counter()
    s = orc.ssc_score(hist[2, 0], hist[1, 0], 0.7)
    cached, idx = orc.select(s, 3141)
    t_sel = time.perf_counter() - t0
    va = np.zeros((len(idx), 8), np.float32)
    t0 = time.perf_counter()
    orc.merge_euler(S, idx, va, hist[2, 0], 0.01)
    t_merge = time.perf_counter() - t0
    (f0, s0), (f1, s1) = pts
    slope = (s1 - s0) / (f1 - f0)
    total = shape.blocks * t_kv
    for c in quota_log[:, 0]:
        a = shape.tokens - int(c)
        if a > 0:
            total += shape.blocks * max(s0 + slope * (block_matmul_flops(a, shape.width, shape.cond_tokens) - f0), 0.0)
        if c > 0:
            total += t_sel
        total += t_merge
    measured = t_kv + s0 + s1 + t_sel + t_merge
    return shape.steps / total, measured


def quota_log_host():
    """The effective cache quotas of one benchmark sample (host-only logic
    of the oracle: phases, PCSC with sigma = 65536, tau = 3)."""
    import oracle
    shape = synth.SHAPES[WORKLOAD]
    gate = oracle.TauGate(3, 0)
    q = []
    for k in range(1, shape.steps + 1):
        c, _ = oracle.phase_quota(shape.tokens, shape.steps, 0.2, 0.75, -0.07, 0.7, 3, shape.gamma_up, SIGMA, k)
        q.append(gate(c))
    return np.array(q, np.int32)[:, None]


def hbm_kernels_b64(f3dc, torch, blob_d, pk):
    """The HBM-bound kernels of the step at batch 64, half of each sample's
    tokens cached, L2 flushed before each measurement, on the benchmark's
    16^3 x 8 grid (the TRELLIS-L model) and on the 32^3 x 8 grid (a width-128,
    one-block model: these kernels do not depend on the transformer, except
    the gather's output width).  The SSC selection alone through
    f3dc_ssc_select (median of 20 calls, CUDA events around each call), and
    the gather/embed and merge/Euler kernels from one profiled f3dc_step.
    Bytes are the algorithmic ones (selection: 33 B per token + 4 B per active
    index; gather: 36 + 4W B per active token; merge: 96 B per token + 32 B
    per active token)."""
    out = {}
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device="cuda")  # 256 MB > L2
    small32 = synth.ModelShape(32, 8, 128, 1, 4, 4, 64, 128, 50, 64)
    for key, shape, blob in (("grid16", synth.SHAPES[WORKLOAD], blob_d),
                             ("grid32", small32, None)):
        B, N = 64, shape.tokens
        if blob is None:
            blob = torch.from_numpy(synth.weights_blob(shape, 0).view(np.int16)).cuda()
        cfg = f3dc.config_for(shape, B)
        h = f3dc.Handle(cfg, blob)
        hist = synth.velocity_history(shape.grid, shape.channels, B, seed=11)
        ring = torch.from_numpy(hist.view(np.int16)).cuda()
        quota = torch.full((B,), N // 2, dtype=torch.int32, device="cuda")
        idx = torch.empty((B, N), dtype=torch.int32, device="cuda")
        nact = torch.empty((B,), dtype=torch.int32, device="cuda")
        mask = torch.empty((B, N), dtype=torch.uint8, device="cuda")
        times = []
        for i in range(23):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            h.ssc_select(ring[2], ring[1], B, quota, idx, nact, mask)
            e1.record()
            torch.cuda.synchronize()
            if i >= 3:
                times.append(e0.elapsed_time(e1))
        ms = float(np.median(times))
        sel_bytes = B * N * 33 + B * (N - N // 2) * 4
        d = {"workload": f"batch {B} x {N} tokens ({shape.grid}^3 x 8), {N // 2} cached per sample, width "
                         f"{shape.width}, L2 flushed",
             "ssc_select": {"us": ms * 1000.0, "bytes": sel_bytes, "gbs": sel_bytes / (ms / 1000.0) / 1e9}}
        d["ssc_select"]["frac_hbm"] = d["ssc_select"]["gbs"] / pk["hbm_gbs"]
        # one profiled step: gather/embed and merge/Euler at batch 64
        cond = torch.from_numpy(np.ascontiguousarray(np.broadcast_to(
            synth.cond_tokens(shape, 1, 3), (B, shape.cond_tokens, shape.cond_dim))).view(np.int16)).cuda()
        h.set_cond(cond, B)
        S = torch.from_numpy(synth.latents(shape, B, 5)).cuda()
        k = 8  # a cached step: history slots k-1, k-2 hold the drift history
        ring_k = torch.empty_like(ring)
        ring_k[(k - 1) % 3] = ring[2]
        ring_k[(k - 2) % 3] = ring[1]
        ring_k[k % 3] = ring[0]
        torch.cuda.synchronize()
        flush.zero_()
        h.profile(True)
        h.step(k, B, S, ring_k, quota)
        torch.cuda.synchronize()
        stats = {st["name"]: st for st in h.profile_read()}
        h.profile(False)
        for name in ("gather_embed", "merge_euler"):
            st = stats.get(name)
            if st and st["total_ms"] > 0:
                d[name] = {"us": st["total_ms"] * 1000.0 / max(st["launches"], 1), "bytes": st["bytes"],
                           "gbs": st["bytes"] / (st["total_ms"] / 1000.0) / 1e9}
                d[name]["frac_hbm"] = d[name]["gbs"] / pk["hbm_gbs"]
        assert h.device_status() == 0
        h.close()
        del ring, ring_k, S, cond
        out[key] = d
    del flush
    return out


def other_configs(f3dc, torch, blob_d, pk, timed, warmup):
    """Throughput of the other workloads of the benchmark suite (secondary;
    not part of `value`), each through f3dc_sample with inputs resident:
      tiny     8^3 x 8 latent, width 128, 2 blocks, 4 heads, 64 x 128
               condition, T = 8, quota 0 for steps 1-2 then 256 of 512
               cached (tau off), batch 1
      ragged8  the TRELLIS-L model at batch 8 with per-sample PCSC budgets:
               sigma_b = a_b gamma_up e^(-mu), so that the first Phase-2
               step keeps a_b ~ U[400, 4096] tokens active (seed 0)
      scaled32 the same model on a 32^3 x 8 latent (32768 tokens), T = 50,
               cache quota ramped linearly from 0 to 80 % of the tokens
               (c_k = floor(0.8 N (k - 1) / (T - 1))) with the tau = 3 rule
    Reported per leg: denoising steps/s (steps of every sample), samples/s,
    and the tensor-core work rate against the sustained bf16 peak."""
    out = {}

    def leg(name, shape, B, blob, quota_schedule=None, sigma=None, n_timed=3, n_warm=1, **hyper):
        cfg = f3dc.config_for(shape, B, **hyper)
        h = f3dc.Handle(cfg, blob)
        noise = torch.from_numpy(synth.latents(shape, B, 200)).cuda()
        cond = torch.from_numpy(synth.cond_tokens(shape, B, 200).view(np.int16)).cuda()
        S = torch.empty_like(noise)

        def run(want_log=False):
            S.copy_(noise)
            return h.sample(S, cond, B, sigma_override=sigma, quota_schedule=quota_schedule, want_log=want_log)

        qlog, _ = run(True)
        for _ in range(max(n_warm - 1, 0)):
            run()
        ms = timed(n_timed, run) / n_timed
        assert h.device_status() == 0
        h.close()
        mm, paper = sample_flops(qlog, shape)
        act = (shape.tokens - qlog).tolist()
        out[name] = {"batch": B, "euler_steps": shape.steps, "ms_per_batch_sample": ms,
                     "steps_per_s": shape.steps * B / (ms / 1000.0), "samples_per_s": B / (ms / 1000.0),
                     "tensor_tflops": mm / (ms / 1000.0) / 1e12,
                     "frac_bf16_sustained": mm / (ms / 1000.0) / 1e12 / pk["bf16_tflops_sustained"],
                     "paper_flops_per_batch_T": paper / 1e12,
                     "active_tokens_per_step": act if B > 1 else [a[0] for a in act]}

    tiny = synth.SHAPES["tiny"]
    tiny_blob = torch.from_numpy(synth.weights_blob(tiny, 0).view(np.int16)).cuda()
    q_tiny = np.zeros((tiny.steps, 1), np.int32)
    q_tiny[2:] = tiny.tokens // 2
    leg("tiny", tiny, 1, tiny_blob, quota_schedule=q_tiny, n_timed=20, n_warm=max(warmup, 3), tau=0)
    del tiny_blob

    shape = synth.SHAPES[WORKLOAD]
    targets = synth.ragged_active_targets(8, shape.tokens, 400, 4096, seed=0)
    sig8 = targets.astype(np.float64) * shape.gamma_up * np.exp(0.07)
    leg("ragged8", shape, 8, blob_d, sigma=sig8, n_timed=3, n_warm=1)
    out["ragged8"]["target_active_first_phase2"] = [int(a) for a in targets]

    sc = synth.SHAPES["scaled"]
    ramp = np.floor(0.8 * sc.tokens * np.arange(sc.steps) / (sc.steps - 1)).astype(np.int32)[:, None]
    leg("scaled32", sc, 1, blob_d, quota_schedule=ramp, n_timed=1, n_warm=1)
    return out


def gpu_step_times(f3dc, torch, h, shape, timed):
    """One standalone f3dc_step (selection, modulation GEMVs, transformer,
    merge) of the benchmark model at the Phase-3 cached quota (2867 cached,
    1229 active) and at quota 0 (4096 active), inputs resident, 20 steps
    each -- the GPU side of the per-step CPU comparison."""
    N = shape.tokens
    hist = synth.velocity_history(shape.grid, shape.channels, 1, seed=31)
    ring0 = np.zeros((3, 1, N, shape.channels), np.uint16)
    out = {}
    for name, q, k in (("cached_1229_active", 2867, 19), ("full_4096_active", 0, 1)):
        ring0[(k - 1) % 3], ring0[(k - 2) % 3] = hist[2], hist[1]
        ring = torch.from_numpy(ring0.view(np.int16)).cuda()
        quota = torch.tensor([q], dtype=torch.int32, device="cuda")
        S = torch.from_numpy(synth.latents(shape, 1, 300)).cuda()
        for _ in range(3):
            h.step(k, 1, S, ring, quota)
        ms = timed(20, lambda: h.step(k, 1, S, ring, quota)) / 20
        out[name] = {"ms": ms, "active": N - q}
    return out


def oracle_step(orc, blob, quota, k=19):
    """Times one complete cached step of the benchmark workload on the CPU
    oracle (host cores, OpenMP over rows): SSC score and selection, the
    24-block transformer on the active tokens, merge and Euler update.  The
    condition K / V (step-invariant, once per sample) are timed apart."""
    shape = synth.SHAPES[WORKLOAD]
    m = orc.Model(shape, blob)
    cond = synth.cond_tokens(shape, 1, 0)
    S = synth.latents(shape, 1, 0)[0]
    hist = synth.velocity_history(shape.grid, shape.channels, 1, seed=1)
    t = orc.time_schedule(shape.steps, 3.0)
    t0 = time.perf_counter()
    kv = m.cond_kv(cond[0])
    t_kv = time.perf_counter() - t0
    t0 = time.perf_counter()
    s = orc.ssc_score(hist[2, 0], hist[1, 0], 0.7)
    _, idx = orc.select(s, quota)
    va = m.forward(S, idx, float(t[k - 1]), kv)
    orc.merge_euler(S, idx, va, hist[2, 0], float(t[k - 1] - t[k]))
    return time.perf_counter() - t0, t_kv, len(idx)


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    os.environ.setdefault("OMP_NUM_THREADS", str(threads))
    qlog = quota_log_host()
    for _ in range(args.warmup):
        oracle_bounded_sample(oracle, qlog)
    vals, cpu_s = [], 0.0
    for _ in range(args.steps):
        v, meas = oracle_bounded_sample(oracle, qlog)
        vals.append(v)
        cpu_s += meas
    value = statistics.median(vals)
    sample = ("per step: 1 of 24 transformer blocks at 1229 and 4096 active tokens, SSC score + selection "
              "and merge/Euler at N=4096, condition K/V of one block; whole 25-step sample extrapolated "
              "by FLOPs (blocks x interpolated block time over the PCSC quota schedule)")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * shape_steps() / value,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": config_block(args),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "cpu_seconds_measured": cpu_s,
            "measured_ms_per_bounded_sample": 1000.0 * cpu_s / max(args.steps, 1),
            "projection": "value and ms_per_step are the whole 25-step sample extrapolated by FLOPs from the "
                          "bounded sample timed each step (measured_ms_per_bounded_sample)"}
    print(json.dumps(line))
    return 0


def shape_steps():
    return synth.SHAPES[WORKLOAD].steps


def config_block(args):
    shape = synth.SHAPES[WORKLOAD]
    return {"workload": "TRELLIS-L-shaped sparse-structure flow DiT: 16^3x8 latent (4096 tokens), width 1024, "
                        "24 blocks, 16 heads, MLP 4x, cross-attn to 1374 cond tokens dim 1024, bf16, 25 Euler "
                        "steps, PCSC schedule (sigma 65536, mu -0.07, tau 3, xi 0.7, f_corr 3), batch 1 per GPU, "
                        "random-init weights",
            "tokens": shape.tokens, "width": shape.width, "blocks": shape.blocks, "heads": shape.heads,
            "cond_tokens": shape.cond_tokens, "euler_steps": shape.steps, "batch_per_gpu": 1,
            "global_batch": args.gpus, "sigma": SIGMA,
            "l2": "inputs larger than L2: ~1.1 GB of weights streamed per denoising step",
            "parallelism": f"replicas x{args.gpus} (independent samples per GPU)"}


# ------------------------------------------------------------------ GPU arm

def run_gpu(args):
    import torch
    import torch.distributed as dist

    from paper_2511_22533_gb300 import f3dc

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("nccl", rank=rank, world_size=world)
    if local == 0:
        f3dc.lib()
    if world > 1:
        dist.barrier()
    L = f3dc.lib()
    shape = synth.SHAPES[WORKLOAD]
    pk, pk_src = peaks()

    blob = synth.weights_blob(shape, 0)
    blob_d = torch.from_numpy(blob.view(np.int16)).cuda()
    cfg = f3dc.config_for(shape, 1)
    h = f3dc.Handle(cfg, blob_d)
    noise = synth.latents(shape, 1, rank_seed(rank))
    cond_np = synth.cond_tokens(shape, 1, rank_seed(rank))
    noise_d = torch.from_numpy(noise).cuda()
    cond_d = torch.from_numpy(cond_np.view(np.int16)).cuda()
    S = torch.empty_like(noise_d)
    sig = np.array([SIGMA])

    def one_sample(quota_schedule=None, want_log=False):
        S.copy_(noise_d)
        return h.sample(S, cond_d, 1, sigma_override=sig, quota_schedule=quota_schedule, want_log=want_log)

    # warm-up (the first also returns the quota log that defines the work)
    qlog, sigma_meas = one_sample(want_log=True)
    for _ in range(max(args.warmup - 1, 0)):
        one_sample()
    torch.cuda.synchronize()
    assert h.device_status() == 0
    mm_flops, paper_flops = sample_flops(qlog, shape)

    def timed(n, fn):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(n):
            fn()
        e1.record()
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        return max_over_ranks(e0.elapsed_time(e1), world, device="cuda")

    # ---- headline: cached sampler, device-resident inputs
    n0 = h.launch_count()
    clocks = ClockSampler(local)
    clocks.start()
    ms = timed(args.steps, one_sample)
    clk = clocks.stop()
    launches = h.launch_count() - n0
    ms_per_sample = ms / args.steps
    value = whole_job_throughput(shape.steps, args.steps, world, ms)

    # ---- uncached comparison: the same kernels with quota 0 at every step
    zeros = np.zeros((shape.steps, 1), np.int32)
    one_sample(zeros)
    n_unc = max(2, args.steps // 2)
    ms_unc = timed(n_unc, lambda: one_sample(zeros)) / n_unc
    zlog = zeros
    mm_unc, _ = sample_flops(zlog, shape)

    # ---- per-kernel CUDA-event timing of the same workload
    h.profile(True)
    n_prof = max(2, args.steps // 4)
    for _ in range(n_prof):
        one_sample()
    stats = h.profile_read()
    h.profile(False)

    # ---- end to end through the public API with host buffers
    import torch as _t
    noise_h = _t.from_numpy(noise).pin_memory()
    cond_h = _t.from_numpy(cond_np.view(np.int16)).pin_memory()
    out_h = _t.empty_like(noise_h).pin_memory()
    cond_e = _t.empty_like(cond_d)

    def e2e_sample():
        S.copy_(noise_h, non_blocking=True)
        cond_e.copy_(cond_h, non_blocking=True)
        h.sample(S, cond_e, 1, sigma_override=sig, want_log=False)
        out_h.copy_(S, non_blocking=True)

    e2e_sample()
    ms_e2e = timed(args.steps, e2e_sample)
    e2e_value = whole_job_throughput(shape.steps, args.steps, world, ms_e2e)
    assert h.device_status() == 0

    # ---- classifier-free guidance over the interval [0.5, 1] (secondary; not
    # part of `value`): the same workload with every step whose t_k >= 0.5 run
    # for the condition and the zero condition on the same active tokens
    cfg_g = f3dc.config_for(shape, 1, cfg_strength=CFG_STRENGTH, cfg_t_lo=0.5)
    hg = f3dc.Handle(cfg_g, blob_d)

    def guided_sample():
        S.copy_(noise_d)
        hg.sample(S, cond_d, 1, sigma_override=sig, want_log=False)

    for _ in range(max(args.warmup, 1)):
        guided_sample()
    n_g = max(2, args.steps // 2)
    ms_g = timed(n_g, guided_sample) / n_g
    assert hg.device_status() == 0
    hg.close()
    t_sched = f3dc.time_schedule(cfg_g)
    guided = [float(t_sched[k]) >= 0.5 for k in range(shape.steps)]
    mm_g, paper_g = sample_flops(qlog, shape, guided)
    cfg_line = {"strength": CFG_STRENGTH, "interval": [0.5, 1.0], "guided_steps": int(sum(guided)),
                "ms_per_sample": ms_g, "steps_per_s": shape.steps * world / (ms_g / 1000.0),
                "tensor_tflops_per_gpu": mm_g / (ms_g / 1000.0) / 1e12,
                "paper_flops_per_sample_T": paper_g / 1e12}

    # ---- the convolutional stand-in decoder of Eq. 1 (secondary): one sample
    # measuring sigma at the anchor step, the decoder's launches timed
    hd = f3dc.Handle(f3dc.config_for(shape, 1, decoder=1), blob_d)
    S.copy_(noise_d)
    hd.sample(S, cond_d, 1, want_log=False)
    hd.profile(True)
    S.copy_(noise_d)
    _, sig_conv = hd.sample(S, cond_d, 1)
    dstats = {st["name"]: st for st in hd.profile_read()}
    hd.profile(False)
    assert hd.device_status() == 0
    hd.close()
    dst = dstats.get("decode_conv")
    dec_line = None
    if dst and dst["launches"] > 0:
        per_decode = dst["total_ms"] / dst["launches"]  # one profiled entry (three kernels) per decode
        dec_line = {"grid_out": [4 * shape.grid] * 3, "decodes_per_sample": int(dst["launches"]),
                    "ms_per_decode": per_decode, "gflops": dst["flops"] / (dst["total_ms"] / 1000.0) / 1e9,
                    "sigma_measured": float(sig_conv[0])}

    # ---- data-driven PCSC slope (secondary): the dynamic-voxel curve of one
    # uncached run with the linear stand-in decoder, fitted over steps 8..18
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    curve = h.dynamic_voxel_curve(S.copy_(noise_d), cond_d, 1)
    curve_ms = (time.perf_counter() - t0) * 1000.0
    mu_fit, _, kept_fit = f3dc.fit_mu(curve.T.astype(np.float64))
    mu_line = {"curve_ms": curve_ms, "curve": [int(x) for x in curve[:, 0]], "steps_fitted": [8, 18],
               "mu": None if not np.isfinite(mu_fit) else float(mu_fit), "kept": bool(kept_fit[0])}

    # ---- the HBM-bound kernels at batch 64 (secondary; not part of `value`)
    hbm64 = hbm_kernels_b64(f3dc, torch, blob_d, pk) if rank == 0 else None

    # ---- the other workloads (tiny, batch 8 ragged, 32^3 scaled; secondary)
    others = other_configs(f3dc, torch, blob_d, pk, timed, args.warmup)
    del blob_d

    # ---- one standalone step of each kind on the GPU (the CPU comparison's pair)
    per_step = gpu_step_times(f3dc, torch, h, shape, timed)
    assert h.device_status() == 0

    # ---- CPU baseline (oracle on the host cores), rank 0 at N = 1 only: one
    # complete cached step measured; the whole-sample figure extrapolated from
    # a bounded sample is reported apart
    cpu = None
    if world == 1 and rank == 0:
        import oracle
        oracle.build()
        t_step, t_kv, n_act = oracle_step(oracle, blob, 2867)
        v_ext, meas = oracle_bounded_sample(oracle, qlog)
        cpu = {"value": 1.0 / t_step, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"one complete cached denoising step of the workload measured on the oracle (step 19, "
                         f"2867 of 4096 tokens cached, {n_act} active, all 24 blocks: SSC score + selection, "
                         f"transformer, merge/Euler) in {t_step:.1f} s; value = 1 / that time",
               "measured_step_s": t_step, "cond_kv_once_per_sample_s": t_kv,
               "gpu_same_step_ms": per_step["cached_1229_active"]["ms"],
               "extrapolated_whole_sample_steps_per_s": v_ext,
               "extrapolation": f"1 of 24 blocks at 1229 and 4096 active tokens + SSC/selection + merge "
                                f"({meas:.1f} s measured), the 25-step schedule's blocks interpolated by FLOPs"}

    if rank != 0:
        h.close()
        if world > 1:
            dist.destroy_process_group()
        return 0

    tensor_tflops = mm_flops / (ms_per_sample / 1000.0) / 1e12
    fam = {s["name"]: s for s in stats}
    dom = max(stats, key=lambda s: s["total_ms"])
    if dom["flops"] > 0:
        peak = pk["bf16_tflops_sustained"]
        achieved = dom["flops"] / (dom["total_ms"] / 1000.0) / 1e12
        roof = {"kernel": dom["name"], "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "traffic": None, "peak_source": f"bf16_tflops_sustained ({pk_src})"}
        gt = gemm_traffic() if dom["name"] == "gemm" else None
        if gt:
            roof["traffic"] = gt["dram_bytes_per_launch"]
            roof["traffic_note"] = (f"ncu dram__bytes_read + write per launch of {gt['shape']} "
                                    f"({gt['profile']}); algorithmic operand bytes "
                                    f"{gt['algorithmic_bytes_per_launch']:.4g} per launch")
    else:
        peak = pk["hbm_gbs"]
        achieved = dom["bytes"] / (dom["total_ms"] / 1000.0) / 1e9
        roof = {"kernel": dom["name"], "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": None, "peak_source": f"hbm_gbs ({pk_src})"}
    kernels = {}
    for s in stats:
        per = s["total_ms"] / n_prof
        entry = {"launches_per_sample": s["launches"] / n_prof, "ms_per_sample": per}
        if s["flops"] > 0:
            entry["tflops"] = s["flops"] / (s["total_ms"] / 1000.0) / 1e12
            entry["frac_bf16_sustained"] = entry["tflops"] / pk["bf16_tflops_sustained"]
        if s["bytes"] > 0:
            entry["gbs"] = s["bytes"] / (s["total_ms"] / 1000.0) / 1e9
            entry["frac_hbm"] = entry["gbs"] / pk["hbm_gbs"]
        kernels[s["name"]] = entry

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_sample,
        "step_unit": "one benchmark step = one 25-step sample (every denoising step of one batch-1 sample)",
        "ms_per_denoising_step": ms_per_sample / shape.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": config_block(args),
        "samples_per_s": args.steps * world / (ms / 1000.0),
        "tensor_pct_of_bf16_sustained": 100.0 * tensor_tflops / pk["bf16_tflops_sustained"],
        "tensor_tflops_per_gpu": tensor_tflops,
        "paper_flops_per_sample_T": paper_flops / 1e12,
        "uncached": {"ms_per_sample": ms_unc, "steps_per_s": shape.steps * world / (ms_unc / 1000.0),
                     "speedup_cached_vs_uncached": ms_unc / ms_per_sample,
                     "tensor_tflops_per_gpu": mm_unc / (ms_unc / 1000.0) / 1e12},
        "active_tokens_per_step": [shape.tokens - int(c) for c in qlog[:, 0]],
        "sigma_measured_by_stand_in_decoder": float(sigma_meas[0]),
        "roofline": roof, "kernels": kernels, "hbm_kernels_b64": hbm64, "cfg": cfg_line, "decoder_conv": dec_line, "mu_fit": mu_line,
        "configs": others, "standalone_step": per_step,
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(noise.nbytes + cond_np.nbytes),
                "d2h_bytes_per_step": int(noise.nbytes),
                "bytes_per": "benchmark step (one 25-step sample: latents + condition in, S_0 out)"},
        "gpu_launches": int(launches),
        "clocks": clk,
    }
    print(json.dumps(line))
    h.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
