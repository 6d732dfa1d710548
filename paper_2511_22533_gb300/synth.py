"""Seeded synthetic inputs for the Fast3Dcache cached denoising step.

This module is shared by the CUDA path's tests/bench and by the CPU oracle's
tests.  It draws random numbers and lays them out in the documented formats;
it holds none of the method's arithmetic (no score, no quota, no transformer
math).  Every generator uses NumPy PCG64 ``default_rng(seed * 1000 + b)`` for
sample ``b``.

Workloads (stand-ins for TRELLIS stage 1 on Toys4K, Sec. 5.1; the datasets,
the TRELLIS weights and DINOv2 are not available, so latents are N(0,1),
condition tokens are N(0,1) DINOv2-shaped tokens and weights are
random-init):

* ``tiny``      8^3 x 8 latent (512 tokens), width 128, 2 blocks, 4 heads,
                64 condition tokens of dim 128, T = 8.
* ``trellis_l`` 16^3 x 8 latent (4096 tokens), width 1024, 24 blocks,
                16 heads, 1374 condition tokens of dim 1024, T = 25.
* ``scaled``    32^3 x 8 latent (32768 tokens), same transformer, T = 50.

Weight blob (layout version 2): every tensor is bf16, row-major
``[out_features, in_features]`` for linear layers, concatenated in the order
returned by :func:`weight_layout`, each tensor starting at a multiple of 64
elements (128 bytes).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

LAYOUT_VERSION = 2
ALIGN_ELEMS = 64


@dataclasses.dataclass(frozen=True)
class ModelShape:
    grid: int          # cubic latent grid side D (tokens N = D^3)
    channels: int      # latent channels C
    width: int         # transformer width W
    blocks: int        # transformer blocks L
    heads: int         # attention heads H
    mlp_ratio: int     # MLP hidden = mlp_ratio * W
    cond_tokens: int   # condition tokens N_c
    cond_dim: int      # condition dim D_c
    steps: int         # Euler steps T
    gamma_up: int      # decoder sub-voxels per latent token

    @property
    def tokens(self) -> int:
        return self.grid ** 3


SHAPES = {
    "tiny": ModelShape(8, 8, 128, 2, 4, 4, 64, 128, 8, 64),
    "trellis_l": ModelShape(16, 8, 1024, 24, 16, 4, 1374, 1024, 25, 64),
    "scaled": ModelShape(32, 8, 1024, 24, 16, 4, 1374, 1024, 50, 64),
}


def _rng(seed: int, b: int = 0) -> np.random.Generator:
    return np.random.default_rng(seed * 1000 + b)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (round-to-nearest-even) and return the raw uint16 bits.

    NaN stays NaN (quiet); this is a storage-format conversion only.
    """
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    rounding = ((u >> 16) & 1) + 0x7FFF
    out = ((u + rounding) >> 16).astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(u: np.ndarray) -> np.ndarray:
    u = np.ascontiguousarray(u, dtype=np.uint16)
    return (u.astype(np.uint32) << 16).view(np.float32)


# --------------------------------------------------------------------------
# latents and condition tokens
# --------------------------------------------------------------------------

def latents(shape: ModelShape, batch: int, seed: int) -> np.ndarray:
    """Initial noise grid S_eps, token-major fp32 [B, N, C] with token index
    i = (d * D + h) * D + w."""
    out = np.empty((batch, shape.tokens, shape.channels), np.float32)
    for b in range(batch):
        out[b] = _rng(seed, b).standard_normal((shape.tokens, shape.channels), dtype=np.float32)
    return out


def cond_tokens(shape: ModelShape, batch: int, seed: int) -> np.ndarray:
    """DINOv2-shaped stand-in condition tokens, bf16 bits [B, N_c, D_c]."""
    out = np.empty((batch, shape.cond_tokens, shape.cond_dim), np.uint16)
    for b in range(batch):
        g = _rng(seed + 7, b).standard_normal((shape.cond_tokens, shape.cond_dim), dtype=np.float32)
        out[b] = f32_to_bf16_bits(g)
    return out


# --------------------------------------------------------------------------
# weight blob
# --------------------------------------------------------------------------

def weight_layout(shape: ModelShape):
    """List of (name, block, dims, init) in blob order.  ``block`` is -1 for
    global tensors.  ``init`` is one of 'w' (N(0, 1/fan_in)), 'b'
    (0.02 N(0,1)), 'g' (1 + 0.1 N(0,1)), 'dec' (N(0,1))."""
    W, C, Dc, G = shape.width, shape.channels, shape.cond_dim, shape.gamma_up
    Wm = shape.mlp_ratio * W
    items = [
        ("in_w", -1, (W, C), "w"), ("in_b", -1, (W,), "b"),
        ("t_w1", -1, (W, 256), "w"), ("t_b1", -1, (W,), "b"),
        ("t_w2", -1, (W, W), "w"), ("t_b2", -1, (W,), "b"),
    ]
    for l in range(shape.blocks):
        items += [
            ("mod_w", l, (6 * W, W), "w"), ("mod_b", l, (6 * W,), "b"),
            ("qkv_w", l, (3 * W, W), "w"), ("qkv_b", l, (3 * W,), "b"),
            ("qn_g", l, (W,), "g"), ("kn_g", l, (W,), "g"),
            ("o_w", l, (W, W), "w"), ("o_b", l, (W,), "b"),
            ("ln2_g", l, (W,), "g"), ("ln2_b", l, (W,), "b"),
            ("cq_w", l, (W, W), "w"), ("cq_b", l, (W,), "b"),
            ("ckv_w", l, (2 * W, Dc), "w"), ("ckv_b", l, (2 * W,), "b"),
            ("co_w", l, (W, W), "w"), ("co_b", l, (W,), "b"),
            ("fc1_w", l, (Wm, W), "w"), ("fc1_b", l, (Wm,), "b"),
            ("fc2_w", l, (W, Wm), "w"), ("fc2_b", l, (W,), "b"),
        ]
    items += [
        ("fmod_w", -1, (2 * W, W), "w"), ("fmod_b", -1, (2 * W,), "b"),
        ("out_w", -1, (C, W), "w"), ("out_b", -1, (C,), "b"),
        ("dec_w", -1, (C, G), "dec"),
        # the convolutional stand-in decoder: 3x3x3 convolutions C -> 16 at
        # D^3, 16 -> 8 at (2D)^3, 8 -> 1 at (4D)^3, [out, in * 27]
        ("dc1_w", -1, (16, C * 27), "w"), ("dc1_b", -1, (16,), "b"),
        ("dc2_w", -1, (8, 16 * 27), "w"), ("dc2_b", -1, (8,), "b"),
        ("dc3_w", -1, (1, 8 * 27), "w"), ("dc3_b", -1, (1,), "b"),
    ]
    return items


def weight_offsets(shape: ModelShape):
    """{(name, block): (offset_elems, dims)} and the total blob size."""
    offs = {}
    pos = 0
    for name, blk, dims, _ in weight_layout(shape):
        offs[(name, blk)] = (pos, dims)
        n = int(np.prod(dims))
        pos += (n + ALIGN_ELEMS - 1) // ALIGN_ELEMS * ALIGN_ELEMS
    return offs, pos


def weights_blob(shape: ModelShape, seed: int) -> np.ndarray:
    """Random-init bf16 weight blob (uint16 bits), layout version 2."""
    offs, total = weight_offsets(shape)
    blob = np.zeros(total, np.uint16)
    g = _rng(seed + 3)
    for name, blk, dims, init in weight_layout(shape):
        n = int(np.prod(dims))
        z = g.standard_normal(n, dtype=np.float32)
        if init == "w":
            z = z / np.float32(math.sqrt(dims[-1]))
        elif init == "b":
            z = np.float32(0.02) * z
        elif init == "g":
            z = np.float32(1.0) + np.float32(0.1) * z
        off, _ = offs[(name, blk)]
        blob[off:off + n] = f32_to_bf16_bits(z)
    return blob


def weight_view(blob: np.ndarray, shape: ModelShape, name: str, block: int = -1) -> np.ndarray:
    """fp32 view of one tensor of the blob (for tests that perturb weights)."""
    offs, _ = weight_offsets(shape)
    off, dims = offs[(name, block)]
    n = int(np.prod(dims))
    return bf16_bits_to_f32(blob[off:off + n]).reshape(dims)


def set_weight(blob: np.ndarray, shape: ModelShape, name: str, block: int, value: np.ndarray) -> None:
    offs, _ = weight_offsets(shape)
    off, dims = offs[(name, block)]
    value = np.broadcast_to(np.asarray(value, np.float32), dims)
    blob[off:off + int(np.prod(dims))] = f32_to_bf16_bits(value.reshape(-1))


# --------------------------------------------------------------------------
# velocity histories for the selection-only workload
# --------------------------------------------------------------------------

def velocity_history(grid: int, channels: int, batch: int, seed: int,
                     kind: str = "drift") -> np.ndarray:
    """Three-slot velocity history, bf16 bits [3, B, N, C]; slot 2 is the
    newest prediction v^(k-1), slot 1 is v^(k-2), slot 0 is the oldest.

    kind='drift':    v^(s) = b + m_i * 0.5^(2-s) * u + 0.1 * n^(s) with b, u,
                     n ~ N(0,1) and m_i = 0.5 (1 + sin(2 pi x/16) cos(2 pi y/16)
                     sin(2 pi z/16)) a smooth per-token drift amplitude.
    kind='ties':     values drawn from {-1, 0, 1} (many equal scores).
    kind='constant': every token carries the same velocity (all scores tie).
    """
    N = grid ** 3
    out = np.empty((3, batch, N, channels), np.uint16)
    z, y, x = np.meshgrid(np.arange(grid), np.arange(grid), np.arange(grid), indexing="ij")
    m = 0.5 * (1.0 + np.sin(2 * np.pi * x / 16) * np.cos(2 * np.pi * y / 16) * np.sin(2 * np.pi * z / 16))
    m = m.reshape(N, 1).astype(np.float32)
    for b in range(batch):
        g = _rng(seed, b)
        if kind == "drift":
            base = g.standard_normal((N, channels), dtype=np.float32)
            u = g.standard_normal((N, channels), dtype=np.float32)
            for s in range(3):
                n = g.standard_normal((N, channels), dtype=np.float32)
                v = base + m * np.float32(0.5 ** (2 - s)) * u + np.float32(0.1) * n
                out[s, b] = f32_to_bf16_bits(v)
        elif kind == "ties":
            for s in range(3):
                out[s, b] = f32_to_bf16_bits(g.integers(-1, 2, (N, channels)).astype(np.float32))
        elif kind == "constant":
            v = g.standard_normal((1, channels), dtype=np.float32)
            for s in range(3):
                out[s, b] = f32_to_bf16_bits(np.repeat(v, N, 0))
        else:
            raise ValueError(kind)
    return out


def ragged_active_targets(batch: int, tokens: int, lo: int, hi: int, seed: int) -> np.ndarray:
    """Target active-token counts a_b ~ U[lo, hi] for the ragged batch workload."""
    return _rng(seed).integers(lo, hi + 1, batch).astype(np.int64)
