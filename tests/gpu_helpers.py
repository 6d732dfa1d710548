"""Shared helpers of the GPU parity tests (no method arithmetic here)."""
import numpy as np
import torch

from paper_2511_22533_gb300 import f3dc, synth

DEV = "cuda:0"


def dev_u16(a: np.ndarray) -> torch.Tensor:
    """uint16 bit patterns (bf16 storage) -> CUDA int16 tensor."""
    return torch.from_numpy(np.ascontiguousarray(a, np.uint16).view(np.int16)).to(DEV)


def dev_bf16(a: np.ndarray) -> torch.Tensor:
    return dev_u16(a).view(torch.bfloat16)


def host_u16(t: torch.Tensor) -> np.ndarray:
    return t.detach().view(torch.int16).cpu().numpy().view(np.uint16)


def dev_f32(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(DEV)


def dev_i32(a) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(DEV)


def rel_l2(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


def max_abs(a, b) -> float:
    return float(np.max(np.abs(np.asarray(a, np.float64) - np.asarray(b, np.float64)))) if np.size(a) else 0.0


# tolerance on the velocities of one denoising step
VEL_MAX_ABS = 2e-2
VEL_REL_L2 = 1e-2


def bf16_ulp(x) -> np.ndarray:
    """Spacing of bf16 values at |x| (8 significant bits)."""
    a = np.maximum(np.abs(np.asarray(x, np.float64)), 2.0 ** -126)
    return 2.0 ** (np.floor(np.log2(a)) - 7)


def stored_vel_excess(got, ref) -> float:
    """Largest amount by which two bf16-STORED velocity arrays differ beyond
    VEL_MAX_ABS plus one bf16 unit.

    Both sides round their computed velocity to bf16 (round to nearest even)
    before storing it, each within half a unit, so computed velocities g, r
    with |g - r| <= VEL_MAX_ABS store as values within VEL_MAX_ABS + ulp.
    At |v| >= 4 one unit (2^-5) already exceeds 2e-2: two computed values a
    hair apart on either side of a rounding boundary store one unit apart."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    if got.size == 0:
        return -1.0
    bound = VEL_MAX_ABS + bf16_ulp(np.maximum(np.abs(got), np.abs(ref)))
    return float(np.max(np.abs(got - ref) - bound))


def handle_for(shape, max_batch=1, seed=0, **hyper):
    blob = synth.weights_blob(shape, seed)
    cfg = f3dc.config_for(shape, max_batch, **hyper)
    h = f3dc.Handle(cfg, dev_u16(blob))
    torch.cuda.synchronize()
    return h, blob, cfg


def assert_clean(h):
    st = h.device_status()
    assert st == 0, f"device status word {st:#x}"
