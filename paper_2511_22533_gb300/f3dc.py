"""Thin ctypes binding of libf3dc.so (declared in include/f3dc.h).

Argument marshalling only: every step of the cached denoising step runs in
the library's CUDA kernels.  Device buffers are torch CUDA tensors (passed by
data pointer); host buffers are NumPy arrays.  If the library has not been
built, loading raises -- there is no CPU fallback.
"""
from __future__ import annotations

import ctypes as C
import os
import re
import threading

import numpy as np

from . import build as _build

F3DC_OK = 0
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "CUDA", 3: "OOM", 4: "UNSUPPORTED", 5: "TIMEOUT",
                6: "NONFINITE", 7: "DEVICE"}
REFRESH_PERIOD, REFRESH_LITERAL = 0, 1
EPI_BIAS, EPI_GELU, EPI_RESID = 0, 1, 2
HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "f3dc.h")


class F3dcError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"f3dc status {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class Config(C.Structure):
    _fields_ = [("grid", C.c_int32), ("channels", C.c_int32), ("width", C.c_int32), ("blocks", C.c_int32),
                ("heads", C.c_int32), ("mlp_ratio", C.c_int32), ("cond_tokens", C.c_int32),
                ("cond_dim", C.c_int32), ("steps", C.c_int32), ("max_batch", C.c_int32),
                ("gamma_up", C.c_int32), ("tau", C.c_int32), ("f_corr", C.c_int32),
                ("refresh_mode", C.c_int32), ("eta", C.c_double), ("rho_a", C.c_double), ("mu", C.c_double),
                ("omega", C.c_double), ("xi", C.c_double), ("rho_cfg_off", C.c_double),
                ("cfg_strength", C.c_double), ("cfg_t_lo", C.c_double), ("ssc_accel", C.c_int32),
                ("decoder", C.c_int32)]


class KernelStats(C.Structure):
    _fields_ = [("name", C.c_char * 24), ("launches", C.c_int64), ("total_ms", C.c_double),
                ("flops", C.c_double), ("bytes", C.c_double)]


class Weights(C.Structure):
    _fields_ = [("layout_version", C.c_int32), ("blob", C.c_void_p), ("blob_elems", C.c_size_t)]


class FaultInjection(C.Structure):
    _fields_ = [("fail_alloc_at", C.c_int32), ("gemm_missing_arrivals", C.c_int32), ("gemm_wait_ns", C.c_int64),
                ("attn_missing_kv", C.c_int32)]


_lock = threading.Lock()
_lib = None
_vp, _i32p, _f32p, _f64p, _u32p = C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_float), C.POINTER(
    C.c_double), C.POINTER(C.c_uint32)


def library_path() -> str:
    return _build.LIB


def lib():
    """Loads libf3dc.so (building it first if the sources are newer)."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build()
            if not os.path.exists(path):
                raise RuntimeError(f"libf3dc.so missing at {path}")
            L = C.CDLL(path)
            cfgp, wp = C.POINTER(Config), C.POINTER(Weights)
            sig = {
                "f3dc_config_default": ([cfgp], C.c_int),
                "f3dc_weights_elems": ([cfgp], C.c_size_t),
                "f3dc_time_schedule": ([cfgp, _f32p], C.c_int),
                "f3dc_pcsc_quota": ([cfgp, C.c_double, C.c_int32, _i32p, _i32p, _i32p], C.c_int),
                "f3dc_create": ([cfgp, wp, _vp, C.POINTER(_vp)], C.c_int),
                "f3dc_destroy": ([_vp], C.c_int),
                "f3dc_last_error": ([_vp], C.c_char_p),
                "f3dc_device_status": ([_vp, _u32p], C.c_int),
                "f3dc_ssc_select": ([_vp, _vp, _vp, C.c_int32, _vp, _vp, _vp, _vp, _vp], C.c_int),
                "f3dc_set_cond": ([_vp, _vp, C.c_int32, _vp], C.c_int),
                "f3dc_step": ([_vp, C.c_int32, C.c_int32, _vp, _vp, _vp, _vp, _vp], C.c_int),
                "f3dc_sample": ([_vp, _vp, _vp, C.c_int32, _f64p, _i32p, _i32p, _f64p, _vp], C.c_int),
                "f3dc_dynamic_voxel_curve": ([_vp, _vp, _vp, C.c_int32, C.POINTER(C.c_int64), _vp], C.c_int),
                "f3dc_fit_mu": ([_f64p, C.c_int32, C.c_int32, C.c_int32, C.c_int32, C.c_double, C.c_double,
                                 _f64p, _f64p, _i32p], C.c_int),
                "f3dc_forward": ([_vp, C.c_float, C.c_int32, _vp, _vp, _vp, _vp, _vp], C.c_int),
                "f3dc_profile": ([_vp, C.c_int32], C.c_int),
                "f3dc_profile_read": ([_vp, C.POINTER(KernelStats), C.c_int32, _i32p], C.c_int),
                "f3dc_launch_count": ([_vp, C.POINTER(C.c_int64)], C.c_int),
                "f3dc_set_graphs": ([_vp, C.c_int32], C.c_int),
                "f3dc_gemm": ([_vp, _vp, _vp, _vp, _vp, C.c_int32, C.c_int32, C.c_int32, C.c_int32, _vp], C.c_int),
                "f3dc_gemm_noalloc": ([_vp, _vp, _vp, _vp, _vp, C.c_int32, C.c_int32, C.c_int32, C.c_int32, _vp],
                                      C.c_int),
                "f3dc_gemm_status": ([_u32p], C.c_int),
                "f3dc_set_fault_injection": ([C.POINTER(FaultInjection)], C.c_int),
                "f3dc_attention": ([_vp, C.c_int32, _vp, _vp, C.c_int32, _vp, C.c_int32, C.c_int32, C.c_int32,
                                    C.c_int32, _vp], C.c_int),
            }
            for name, (args, res) in sig.items():
                fn = getattr(L, name)
                fn.argtypes = args
                fn.restype = res
            _lib = L
    return _lib


def declared_symbols():
    """Names of the functions include/f3dc.h declares."""
    with open(HEADER) as f:
        text = f.read()
    return sorted(set(re.findall(r"\b(f3dc_\w+)\s*\(", text)))


def _check(status, handle=None):
    if status != F3DC_OK:
        msg = lib().f3dc_last_error(handle)
        raise F3dcError(status, msg.decode() if msg else "")


def _ptr(t):
    if t is None:
        return None
    return C.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is not None:
        return C.c_void_p(stream)
    import torch
    return C.c_void_p(torch.cuda.current_stream().cuda_stream)


def _np_ptr(a, typ):
    return None if a is None else a.ctypes.data_as(typ)


# ---------------------------------------------------------------- host calls

def default_config() -> Config:
    c = Config()
    _check(lib().f3dc_config_default(C.byref(c)))
    return c


def config_for(shape, max_batch: int = 1, **hyper) -> Config:
    """Config for a synth.ModelShape; keyword arguments override fields."""
    c = default_config()
    c.grid, c.channels, c.width, c.blocks = shape.grid, shape.channels, shape.width, shape.blocks
    c.heads, c.mlp_ratio, c.cond_tokens, c.cond_dim = shape.heads, shape.mlp_ratio, shape.cond_tokens, shape.cond_dim
    c.steps, c.gamma_up, c.max_batch = shape.steps, shape.gamma_up, max_batch
    for k, v in hyper.items():
        setattr(c, k, v)
    return c


def weights_elems(cfg: Config) -> int:
    return int(lib().f3dc_weights_elems(C.byref(cfg)))


def time_schedule(cfg: Config) -> np.ndarray:
    out = np.empty(cfg.steps + 1, np.float32)
    _check(lib().f3dc_time_schedule(C.byref(cfg), out.ctypes.data_as(_f32p)))
    return out


def pcsc_quota(cfg: Config, sigma: float, k: int, consec=None):
    """Returns (quota, phase); consec is a one-element int32 array updated in
    place when the tau rule should apply."""
    q, ph = C.c_int32(0), C.c_int32(0)
    cp = consec.ctypes.data_as(_i32p) if consec is not None else None
    _check(lib().f3dc_pcsc_quota(C.byref(cfg), float(sigma), int(k), cp, C.byref(q), C.byref(ph)))
    return q.value, ph.value


# ---------------------------------------------------------------- handle

class Handle:
    """Owns an f3dc_handle.  `blob` is a CUDA tensor of the layout-v2 bf16
    weights (any 16-bit dtype); it may be freed after construction."""

    def __init__(self, cfg: Config, blob, stream=None):
        self.cfg = cfg
        self.h = C.c_void_p()
        w = Weights(2, blob.data_ptr(), blob.numel())
        _check(lib().f3dc_create(C.byref(cfg), C.byref(w), _stream(stream), C.byref(self.h)))

    def close(self):
        if self.h:
            lib().f3dc_destroy(self.h)
            self.h = C.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _ck(self, st):
        _check(st, self.h)

    def device_status(self) -> int:
        v = C.c_uint32(0)
        self._ck(lib().f3dc_device_status(self.h, C.byref(v)))
        return v.value

    def ssc_select(self, v_prev1, v_prev2, B, quota_dev, active_idx_out, n_active_out, cached_mask_out=None,
                   stream=None):
        self._ck(lib().f3dc_ssc_select(self.h, _ptr(v_prev1), _ptr(v_prev2), B, _ptr(quota_dev),
                                       _ptr(active_idx_out), _ptr(n_active_out), _ptr(cached_mask_out),
                                       _stream(stream)))

    def set_cond(self, cond, B, stream=None):
        self._ck(lib().f3dc_set_cond(self.h, _ptr(cond), B, _stream(stream)))

    def step(self, k, B, S, ring, quota_dev, dyn_voxels=None, stream=None):
        self._ck(lib().f3dc_step(self.h, k, B, _ptr(S), _ptr(ring), _ptr(quota_dev), _ptr(dyn_voxels),
                                 _stream(stream)))

    def sample(self, S, cond, B, sigma_override=None, quota_schedule=None, want_log=True, stream=None):
        """Algorithm 1 in place on S; returns (quota_log [T, B], sigma [B]) or
        (None, None) when want_log is False (no host synchronisation)."""
        T = self.cfg.steps
        so = None if sigma_override is None else np.ascontiguousarray(sigma_override, np.float64)
        qs = None if quota_schedule is None else np.ascontiguousarray(quota_schedule, np.int32)
        ql = np.zeros((T, B), np.int32) if want_log else None
        sg = np.zeros(B, np.float64) if want_log else None
        self._ck(lib().f3dc_sample(self.h, _ptr(S), _ptr(cond), B, _np_ptr(so, _f64p), _np_ptr(qs, _i32p),
                                   _np_ptr(ql, _i32p), _np_ptr(sg, _f64p), _stream(stream)))
        return ql, sg

    def dynamic_voxel_curve(self, S, cond, B, stream=None) -> np.ndarray:
        """Eq. 1's dS at every step of an uncached sampler run: int64 [T, B]."""
        out = np.zeros((self.cfg.steps, B), np.int64)
        self._ck(lib().f3dc_dynamic_voxel_curve(self.h, _ptr(S), _ptr(cond), B,
                                                out.ctypes.data_as(C.POINTER(C.c_int64)), _stream(stream)))
        return out

    def profile(self, enable: bool):
        self._ck(lib().f3dc_profile(self.h, 1 if enable else 0))

    def profile_read(self):
        arr = (KernelStats * 32)()
        n = C.c_int32(0)
        self._ck(lib().f3dc_profile_read(self.h, arr, 32, C.byref(n)))
        return [{"name": arr[i].name.decode(), "launches": arr[i].launches, "total_ms": arr[i].total_ms,
                 "flops": arr[i].flops, "bytes": arr[i].bytes} for i in range(min(n.value, 32))]

    def set_graphs(self, enable: bool):
        self._ck(lib().f3dc_set_graphs(self.h, 1 if enable else 0))

    def launch_count(self) -> int:
        n = C.c_int64(0)
        self._ck(lib().f3dc_launch_count(self.h, C.byref(n)))
        return n.value

    def forward(self, t, B, S, active_idx, n_active, v_out, stream=None):
        self._ck(lib().f3dc_forward(self.h, float(t), B, _ptr(S), _ptr(active_idx), _ptr(n_active), _ptr(v_out),
                                    _stream(stream)))


# ---------------------------------------------------------------- kernels

def fit_mu(curves, k_lo=8, k_hi=18, tol=0.1, min_frac=0.6):
    """Data-driven PCSC slope from dS curves [n, T]: (mu, slopes [n], kept [n] bool)."""
    c = np.ascontiguousarray(curves, np.float64)
    n, T = c.shape
    mu = C.c_double(0.0)
    slopes = np.empty(n, np.float64)
    kept = np.empty(n, np.int32)
    _check(lib().f3dc_fit_mu(c.ctypes.data_as(_f64p), n, T, k_lo, k_hi, tol, min_frac, C.byref(mu),
                             slopes.ctypes.data_as(_f64p), kept.ctypes.data_as(_i32p)))
    return mu.value, slopes, kept.astype(bool)


def gemm(A, Bw, bias, gate, out, M, N, K, epilogue, stream=None):
    _check(lib().f3dc_gemm(_ptr(A), _ptr(Bw), _ptr(bias), _ptr(gate), _ptr(out), M, N, K, epilogue,
                           _stream(stream)))


def gemm_noalloc(A, Bw, bias, gate, out, M, N, K, epilogue, stream=None):
    """f3dc_gemm without any allocation (split-K scratch in a static array)."""
    _check(lib().f3dc_gemm_noalloc(_ptr(A), _ptr(Bw), _ptr(bias), _ptr(gate), _ptr(out), M, N, K, epilogue,
                                   _stream(stream)))


def set_fault_injection(fail_alloc_at=-1, gemm_missing_arrivals=0, gemm_wait_ns=0, attn_missing_kv=0):
    """Test-only, host-side fault injection (see f3dc_set_fault_injection);
    called with no arguments it turns everything off."""
    fi = FaultInjection(fail_alloc_at, gemm_missing_arrivals, gemm_wait_ns, attn_missing_kv)
    _check(lib().f3dc_set_fault_injection(C.byref(fi)))


def gemm_status() -> int:
    """Reads and clears the current device's status word of the standalone
    kernel calls: GEMMs and attention (synchronizes the device)."""
    v = C.c_uint32(0)
    _check(lib().f3dc_gemm_status(C.byref(v)))
    return v.value


def attention(q, ldq, k, v, ldkv, out, nq, nk, heads, dh, stream=None):
    _check(lib().f3dc_attention(_ptr(q), ldq, _ptr(k), _ptr(v), ldkv, _ptr(out), nq, nk, heads, dh,
                                _stream(stream)))
