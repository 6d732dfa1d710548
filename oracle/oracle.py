"""ctypes wrapper of the C oracle (test infrastructure only; see package doc)."""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "f3dc_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liborc.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP over independent rows,
    -ffp-contract=off so every fp32 + and * rounds on its own)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
           "-fno-fast-math", _SRC, "-o", tmp, "-lm"]
    subprocess.check_call(cmd)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_f32p = C.POINTER(C.c_float)
_u16p = C.POINTER(C.c_uint16)
_i32p = C.POINTER(C.c_int32)
_u8p = C.POINTER(C.c_uint8)
_f64p = C.POINTER(C.c_double)


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            L.orc_time_schedule.argtypes = [C.c_int, C.c_double, _f32p]
            L.orc_ceil_steps.argtypes = [C.c_int, C.c_double]
            L.orc_ceil_steps.restype = C.c_int
            L.orc_phase_quota.argtypes = [C.c_int, C.c_int, C.c_double, C.c_double, C.c_double,
                                          C.c_double, C.c_int, C.c_int, C.c_double, C.c_int,
                                          C.POINTER(C.c_int)]
            L.orc_phase_quota.restype = C.c_int
            L.orc_tau_gate.argtypes = [C.c_int, C.c_int, C.c_int, C.POINTER(C.c_int)]
            L.orc_tau_gate.restype = C.c_int
            L.orc_ssc_score.argtypes = [_u16p, _u16p, C.c_int, C.c_int, C.c_double, _f32p]
            L.orc_select.argtypes = [_f32p, C.c_int, C.c_int, _u8p, _i32p]
            L.orc_select.restype = C.c_int
            L.orc_occupancy.argtypes = [_f32p, C.c_int, C.c_int, _u16p, C.c_int, _u8p]
            L.orc_dynamic_voxels.argtypes = [_u8p, _u8p, C.c_longlong]
            L.orc_dynamic_voxels.restype = C.c_longlong
            L.orc_merge_euler.argtypes = [C.c_int, C.c_int, _i32p, C.c_int, _f32p, _u16p,
                                          C.c_float, _f32p, _u16p]
            L.orc_model_create.argtypes = [C.c_int] * 9 + [_u16p]
            L.orc_model_create.restype = C.c_void_p
            L.orc_model_free.argtypes = [C.c_void_p]
            L.orc_linear.argtypes = [_f32p, C.c_int, C.c_int, _f32p, _f32p, C.c_int, _f32p]
            L.orc_layernorm.argtypes = [_f32p, C.c_int, C.c_int, _f32p]
            L.orc_gelu.argtypes = [C.c_float]
            L.orc_gelu.restype = C.c_float
            L.orc_attention.argtypes = [_f32p, C.c_int, _f32p, C.c_int, _f32p, C.c_int,
                                        C.c_int, C.c_int, C.c_int, C.c_int, _f32p]
            L.orc_pos_embed.argtypes = [C.c_int, C.c_int, C.c_int, _f32p]
            L.orc_time_embed.argtypes = [C.c_void_p, C.c_float, _f32p]
            L.orc_modulation.argtypes = [C.c_void_p, _f32p, C.c_int, _f32p]
            L.orc_cond_kv.argtypes = [C.c_void_p, _u16p, _f32p]
            L.orc_dit_forward.argtypes = [C.c_void_p, _f32p, _i32p, C.c_int, C.c_float, _f32p, _f32p]
            L.orc_sample.argtypes = [C.c_void_p, C.c_int, C.c_double, C.c_double, C.c_double,
                                     C.c_double, C.c_double, C.c_double, C.c_int, C.c_int, C.c_int,
                                     _f32p, _u16p, C.c_int, _f64p, _i32p, _i32p, _i32p, _f64p, _u16p,
                                     C.c_int, C.c_double, C.c_double, C.c_int, C.c_int, C.POINTER(C.c_int64)]
            L.orc_decode_conv.argtypes = [C.c_void_p, _f32p, _u8p]
            L.orc_fit_mu.argtypes = [_f64p, C.c_int, C.c_int, C.c_int, C.c_int, C.c_double, C.c_double,
                                     _f64p, _f64p, C.POINTER(C.c_int)]
            L.orc_ssc_score3.argtypes = [_u16p, _u16p, _u16p, C.c_int, C.c_int, C.c_double, _f32p]
            L.orc_cfg_on.argtypes = [C.c_int, C.c_double, C.c_double, C.c_int]
            L.orc_cfg_combine.argtypes = [C.c_longlong, _f32p, _f32p, C.c_double, _f32p]
            L.orc_f32_to_bf16.argtypes = [C.c_float]
            L.orc_f32_to_bf16.restype = C.c_uint16
            _lib = L
    return _lib


def _p(a: np.ndarray, typ):
    return a.ctypes.data_as(typ)


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def _u16(a):
    return np.ascontiguousarray(a, dtype=np.uint16)


# ------------------------------------------------------------------ schedule

def time_schedule(T: int, eta: float) -> np.ndarray:
    out = np.empty(T + 1, np.float32)
    lib().orc_time_schedule(T, eta, _p(out, _f32p))
    return out


def ceil_steps(T: int, rho: float) -> int:
    return lib().orc_ceil_steps(T, rho)


def phase_quota(N, T, rho_a, rho_off, mu, xi, f_corr, gamma_up, sigma, k):
    ph = C.c_int(0)
    c = lib().orc_phase_quota(N, T, rho_a, rho_off, mu, xi, f_corr, gamma_up, sigma, k, C.byref(ph))
    return c, ph.value


class TauGate:
    def __init__(self, tau: int, mode: int = 0):
        self.tau, self.mode, self.consec = tau, mode, C.c_int(0)

    def __call__(self, quota: int) -> int:
        return lib().orc_tau_gate(quota, self.tau, self.mode, C.byref(self.consec))


# ------------------------------------------------------------------ SSC

def ssc_score(v1_bits: np.ndarray, v2_bits: np.ndarray, omega: float) -> np.ndarray:
    v1, v2 = _u16(v1_bits), _u16(v2_bits)
    N, Cc = v1.shape
    out = np.empty(N, np.float32)
    lib().orc_ssc_score(_p(v1, _u16p), _p(v2, _u16p), N, Cc, omega, _p(out, _f32p))
    return out


def ssc_score3(v1_bits: np.ndarray, v2_bits: np.ndarray, v3_bits: np.ndarray, omega: float) -> np.ndarray:
    """SSC score with the second-difference acceleration over v(t-1), v(t-2), v(t-3)."""
    v1, v2, v3 = _u16(v1_bits), _u16(v2_bits), _u16(v3_bits)
    N, Cc = v1.shape
    out = np.empty(N, np.float32)
    lib().orc_ssc_score3(_p(v1, _u16p), _p(v2, _u16p), _p(v3, _u16p), N, Cc, omega, _p(out, _f32p))
    return out


def select(score: np.ndarray, c: int):
    s = _f32(score)
    N = s.shape[0]
    cached = np.zeros(N, np.uint8)
    idx = np.zeros(max(N, 1), np.int32)
    na = lib().orc_select(_p(s, _f32p), N, c, _p(cached, _u8p), _p(idx, _i32p))
    return cached, idx[:na].copy()


# ------------------------------------------------------------------ ops

def linear(x, w, b=None):
    x, w = _f32(x), _f32(w)
    rows, n_in = x.shape
    n_out = w.shape[0]
    y = np.empty((rows, n_out), np.float32)
    bp = _p(_f32(b), _f32p) if b is not None else None
    bb = _f32(b) if b is not None else None
    lib().orc_linear(_p(x, _f32p), rows, n_in, _p(w, _f32p),
                     _p(bb, _f32p) if bb is not None else bp, n_out, _p(y, _f32p))
    return y


def layernorm(x):
    x = _f32(x)
    y = np.empty_like(x)
    lib().orc_layernorm(_p(x, _f32p), x.shape[0], x.shape[1], _p(y, _f32p))
    return y


def gelu(x: float) -> float:
    return lib().orc_gelu(x)


def attention(q, k, v, heads: int):
    """q [nq, H*dh], k/v [nk, H*dh] -> [nq, H*dh]."""
    q, k, v = _f32(q), _f32(k), _f32(v)
    nq, Wd = q.shape
    nk = k.shape[0]
    dh = Wd // heads
    out = np.empty((nq, Wd), np.float32)
    lib().orc_attention(_p(q, _f32p), Wd, _p(k, _f32p), Wd, _p(v, _f32p), Wd, nq, nk, heads, dh,
                        _p(out, _f32p))
    return out


def pos_embed(grid: int, W: int, i: int) -> np.ndarray:
    out = np.empty(W, np.float32)
    lib().orc_pos_embed(grid, W, i, _p(out, _f32p))
    return out


def occupancy(S: np.ndarray, dec_w_bits: np.ndarray) -> np.ndarray:
    S = _f32(S)
    dw = _u16(dec_w_bits)
    N, Cc = S.shape
    G = dw.size // Cc
    occ = np.empty((N, G), np.uint8)
    lib().orc_occupancy(_p(S, _f32p), N, Cc, _p(dw, _u16p), G, _p(occ, _u8p))
    return occ


def dynamic_voxels(occ_a: np.ndarray, occ_b: np.ndarray) -> int:
    a = np.ascontiguousarray(occ_a, np.uint8)
    b = np.ascontiguousarray(occ_b, np.uint8)
    return int(lib().orc_dynamic_voxels(_p(a, _u8p), _p(b, _u8p), a.size))


def fit_mu(curves, k_lo=8, k_hi=18, tol=0.1, min_frac=0.6):
    """Data-driven PCSC slope from dynamic-voxel curves [n, T]: returns
    (mu, slopes [n], kept [n] bool)."""
    c = np.ascontiguousarray(curves, np.float64)
    n, T = c.shape
    mu = C.c_double(0.0)
    slopes = np.empty(n, np.float64)
    kept = (C.c_int * max(n, 1))()
    lib().orc_fit_mu(_p(c, _f64p), n, T, k_lo, k_hi, tol, min_frac, C.byref(mu), _p(slopes, _f64p), kept)
    return mu.value, slopes, np.array([bool(kept[i]) for i in range(n)])


def cfg_on(T: int, eta: float, t_lo: float, k: int) -> bool:
    """Whether step k (1-based) is guided: t_k in the CFG interval [t_lo, 1]."""
    return bool(lib().orc_cfg_on(T, eta, t_lo, k))


def cfg_combine(v_c, v_u, s: float) -> np.ndarray:
    """Guided velocity v_u + s (v_c - v_u) in fp32 (subtract, multiply, add)."""
    vc, vu = _f32(v_c), _f32(v_u)
    out = np.empty_like(vc)
    lib().orc_cfg_combine(vc.size, _p(vc, _f32p), _p(vu, _f32p), s, _p(out, _f32p))
    return out


def merge_euler(S, active_idx, v_active, v_cache_bits, dt: float):
    """Returns (S_new, v_t_bits); inputs are not modified."""
    S = _f32(S).copy()
    N, Cc = S.shape
    idx = np.ascontiguousarray(active_idx, np.int32)
    va = _f32(v_active).reshape(-1, Cc) if len(idx) else np.zeros((1, Cc), np.float32)
    vc = _u16(v_cache_bits)
    vt = np.empty((N, Cc), np.uint16)
    lib().orc_merge_euler(N, Cc, _p(idx, _i32p) if len(idx) else None, len(idx), _p(va, _f32p),
                          _p(vc, _u16p), C.c_float(dt), _p(S, _f32p), _p(vt, _u16p))
    return S, vt


def f32_to_bf16(x: float) -> int:
    return lib().orc_f32_to_bf16(x)


# ------------------------------------------------------------------ model

class Model:
    """Oracle flow transformer built from a layout-v2 weight blob."""

    def __init__(self, shape, blob_bits: np.ndarray):
        self.shape = shape
        self._blob = _u16(blob_bits)
        s = shape
        self.h = lib().orc_model_create(s.grid, s.channels, s.width, s.blocks, s.heads,
                                        s.mlp_ratio, s.cond_tokens, s.cond_dim, s.gamma_up,
                                        _p(self._blob, _u16p))

    def __del__(self):
        try:
            if self.h:
                lib().orc_model_free(self.h)
                self.h = None
        except Exception:
            pass

    def time_embed(self, t: float) -> np.ndarray:
        out = np.empty(self.shape.width, np.float32)
        lib().orc_time_embed(self.h, C.c_float(t), _p(out, _f32p))
        return out

    def modulation(self, temb: np.ndarray, block: int) -> np.ndarray:
        n = 6 * self.shape.width if block >= 0 else 2 * self.shape.width
        out = np.empty(n, np.float32)
        te = _f32(temb)
        lib().orc_modulation(self.h, _p(te, _f32p), block, _p(out, _f32p))
        return out

    def decode_conv(self, S: np.ndarray) -> np.ndarray:
        """Occupancy of the convolutional stand-in decoder: uint8 [(4D)^3], index (z 4D + y) 4D + x."""
        S = _f32(S)
        out = np.empty(self.shape.tokens * 64, np.uint8)
        lib().orc_decode_conv(self.h, _p(S, _f32p), _p(out, _u8p))
        return out

    def cond_kv(self, cond_bits: np.ndarray) -> np.ndarray:
        s = self.shape
        cb = _u16(cond_bits)
        out = np.empty((s.blocks, 2, s.cond_tokens, s.width), np.float32)
        lib().orc_cond_kv(self.h, _p(cb, _u16p), _p(out, _f32p))
        return out

    def forward(self, S: np.ndarray, active_idx: np.ndarray, t: float, cond_kv: np.ndarray) -> np.ndarray:
        S = _f32(S)
        idx = np.ascontiguousarray(active_idx, np.int32)
        a = len(idx)
        out = np.empty((max(a, 1), self.shape.channels), np.float32)
        kv = _f32(cond_kv)
        lib().orc_dit_forward(self.h, _p(S, _f32p), _p(idx, _i32p), a, C.c_float(t),
                              _p(kv, _f32p), _p(out, _f32p))
        return out[:a]

    def sample(self, S: np.ndarray, cond_bits: np.ndarray, *, T, eta=3.0, rho_a=0.2, rho_off=0.75,
               mu=-0.07, omega=0.7, xi=0.7, f_corr=3, tau=3, refresh_mode=0,
               sigma_override=None, quota_schedule=None, cfg=None, cfg_t_lo=0.5, ssc_accel=0, decoder=0,
               want_curve=False):
        """Algorithm 1 for B samples.  Returns dict(S, quota, n_active, sigma, v_hist).
        cfg: guidance strength s (None: unguided) for the steps with t_k >= cfg_t_lo."""
        S = _f32(S).copy()
        B = S.shape[0]
        N = self.shape.tokens
        cb = _u16(cond_bits)
        ql = np.zeros((T, B), np.int32)
        nl = np.zeros((T, B), np.int32)
        so = np.zeros(B, np.float64)
        vh = np.zeros((2, B, N, self.shape.channels), np.uint16)
        sov = np.ascontiguousarray(sigma_override, np.float64) if sigma_override is not None else None
        qs = np.ascontiguousarray(quota_schedule, np.int32) if quota_schedule is not None else None
        dl = np.zeros((T, B), np.int64) if want_curve else None
        lib().orc_sample(self.h, T, eta, rho_a, rho_off, mu, omega, xi, f_corr, tau, refresh_mode,
                         _p(S, _f32p), _p(cb, _u16p), B,
                         _p(sov, _f64p) if sov is not None else None,
                         _p(qs, _i32p) if qs is not None else None,
                         _p(ql, _i32p), _p(nl, _i32p), _p(so, _f64p), _p(vh, _u16p),
                         0 if cfg is None else 1, 0.0 if cfg is None else float(cfg), float(cfg_t_lo),
                         int(ssc_accel), int(decoder),
                         dl.ctypes.data_as(C.POINTER(C.c_int64)) if dl is not None else None)
        return dict(S=S, quota=ql, n_active=nl, sigma=so, v_hist=vh, dyn=dl)
