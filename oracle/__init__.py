"""ctypes wrapper of the SMAT CPU oracle.

TEST INFRASTRUCTURE ONLY: imported by tests/, by the smoke check and by the
bench's CPU-baseline / reference leg; never by the product path. The oracle
shares no code with the CUDA library (see smat_oracle.cpp for the stream
specification it implements, Eq. smat-state / smat-mask / smat-gradient).

Arrays are numpy: fp32 tensors as float32, bf16 tensors as their raw uint16
bits.
"""

import ctypes
import os

import numpy as np

from . import build as _build

F32, BF16 = 0, 1
ALPHA_GLOBAL, ALPHA_PER_TENSOR, ALPHA_PER_ELEMENT = 0, 1, 2
NOISE_UNIFORM, NOISE_GAUSSIAN, NOISE_LAPLACE = 0, 1, 2
S_MASK, S_NOISE, S_ALPHA_E, S_ALPHA_T, S_MASK_LO = 0, 1, 2, 3, 4
MERGE_WA, MERGE_TA, MERGE_DARE_TA, MERGE_TIES = 0, 1, 2, 3
GLOBAL_ALPHA_ID = 0x0FFFFFFF


class OrcConfig(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("step", ctypes.c_uint32),
                ("rounds", ctypes.c_int32), ("alpha_mode", ctypes.c_int32),
                ("noise", ctypes.c_int32), ("alpha_min", ctypes.c_float),
                ("alpha_max", ctypes.c_float), ("draw_bits", ctypes.c_int32)]


class OrcTensor(ctypes.Structure):
    _fields_ = [("tensor_id", ctypes.c_uint32), ("dtype", ctypes.c_int32),
                ("numel", ctypes.c_int64), ("elem_offset", ctypes.c_int64),
                ("keep_prob", ctypes.c_float), ("sigma", ctypes.c_float),
                ("sigma_rel", ctypes.c_float)]


class OrcAdamW(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float), ("weight_decay", ctypes.c_float), ("step", ctypes.c_int32)]


class OrcMerge(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("rounds", ctypes.c_int32), ("method", ctypes.c_int32),
                ("n_experts", ctypes.c_int32), ("gamma", ctypes.c_float), ("p_drop", ctypes.c_float),
                ("retention", ctypes.c_float)]


_lib = None


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        P = ctypes.c_void_p
        L.orc_philox.argtypes = [P, P, ctypes.c_int32, P]
        L.orc_stream_words.argtypes = [P, ctypes.c_uint32, ctypes.c_uint32, P, P, ctypes.c_int64, P]
        L.orc_f32_to_bf16.argtypes = [P, ctypes.c_int64, P]
        L.orc_erfinv.argtypes = [P, ctypes.c_int64, P]
        L.orc_scalars.argtypes = [P, P, P, P, P]
        L.orc_delta_stats.argtypes = [P, P, P, P]
        L.orc_simulate.argtypes = [P, P, P, P, P]
        L.orc_simulate_at.argtypes = [P, P, ctypes.c_float, P, ctypes.c_int64, P, P, P, P]
        L.orc_gradmap.argtypes = [P, P, ctypes.c_int32, ctypes.c_int32, P, P]
        L.orc_gradmap_at.argtypes = [P, P, ctypes.c_int32, ctypes.c_int32, P, ctypes.c_int64, P, P, P]
        L.orc_mask_bits.argtypes = [P, P, P]
        L.orc_gradmap_adamw.argtypes = [P, P, ctypes.c_int32, P, P, P, P, P]
        L.orc_gradmap_adamw_at.argtypes = [P, P, ctypes.c_int32, P, ctypes.c_int64, P, P, P, P, P, P]
        L.orc_gauss_z.argtypes = [P, P, P, ctypes.c_int64, P]
        L.orc_noise_z.argtypes = [P, P, P, ctypes.c_int64, P]
        L.orc_laplace.argtypes = [P, ctypes.c_int64, P]
        L.orc_merge.argtypes = [P, ctypes.c_uint32, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64, P, P, P, P]
        L.orc_simulate_f64.argtypes = [P, P, ctypes.c_float, P, P, P]
        L.orc_gradmap_f64.argtypes = [P, P, P, P]
        for name in ("orc_philox", "orc_stream_words", "orc_f32_to_bf16", "orc_erfinv", "orc_scalars",
                     "orc_delta_stats", "orc_simulate", "orc_simulate_at", "orc_gradmap",
                     "orc_gradmap_at", "orc_mask_bits", "orc_gauss_z", "orc_simulate_f64",
                     "orc_gradmap_f64", "orc_noise_z", "orc_laplace", "orc_merge", "orc_gradmap_adamw",
                     "orc_gradmap_adamw_at"):
            getattr(L, name).restype = None
        _lib = L
    return _lib


def _p(a):
    return ctypes.c_void_p(a.ctypes.data) if a is not None else ctypes.c_void_p(0)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def config(seed=0, step=0, rounds=10, alpha_mode=ALPHA_PER_TENSOR, noise=NOISE_UNIFORM,
           alpha_min=0.3, alpha_max=1.0, draw_bits=32):
    return OrcConfig(seed, step, rounds, alpha_mode, noise, alpha_min, alpha_max, draw_bits)


def tensor(tensor_id, numel, dtype=F32, keep_prob=0.9, sigma=0.0, sigma_rel=0.0, elem_offset=0):
    return OrcTensor(tensor_id, dtype, numel, elem_offset, keep_prob, sigma, sigma_rel)


def _store_dtype(dtype):
    return np.uint16 if dtype == BF16 else np.float32


def philox(ctr4, key2, rounds=10):
    c = _c(ctr4, np.uint32)
    k = _c(key2, np.uint32)
    out = np.zeros(4, np.uint32)
    lib().orc_philox(_p(c), _p(k), rounds, _p(out))
    return out


def stream_words(cfg, stream, tid, j, w):
    j = _c(j, np.uint64)
    w = _c(w, np.uint32)
    out = np.zeros(j.shape[0], np.uint32)
    lib().orc_stream_words(ctypes.byref(cfg), stream, tid, _p(j), _p(w), j.shape[0], _p(out))
    return out


def f32_to_bf16(x):
    x = _c(x, np.float32).ravel()
    out = np.zeros(x.shape[0], np.uint16)
    lib().orc_f32_to_bf16(_p(x), x.shape[0], _p(out))
    return out


def erfinv(v):
    v = _c(v, np.float64).ravel()
    out = np.zeros(v.shape[0], np.float64)
    lib().orc_erfinv(_p(v), v.shape[0], _p(out))
    return out


def laplace(v):
    """-sign(v) ln(1 - |v|) in double (the Laplace inverse-CDF transform)."""
    v = _c(v, np.float64).ravel()
    out = np.zeros(v.shape[0], np.float64)
    lib().orc_laplace(_p(v), v.shape[0], _p(out))
    return out


def bf16_to_f32(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def scalars(cfg, t, theta=None, theta0=None):
    """{alpha, inv_keep, c, T, sigma, noise_scale} of tensor t for this call."""
    out = np.zeros(6, np.float64)
    th = _c(theta, _store_dtype(t.dtype)) if theta is not None else None
    t0 = _c(theta0, _store_dtype(t.dtype)) if theta0 is not None else None
    lib().orc_scalars(ctypes.byref(cfg), ctypes.byref(t), _p(th), _p(t0), _p(out))
    return dict(alpha=out[0], inv_keep=out[1], c=out[2], T=int(out[3]), sigma=out[4],
                noise_scale=out[5])


def delta_stats(t, theta, theta0):
    out = np.zeros(3, np.float64)
    th = _c(theta, _store_dtype(t.dtype))
    t0 = _c(theta0, _store_dtype(t.dtype))
    lib().orc_delta_stats(ctypes.byref(t), _p(th), _p(t0), _p(out))
    return dict(mean=out[0], m2=out[1], sigma=out[2])


def simulate(cfg, t, theta, theta0):
    dt = _store_dtype(t.dtype)
    th = _c(theta, dt)
    t0 = _c(theta0, dt)
    assert th.size == t.numel and t0.size == t.numel
    out = np.zeros(t.numel, dt)
    lib().orc_simulate(ctypes.byref(cfg), ctypes.byref(t), _p(th), _p(t0), _p(out))
    return out


def simulate_at(cfg, t, sigma_t, idx, theta_vals, theta0_vals):
    """Stored bits (uint32; bf16 in the low half) and kept flags at local indices idx."""
    idx = _c(idx, np.int64)
    thv = _c(theta_vals, np.float32)
    t0v = _c(theta0_vals, np.float32)
    out = np.zeros(idx.shape[0], np.uint32)
    kept = np.zeros(idx.shape[0], np.uint8)
    lib().orc_simulate_at(ctypes.byref(cfg), ctypes.byref(t), float(sigma_t), _p(idx), idx.shape[0],
                          _p(thv), _p(t0v), _p(out), _p(kept))
    return out, kept


def gradmap(cfg, t, g_sim, gdtype=F32, accumulate=False, g_old=None):
    dt = _store_dtype(gdtype)
    gs = _c(g_sim, dt)
    if accumulate:
        out = np.array(g_old, dtype=dt, copy=True)
    else:
        out = np.zeros(t.numel, dt)
    lib().orc_gradmap(ctypes.byref(cfg), ctypes.byref(t), gdtype, int(bool(accumulate)), _p(gs),
                      _p(out))
    return out


def gradmap_at(cfg, t, idx, gsim_vals, gdtype=F32, accumulate=False, gold_vals=None):
    idx = _c(idx, np.int64)
    gs = _c(gsim_vals, np.float32)
    go = _c(gold_vals, np.float32) if gold_vals is not None else np.zeros_like(gs)
    out = np.zeros(idx.shape[0], np.uint32)
    lib().orc_gradmap_at(ctypes.byref(cfg), ctypes.byref(t), gdtype, int(bool(accumulate)), _p(idx),
                         idx.shape[0], _p(gs), _p(go), _p(out))
    return out


def gradmap_adamw(cfg, t, g_sim, theta, m1, m2, lr, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0,
                  adam_step=1, gdtype=F32):
    """The gradient map fused with an AdamW step (see orc_gradmap_adamw):
    returns new (theta, m1, m2); the inputs are not modified."""
    gs = _c(g_sim, _store_dtype(gdtype))
    th = np.array(theta, dtype=_store_dtype(t.dtype), copy=True)
    a = np.array(m1, dtype=np.float32, copy=True)
    b = np.array(m2, dtype=np.float32, copy=True)
    o = OrcAdamW(lr, beta1, beta2, eps, weight_decay, adam_step)
    lib().orc_gradmap_adamw(ctypes.byref(cfg), ctypes.byref(t), gdtype, _p(gs), _p(th), _p(a), _p(b),
                            ctypes.byref(o))
    return th, a, b


def gradmap_adamw_at(cfg, t, idx, gsim_vals, theta_vals, m1_vals, m2_vals, lr, beta1=0.9, beta2=0.999, eps=1e-8,
                     weight_decay=0.0, adam_step=1, gdtype=F32):
    """gradmap_adamw at sampled local indices (g~ and theta as fp32 values):
    returns (theta stored bits as uint32, m1, m2)."""
    idx = _c(idx, np.int64)
    gs = _c(gsim_vals, np.float32)
    th = _c(theta_vals, np.float32)
    a = np.array(m1_vals, dtype=np.float32, copy=True)
    b = np.array(m2_vals, dtype=np.float32, copy=True)
    out = np.zeros(idx.shape[0], np.uint32)
    o = OrcAdamW(lr, beta1, beta2, eps, weight_decay, adam_step)
    lib().orc_gradmap_adamw_at(ctypes.byref(cfg), ctypes.byref(t), gdtype, _p(idx), idx.shape[0], _p(gs), _p(th),
                               _p(a), _p(b), ctypes.byref(o), _p(out))
    return out, a, b


def mask_bits(cfg, t):
    out = np.zeros((t.numel + 31) // 32, np.uint32)
    lib().orc_mask_bits(ctypes.byref(cfg), ctypes.byref(t), _p(out))
    return out


def unpack_bits(words, n):
    w = np.asarray(words, np.uint32)
    bits = (w[:, None] >> np.arange(32, dtype=np.uint32)[None, :]) & 1
    return bits.ravel()[:n].astype(np.uint8)


def gauss_z(cfg, t, gidx):
    g = _c(gidx, np.uint64)
    out = np.zeros(g.shape[0], np.float64)
    lib().orc_gauss_z(ctypes.byref(cfg), ctypes.byref(t), _p(g), g.shape[0], _p(out))
    return out


def noise_z(cfg, t, gidx):
    """Unit-variance variates of the elements' noise under the config's law."""
    g = _c(gidx, np.uint64)
    out = np.zeros(g.shape[0], np.float64)
    lib().orc_noise_z(ctypes.byref(cfg), ctypes.byref(t), _p(g), g.shape[0], _p(out))
    return out


def simulate_f64(cfg, t, sigma_t, theta, theta0):
    th = _c(theta, np.float64)
    t0 = _c(theta0, np.float64)
    out = np.zeros(t.numel, np.float64)
    lib().orc_simulate_f64(ctypes.byref(cfg), ctypes.byref(t), float(sigma_t), _p(th), _p(t0), _p(out))
    return out


def gradmap_f64(cfg, t, g_sim):
    gs = _c(g_sim, np.float64)
    out = np.zeros(t.numel, np.float64)
    lib().orc_gradmap_f64(ctypes.byref(cfg), ctypes.byref(t), _p(gs), _p(out))
    return out


def stored_to_f32(bits, dtype):
    """Stored bits (uint32 as returned by *_at) to fp32 values."""
    b = np.asarray(bits, np.uint32)
    if dtype == BF16:
        return (b << 16).view(np.float32)
    return b.view(np.float32)


def library_path():
    return os.path.abspath(_build.LIB)


def merge(method, theta0, experts, dtype=F32, gamma=1.0, p_drop=0.0, retention=1.0, seed=0, tensor_id=0,
          elem_offset=0, rounds=10):
    """Eq. merged-state over the K experts (WA, TA, DARE + TA or TIES); returns
    (theta_merge in storage form, the K TIES threshold keys)."""
    dt = _store_dtype(dtype)
    t0 = _c(theta0, dt).ravel()
    ex = [_c(x, dt).ravel() for x in experts]
    n = t0.size
    assert all(x.size == n for x in ex)
    K = len(ex)
    m = OrcMerge(seed, rounds, method, K, gamma, p_drop, retention)
    ptrs = (ctypes.c_void_p * K)(*[x.ctypes.data for x in ex])
    out = np.zeros(n, dt)
    thr = np.zeros(K, np.uint32)
    lib().orc_merge(ctypes.byref(m), tensor_id, dtype, n, elem_offset, _p(t0), ctypes.cast(ptrs, ctypes.c_void_p),
                    _p(out), _p(thr))
    return out, thr
