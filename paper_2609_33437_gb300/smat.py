"""Thin Python binding of libsmat (include/smat.h).

Argument marshalling only: PyTorch provides device memory and streams, every
step of the simulated-merge path runs in the library's CUDA kernels. There is
no CPU fallback: if the library cannot be loaded the calls raise.

Names follow the C ABI: smat_init -> SmatSession(...), smat_simulate_multi ->
SmatSession.simulate_multi, smat_grad_map_multi -> SmatSession.grad_map_multi,
smat_grad_map_adamw_multi -> SmatSession.grad_map_adamw_multi,
smat_swap -> SmatSession.swap, smat_mask_bits -> SmatSession.mask_bits,
smat_tensor_scalars -> SmatSession.tensor_scalars.
"""

import ctypes
import os
from typing import List, Optional, Sequence

import torch

from . import build as _build

SMAT_F32, SMAT_BF16 = 0, 1
SMAT_NOISE_UNIFORM, SMAT_NOISE_GAUSSIAN, SMAT_NOISE_LAPLACE = 0, 1, 2
SMAT_ALPHA_GLOBAL, SMAT_ALPHA_PER_TENSOR, SMAT_ALPHA_PER_ELEMENT = 0, 1, 2

EXPORTED = ("smat_workspace_bytes", "smat_init", "smat_simulate_multi", "smat_grad_map_multi",
            "smat_swap", "smat_active", "smat_mask_bits", "smat_tensor_scalars", "smat_destroy",
            "smat_debug_philox", "smat_debug_noise_unit", "smat_debug_fused", "smat_poll_errors",
            "smat_delta_sigma_noalloc", "smat_timing_enable", "smat_timing_read", "smat_status_string",
            "smat_last_error", "smat_abi_version", "smat_refill_theta0", "smat_mark_theta0_resident",
            "smat_merge_workspace_bytes", "smat_merge", "smat_merge_ties_thresholds",
            "smat_grad_map_adamw_multi")


class AdamW(ctypes.Structure):
    """smat_adamw: AdamW hyperparameters (decoupled weight decay); step is the
    optimizer's own step count t >= 1."""
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float), ("weight_decay", ctypes.c_float), ("step", ctypes.c_int32)]


class SmatError(RuntimeError):
    def __init__(self, func, status, detail):
        super().__init__(f"{func} failed: {status} ({detail})")
        self.status = status
        self.detail = detail


class TensorDesc(ctypes.Structure):
    _fields_ = [("theta", ctypes.c_void_p), ("theta0", ctypes.c_void_p), ("sim", ctypes.c_void_p),
                ("numel", ctypes.c_int64), ("elem_offset", ctypes.c_int64),
                ("tensor_id", ctypes.c_uint32), ("dtype", ctypes.c_int32),
                ("keep_prob", ctypes.c_float), ("sigma", ctypes.c_float), ("sigma_rel", ctypes.c_float)]


class Config(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("alpha_min", ctypes.c_float), ("alpha_max", ctypes.c_float),
                ("alpha_mode", ctypes.c_int32), ("noise", ctypes.c_int32), ("philox_rounds", ctypes.c_int32),
                ("flags", ctypes.c_int32), ("draw_bits", ctypes.c_int32)]


SMAT_FLAG_UNFUSED_STATS = 1


def SMAT_FLAG_CHUNK_LOG2(k: int) -> int:
    """Force the work-chunk size to 2^k elements (12 <= k <= 18)."""
    return k << 8


_lib = None


def library_path() -> str:
    return _build.LIB


def load_library(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load the in-tree libsmat.so (building it with nvcc if it is missing)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_build.LIB) or not _build.up_to_date():
        if not build_if_missing:
            raise ImportError("libsmat.so is not built; run paper_2609_33437_gb300/build.py")
        _build.build()
    L = ctypes.CDLL(_build.LIB)
    P, I32, I64, U32, U64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32, ctypes.c_uint64
    L.smat_workspace_bytes.argtypes = [P, I32, P]
    L.smat_workspace_bytes.restype = ctypes.c_size_t
    L.smat_init.argtypes = [ctypes.POINTER(P), P, I32, P, P, ctypes.c_size_t, P]
    L.smat_simulate_multi.argtypes = [P, U32, P]
    L.smat_grad_map_multi.argtypes = [P, U32, P, P, I32, I32, P]
    L.smat_grad_map_adamw_multi.argtypes = [P, U32, P, P, P, I32, ctypes.POINTER(AdamW), P]
    L.smat_swap.argtypes = [P, ctypes.POINTER(I32)]
    L.smat_active.argtypes = [P, ctypes.POINTER(I32)]
    L.smat_mask_bits.argtypes = [P, U32, I32, P, P]
    L.smat_tensor_scalars.argtypes = [P, U32, P, P]
    L.smat_destroy.argtypes = [P]
    L.smat_refill_theta0.argtypes = [P, P, P]
    L.smat_merge_workspace_bytes.argtypes = [P, I32, P]
    L.smat_merge_workspace_bytes.restype = ctypes.c_size_t
    L.smat_merge.argtypes = [P, I32, P, P, ctypes.c_size_t, P]
    L.smat_merge_ties_thresholds.argtypes = [P, I32, P, P, P, P]
    L.smat_mark_theta0_resident.argtypes = [P]
    L.smat_debug_philox.argtypes = [P, I64, U64, I32, P, P, P]
    L.smat_debug_noise_unit.argtypes = [P, I64, I32, P, P]
    L.smat_poll_errors.argtypes = [P, P, ctypes.POINTER(I32)]
    L.smat_debug_fused.argtypes = [P, U32, P, I32, U32, P]
    L.smat_delta_sigma_noalloc.argtypes = [P, P, I64, I32, ctypes.c_float, P, P]
    L.smat_delta_sigma_noalloc.restype = I32
    L.smat_timing_enable.argtypes = [P, I32]
    L.smat_timing_read.argtypes = [P, P, P]
    L.smat_status_string.argtypes = [I32]
    L.smat_status_string.restype = ctypes.c_char_p
    L.smat_last_error.argtypes = []
    L.smat_last_error.restype = ctypes.c_char_p
    L.smat_abi_version.restype = I32
    for name in ("smat_init", "smat_simulate_multi", "smat_grad_map_multi", "smat_grad_map_adamw_multi",
                 "smat_swap", "smat_active",
                 "smat_mask_bits", "smat_tensor_scalars", "smat_destroy", "smat_debug_philox", "smat_debug_noise_unit",
                 "smat_poll_errors", "smat_debug_fused", "smat_timing_enable", "smat_timing_read",
                 "smat_refill_theta0", "smat_mark_theta0_resident", "smat_merge", "smat_merge_ties_thresholds"):
        getattr(L, name).restype = I32
    _lib = L
    return L


def check(func: str, status: int):
    if status != 0:
        L = load_library()
        raise SmatError(func, L.smat_status_string(status).decode(), L.smat_last_error().decode())


def dtype_code(dt: torch.dtype) -> int:
    if dt == torch.float32:
        return SMAT_F32
    if dt == torch.bfloat16:
        return SMAT_BF16
    raise TypeError(f"unsupported dtype {dt} (float32 or bfloat16)")


def _stream_handle(stream: Optional[torch.cuda.Stream]):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


class SmatSession:
    """One smat_ctx over a list of trainable tensors.

    thetas / theta0s / sims: lists of contiguous CUDA tensors (theta read,
    theta0 read, sim = theta~ written), same dtype and numel per position.
    keep_probs, sigmas, sigma_rels: per-tensor p_keep (Eq. smat-mask, 1 - p),
    Perturb RMS, relative Perturb RMS. draw_bits: 32 (the default draw
    layout) or 16 (the 16-bit draw option, include/smat.h). The workspace is
    allocated here with torch and handed to the library.
    """

    def __init__(self, thetas: Sequence[torch.Tensor], theta0s: Sequence[torch.Tensor],
                 sims: Sequence[torch.Tensor], keep_probs: Sequence[float], sigmas: Sequence[float],
                 sigma_rels: Optional[Sequence[float]] = None, tensor_ids: Optional[Sequence[int]] = None,
                 elem_offsets: Optional[Sequence[int]] = None, seed: int = 0, alpha_min: float = 0.0,
                 alpha_max: float = 1.0, alpha_mode: int = SMAT_ALPHA_GLOBAL,
                 noise: int = SMAT_NOISE_UNIFORM, philox_rounds: int = 10, flags: int = 0,
                 stream: Optional[torch.cuda.Stream] = None, draw_bits: int = 32):
        self._L = load_library()
        n = len(thetas)
        if not (len(theta0s) == n and len(sims) == n and len(keep_probs) == n and len(sigmas) == n):
            raise ValueError("per-tensor lists differ in length")
        sigma_rels = sigma_rels if sigma_rels is not None else [0.0] * n
        tensor_ids = tensor_ids if tensor_ids is not None else list(range(n))
        elem_offsets = elem_offsets if elem_offsets is not None else [0] * n
        self.n = n
        self.numels = []
        descs = (TensorDesc * max(n, 1))()
        for k in range(n):
            th, t0, sm = thetas[k], theta0s[k], sims[k]
            for t in (th, t0, sm):
                # theta0 may live in pinned host memory: the kernels read it there
                if not t.is_contiguous() or not (t.is_cuda or (t is t0 and t.is_pinned())):
                    raise ValueError(f"tensor {k}: must be a contiguous CUDA tensor (theta0: or pinned host)")
            if th.dtype != t0.dtype or th.dtype != sm.dtype or th.numel() != t0.numel() or th.numel() != sm.numel():
                raise ValueError(f"tensor {k}: theta / theta0 / sim differ in dtype or numel")
            d = descs[k]
            d.theta, d.theta0, d.sim = th.data_ptr(), t0.data_ptr(), sm.data_ptr()
            d.numel = th.numel()
            d.elem_offset = int(elem_offsets[k])
            d.tensor_id = int(tensor_ids[k])
            d.dtype = dtype_code(th.dtype)
            d.keep_prob = float(keep_probs[k])
            d.sigma = float(sigmas[k])
            d.sigma_rel = float(sigma_rels[k])
            self.numels.append(th.numel())
        self._descs = descs
        self.config = Config(int(seed) & (2**64 - 1), float(alpha_min), float(alpha_max), int(alpha_mode),
                             int(noise), int(philox_rounds), int(flags), int(draw_bits))
        self.device = thetas[0].device if n else torch.device("cuda", torch.cuda.current_device())
        nbytes = self._L.smat_workspace_bytes(ctypes.byref(descs), n, ctypes.byref(self.config))
        if nbytes == 0 and n > 0:
            # size query failed: let smat_init report the reason
            nbytes = 256
        self.workspace = torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=self.device)
        self._keep = (list(thetas), list(theta0s), list(sims))  # the library holds raw pointers
        ctx = ctypes.c_void_p()
        check("smat_init", self._L.smat_init(ctypes.byref(ctx), ctypes.byref(descs), n, ctypes.byref(self.config),
                                             ctypes.c_void_p(self.workspace.data_ptr()), self.workspace.numel(),
                                             _stream_handle(stream)))
        self._ctx = ctx
        self._gkeep = None

    # -- hot path ------------------------------------------------------------
    def simulate_multi(self, step: int, stream: Optional[torch.cuda.Stream] = None):
        check("smat_simulate_multi", self._L.smat_simulate_multi(self._ctx, int(step), _stream_handle(stream)))

    def grad_map_multi(self, step: int, g_sims: Sequence[torch.Tensor], g_outs: Optional[Sequence[torch.Tensor]] = None,
                       accumulate: bool = False, stream: Optional[torch.cuda.Stream] = None):
        g_outs = g_sims if g_outs is None else g_outs
        if len(g_sims) != self.n or len(g_outs) != self.n:
            raise ValueError("one gradient per tensor expected")
        gd = None
        ins = (ctypes.c_void_p * max(self.n, 1))()
        outs = (ctypes.c_void_p * max(self.n, 1))()
        for k in range(self.n):
            a, b = g_sims[k], g_outs[k]
            if a.numel() != self.numels[k] or b.numel() != self.numels[k] or a.dtype != b.dtype:
                raise ValueError(f"gradient {k}: numel or dtype mismatch")
            if not (a.is_cuda and b.is_cuda and a.is_contiguous() and b.is_contiguous()):
                raise ValueError(f"gradient {k}: must be contiguous CUDA tensors")
            code = dtype_code(a.dtype)
            if gd is None:
                gd = code
            elif gd != code:
                raise ValueError("all gradients must share one dtype")
            ins[k], outs[k] = a.data_ptr(), b.data_ptr()
        self._gkeep = (list(g_sims), list(g_outs))
        check("smat_grad_map_multi",
              self._L.smat_grad_map_multi(self._ctx, int(step), ins, outs, SMAT_F32 if gd is None else gd,
                                          int(bool(accumulate)), _stream_handle(stream)))

    def grad_map_adamw_multi(self, step: int, g_sims: Sequence[torch.Tensor], m1s: Sequence[torch.Tensor],
                             m2s: Sequence[torch.Tensor], lr: float, beta1: float = 0.9, beta2: float = 0.999,
                             eps: float = 1e-8, weight_decay: float = 0.0, adam_step: int = 1,
                             stream: Optional[torch.cuda.Stream] = None):
        """The gradient map fused with one AdamW step: theta (the descriptors'
        own storage) and the fp32 moments m1s, m2s are updated in place."""
        if len(g_sims) != self.n or len(m1s) != self.n or len(m2s) != self.n:
            raise ValueError("one gradient and two moment buffers per tensor expected")
        gd = None
        gp = (ctypes.c_void_p * max(self.n, 1))()
        p1 = (ctypes.c_void_p * max(self.n, 1))()
        p2 = (ctypes.c_void_p * max(self.n, 1))()
        for k in range(self.n):
            g, a, b = g_sims[k], m1s[k], m2s[k]
            if g.numel() != self.numels[k] or a.numel() != self.numels[k] or b.numel() != self.numels[k]:
                raise ValueError(f"tensor {k}: numel mismatch")
            if a.dtype != torch.float32 or b.dtype != torch.float32:
                raise ValueError(f"tensor {k}: moments must be float32")
            if not all(x.is_cuda and x.is_contiguous() for x in (g, a, b)):
                raise ValueError(f"tensor {k}: must be contiguous CUDA tensors")
            code = dtype_code(g.dtype)
            if gd is None:
                gd = code
            elif gd != code:
                raise ValueError("all gradients must share one dtype")
            gp[k], p1[k], p2[k] = g.data_ptr(), a.data_ptr(), b.data_ptr()
        self._gkeep = (list(g_sims), list(m1s), list(m2s))
        opt = AdamW(float(lr), float(beta1), float(beta2), float(eps), float(weight_decay), int(adam_step))
        check("smat_grad_map_adamw_multi",
              self._L.smat_grad_map_adamw_multi(self._ctx, int(step), gp, p1, p2, SMAT_F32 if gd is None else gd,
                                                ctypes.byref(opt), _stream_handle(stream)))

    def swap(self) -> int:
        a = ctypes.c_int32()
        check("smat_swap", self._L.smat_swap(self._ctx, ctypes.byref(a)))
        return a.value

    @property
    def active(self) -> int:
        a = ctypes.c_int32()
        check("smat_active", self._L.smat_active(self._ctx, ctypes.byref(a)))
        return a.value

    # -- in-place mode (a tensor passed with sim == theta0) --------------------
    def refill_theta0(self, host_theta0s: Sequence[Optional[torch.Tensor]],
                      stream: Optional[torch.cuda.Stream] = None):
        """Copy theta0 from host tensors (pinned for an asynchronous copy) back
        into the sim buffers of the in-place tensors; other entries may be None."""
        if len(host_theta0s) != self.n:
            raise ValueError("one entry per tensor")
        ptrs = (ctypes.c_void_p * max(self.n, 1))()
        for k, h in enumerate(host_theta0s):
            if h is not None:
                if h.is_cuda or not h.is_contiguous() or h.numel() != self.numels[k]:
                    raise ValueError(f"tensor {k}: host theta0 must be a contiguous CPU tensor of the same size")
                ptrs[k] = h.data_ptr()
        self._hkeep = list(host_theta0s)  # the copies read them asynchronously
        check("smat_refill_theta0", self._L.smat_refill_theta0(self._ctx, ptrs, _stream_handle(stream)))

    def mark_theta0_resident(self):
        check("smat_mark_theta0_resident", self._L.smat_mark_theta0_resident(self._ctx))

    # -- test hooks ----------------------------------------------------------
    def mask_bits(self, step: int, k: int, stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
        # an out-of-range k is passed through so the library reports it
        words = (self.numels[k] + 31) // 32 if 0 <= k < self.n else 0
        out = torch.zeros(max(words, 1), dtype=torch.int32, device=self.device)
        check("smat_mask_bits", self._L.smat_mask_bits(self._ctx, int(step), int(k), ctypes.c_void_p(out.data_ptr()),
                                                       _stream_handle(stream)))
        return out[:words]

    def tensor_scalars(self, step: int, stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
        out = torch.zeros(max(self.n, 1), 4, dtype=torch.float32, device=self.device)
        check("smat_tensor_scalars", self._L.smat_tensor_scalars(self._ctx, int(step), ctypes.c_void_p(out.data_ptr()),
                                                                 _stream_handle(stream)))
        return out[:self.n]

    def poll_errors(self, stream: Optional[torch.cuda.Stream] = None) -> int:
        """Read and clear the device error flags (0 = none); synchronises the stream."""
        v = ctypes.c_int32()
        check("smat_poll_errors", self._L.smat_poll_errors(self._ctx, _stream_handle(stream), ctypes.byref(v)))
        return v.value

    def debug_fused(self, step: int, items: torch.Tensor, epoch_skew: int,
                    stream: Optional[torch.cuda.Stream] = None):
        """Test hook smat_debug_fused (items: int32 CUDA tensor of work items)."""
        items = items.contiguous()
        check("smat_debug_fused", self._L.smat_debug_fused(self._ctx, int(step), ctypes.c_void_p(items.data_ptr()),
                                                           items.numel(), int(epoch_skew), _stream_handle(stream)))

    def timing_enable(self, enable: bool = True):
        check("smat_timing_enable", self._L.smat_timing_enable(self._ctx, int(bool(enable))))

    TIMING_KINDS = ("delta_stats", "scalars", "simulate", "gradmap")

    def timing_read(self):
        """{kind: (total kernel ms, launches)} since timing_enable()."""
        ms = (ctypes.c_double * 4)()
        n = (ctypes.c_int64 * 4)()
        check("smat_timing_read", self._L.smat_timing_read(self._ctx, ms, n))
        return {k: (ms[i], n[i]) for i, k in enumerate(self.TIMING_KINDS)}

    def close(self):
        if getattr(self, "_ctx", None):
            self._L.smat_destroy(self._ctx)
            self._ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def debug_philox(ctr: torch.Tensor, seed: int, rounds: int = 10, with_curand: bool = True,
                 stream: Optional[torch.cuda.Stream] = None):
    """Device Philox blocks for counters ctr (int32 CUDA tensor [n, 4]); also
    cuRAND's curand_Philox4x32_10 on the same inputs when with_curand."""
    L = load_library()
    ctr = ctr.contiguous()
    n = ctr.shape[0]
    out = torch.zeros_like(ctr)
    ref = torch.zeros_like(ctr) if with_curand else None
    check("smat_debug_philox", L.smat_debug_philox(ctypes.c_void_p(ctr.data_ptr()), n, int(seed) & (2**64 - 1), rounds,
                                                   ctypes.c_void_p(out.data_ptr()),
                                                   ctypes.c_void_p(ref.data_ptr() if ref is not None else 0),
                                                   _stream_handle(stream)))
    return out, ref


def debug_noise_unit(words: torch.Tensor, noise: int, stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """Unit noise transform of raw words (int32 CUDA tensor): sym(w) or
    erfinv(sym(w)) exactly as the forward evaluates it."""
    L = load_library()
    words = words.contiguous()
    out = torch.empty(words.shape, dtype=torch.float32, device=words.device)
    check("smat_debug_noise_unit", L.smat_debug_noise_unit(ctypes.c_void_p(words.data_ptr()), words.numel(), int(noise),
                                                           ctypes.c_void_p(out.data_ptr()), _stream_handle(stream)))
    return out


def delta_sigma_noalloc(theta: torch.Tensor, theta0: torch.Tensor, sigma_rel: float,
                        out: Optional[torch.Tensor] = None, stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """smat_delta_sigma_noalloc: sigma_rel * std(theta - theta0) computed with
    the library's fixed scratch array instead of any device allocation (the
    result buffer `out`, one float on the device, is the caller's)."""
    L = load_library()
    if theta.dtype != theta0.dtype or theta.numel() != theta0.numel():
        raise ValueError("theta and theta0 differ in dtype or numel")
    if not (theta.is_cuda and theta0.is_cuda and theta.device == theta0.device):
        raise ValueError("theta and theta0 must be CUDA tensors on one device")
    if not (theta.is_contiguous() and theta0.is_contiguous()):
        raise ValueError("theta and theta0 must be contiguous")
    if out is None:
        out = torch.empty(1, dtype=torch.float32, device=theta.device)
    if not (out.is_cuda and out.device == theta.device and out.dtype == torch.float32 and out.numel() >= 1):
        raise ValueError("out must be a float32 CUDA tensor of at least one element on theta's device")
    with torch.cuda.device(theta.device):
        check("smat_delta_sigma_noalloc",
              L.smat_delta_sigma_noalloc(ctypes.c_void_p(theta.data_ptr()), ctypes.c_void_p(theta0.data_ptr()),
                                         theta.numel(), dtype_code(theta.dtype), float(sigma_rel),
                                         ctypes.c_void_p(out.data_ptr()), _stream_handle(stream)))
    return out


class SmatParameters:
    """Parameter storage switching for a list of torch Parameters (Sec. 4.3):
    keeps theta0 and one reusable simulated-weight buffer per parameter and
    rebinds each parameter's storage between theta and theta~ on swap(), with
    no copy. The optimizer must run with the original storage active."""

    def __init__(self, params: List[torch.nn.Parameter], theta0s: Sequence[torch.Tensor],
                 keep_probs: Sequence[float], sigmas: Sequence[float], **cfg):
        self.params = list(params)
        self.theta = [p.data for p in self.params]
        self.sims = [torch.empty_like(p.data) for p in self.params]
        self.session = SmatSession(self.theta, list(theta0s), self.sims, keep_probs, sigmas, **cfg)

    def simulate(self, step: int):
        self.session.simulate_multi(step)

    def swap(self) -> int:
        active = self.session.swap()
        src = self.sims if active == 1 else self.theta
        for p, t in zip(self.params, src):
            p.data = t
        return active

    def grad_map(self, step: int, accumulate: bool = False):
        gs = [p.grad for p in self.params]
        self.session.grad_map_multi(step, gs, gs, accumulate=accumulate)


# ------------------------------------------------------------------ merging ---
SMAT_MERGE_WA, SMAT_MERGE_TA, SMAT_MERGE_DARE_TA, SMAT_MERGE_TIES = 0, 1, 2, 3


class MergeTensor(ctypes.Structure):
    _fields_ = [("theta0", ctypes.c_void_p), ("experts", ctypes.c_void_p), ("out", ctypes.c_void_p),
                ("numel", ctypes.c_int64), ("elem_offset", ctypes.c_int64), ("tensor_id", ctypes.c_uint32),
                ("dtype", ctypes.c_int32)]


class MergeConfig(ctypes.Structure):
    _fields_ = [("method", ctypes.c_int32), ("n_experts", ctypes.c_int32), ("gamma", ctypes.c_float),
                ("p_drop", ctypes.c_float), ("retention", ctypes.c_float), ("seed", ctypes.c_uint64),
                ("philox_rounds", ctypes.c_int32), ("flags", ctypes.c_int32)]


def merge(theta0s: Sequence[torch.Tensor], experts: Sequence[Sequence[torch.Tensor]], outs: Sequence[torch.Tensor],
          method: int, gamma: float = 1.0, p_drop: float = 0.0, retention: float = 1.0, seed: int = 0,
          tensor_ids: Optional[Sequence[int]] = None, elem_offsets: Optional[Sequence[int]] = None,
          philox_rounds: int = 10, stream: Optional[torch.cuda.Stream] = None, return_thresholds: bool = False):
    """Merge K experts per tensor into outs (Eq. merged-state; see smat_merge
    in include/smat.h): experts[k] lists tensor k's K expert tensors. outs[k]
    may be theta0s[k]. With return_thresholds (TIES), returns the
    n_tensors x K threshold keys (int32 view of the uint32 bits)."""
    L = load_library()
    n = len(theta0s)
    if len(experts) != n or len(outs) != n:
        raise ValueError("per-tensor lists differ in length")
    K = len(experts[0]) if n else 0
    tensor_ids = tensor_ids if tensor_ids is not None else list(range(n))
    elem_offsets = elem_offsets if elem_offsets is not None else [0] * n
    descs = (MergeTensor * max(n, 1))()
    keep = []
    for k in range(n):
        if len(experts[k]) != K:
            raise ValueError("every tensor needs the same number of experts")
        for t in [theta0s[k], outs[k], *experts[k]]:
            if not t.is_contiguous() or t.numel() != theta0s[k].numel() or t.dtype != theta0s[k].dtype:
                raise ValueError(f"tensor {k}: contiguous tensors of one shape and dtype")
        ptrs = (ctypes.c_void_p * max(K, 1))(*[x.data_ptr() for x in experts[k]])
        keep.append(ptrs)
        d = descs[k]
        d.theta0, d.out = theta0s[k].data_ptr(), outs[k].data_ptr()
        d.experts = ctypes.cast(ptrs, ctypes.c_void_p)
        d.numel = theta0s[k].numel()
        d.elem_offset = int(elem_offsets[k])
        d.tensor_id = int(tensor_ids[k])
        d.dtype = dtype_code(theta0s[k].dtype)
    cfg = MergeConfig(int(method), K, float(gamma), float(p_drop), float(retention), int(seed) & (2**64 - 1),
                      int(philox_rounds), 0)
    nbytes = L.smat_merge_workspace_bytes(ctypes.byref(descs), n, ctypes.byref(cfg))
    device = outs[0].device if n else torch.device("cuda", torch.cuda.current_device())
    ws = torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)
    check("smat_merge", L.smat_merge(ctypes.byref(descs), n, ctypes.byref(cfg), ctypes.c_void_p(ws.data_ptr()),
                                     ws.numel(), _stream_handle(stream)))
    if stream is not None:
        ws.record_stream(stream)
    if return_thresholds:
        thr = torch.empty(max(n * K, 1), dtype=torch.int32, device=device)
        check("smat_merge_ties_thresholds",
              L.smat_merge_ties_thresholds(ctypes.byref(descs), n, ctypes.byref(cfg), ctypes.c_void_p(ws.data_ptr()),
                                           ctypes.c_void_p(thr.data_ptr()), _stream_handle(stream)))
        return thr[:n * K].view(n, K)
    return None
