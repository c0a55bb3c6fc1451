"""Helpers of the GPU-vs-oracle parity tests: run a workload through the C ABI
and compare with the CPU oracle element by element (small lists) or at
sampled elements (full-size lists).

Tolerances (written out in compare()):
  masks, gradient map, uniform-noise forward: bit-exact;
  Gaussian-noise forward, fp32: |gpu - cpu| <= 1e-6 max(|cpu|, |theta|, |theta0|, 2^-126);
  Gaussian-noise forward, bf16: at most 1 bf16 ulp apart, or, only where the
    sum cancels (|cpu| <= 2^-8 max(|theta|, |theta0|): the result is at least
    256 times smaller than its inputs), |gpu - cpu| <= 1e-6 max(|theta|,
    |theta0|) (the fp32 bound on the input scale); at most CANCEL_MAX elements
    per comparison may use that escape, and the count is printed.
"""

import numpy as np
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300 import workloads as W

FP32_RTOL = 1e-6
BF16_ULPS = 1
CANCEL_RATIO = 2.0**-8
CANCEL_MAX = 8


def to_host(x: torch.Tensor) -> np.ndarray:
    x = x.detach().cpu().contiguous()
    if x.dtype == torch.bfloat16:
        return x.view(torch.int16).numpy().view(np.uint16).copy()
    return x.numpy().copy()


def f32_of(bits: np.ndarray) -> np.ndarray:
    if bits.dtype == np.uint16:
        return O.bf16_to_f32(bits)
    return bits.astype(np.float32)


def orc_config(w: W.Workload, step: int, rounds: int = 10, draw_bits: int = 32):
    return O.config(seed=w.seed, step=step, rounds=rounds, alpha_mode=w.alpha_mode, noise=w.noise,
                    alpha_min=w.alpha_min, alpha_max=w.alpha_max, draw_bits=draw_bits)


def orc_tensor(w: W.Workload, k: int, numel=None, elem_offset=0):
    t = w.tensors[k]
    return O.tensor(k, t.numel if numel is None else numel, dtype=w.dtype, keep_prob=t.keep_prob, sigma=t.sigma,
                    sigma_rel=t.sigma_rel, elem_offset=elem_offset)


def session_for(w: W.Workload, th, t0, sim, rounds: int = 10, elem_offsets=None, flags: int = 0,
                draw_bits: int = 32):
    return S.SmatSession(th, t0, sim, [t.keep_prob for t in w.tensors], [t.sigma for t in w.tensors],
                         [t.sigma_rel for t in w.tensors], elem_offsets=elem_offsets, seed=w.seed,
                         alpha_min=w.alpha_min, alpha_max=w.alpha_max, alpha_mode=w.alpha_mode, noise=w.noise,
                         philox_rounds=rounds, flags=flags, draw_bits=draw_bits)


def _ordered_bf16(b: np.ndarray) -> np.ndarray:
    b = b.astype(np.int64)
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


def as_bits(a, dtype) -> np.ndarray:
    """Storage bits of an output: bf16 as uint16, fp32 as uint32 (float arrays
    are reinterpreted, never converted)."""
    a = np.asarray(a)
    if dtype == O.BF16:
        if a.dtype == np.uint16:
            return a
        if a.dtype == np.uint32:
            assert int(a.max(initial=0)) < 65536
            return a.astype(np.uint16)
    else:
        if a.dtype == np.float32:
            return a.view(np.uint32)
        if a.dtype == np.uint32:
            return a
    raise TypeError(f"unexpected array dtype {a.dtype} for storage dtype {dtype}")


def compare(got_bits, ref_bits, dtype, noise, th=None, t0=None, what=""):
    """Assert GPU bits match oracle bits within the stated tolerance."""
    got_bits = as_bits(got_bits, dtype)
    ref_bits = as_bits(ref_bits, dtype)
    g = f32_of(got_bits) if dtype == O.BF16 else got_bits.view(np.float32)
    r = f32_of(ref_bits) if dtype == O.BF16 else ref_bits.view(np.float32)
    nan_g, nan_r = np.isnan(g), np.isnan(r)
    assert np.array_equal(nan_g, nan_r), f"{what}: NaN pattern differs"
    # an infinity on either side must be the same infinity on both
    inf = np.isinf(g) | np.isinf(r)
    assert np.array_equal(g[inf], r[inf]), f"{what}: {int((g[inf] != r[inf]).sum())} infinities differ"
    ok = ~nan_r & ~inf
    if noise == O.NOISE_UNIFORM:
        bad = np.nonzero(got_bits[ok] != ref_bits[ok])[0]
        assert bad.size == 0, f"{what}: {bad.size} elements differ (exact expected); first {np.nonzero(ok)[0][bad[:5]]}"
        return
    if dtype == O.BF16:
        d = np.abs(_ordered_bf16(got_bits[ok]) - _ordered_bf16(ref_bits[ok]))
        far = d > BF16_ULPS
        if far.any() and th is not None:
            # Where theta0 + ... + eps cancels, a bf16 ulp of the result is far
            # below the fp32 rounding of the inputs: such elements (and only
            # those) take the fp32 bound on the input scale instead.
            scale = np.maximum(np.abs(np.asarray(th, np.float64)[ok]), np.abs(np.asarray(t0, np.float64)[ok]))
            rr = np.abs(r[ok].astype(np.float64))
            err = np.abs(g[ok].astype(np.float64) - r[ok].astype(np.float64))
            cancels = rr <= CANCEL_RATIO * scale
            escaped = far & cancels & (err <= FP32_RTOL * np.maximum(scale, 2.0**-126))
            n_esc = int(escaped.sum())
            if n_esc:
                print(f"{what}: {n_esc} cancelling element(s) compared on the fp32 input-scale bound")
            assert n_esc <= CANCEL_MAX, f"{what}: {n_esc} elements needed the cancellation escape (at most {CANCEL_MAX})"
            far &= ~escaped
        assert not far.any(), f"{what}: {int(far.sum())} elements beyond {BF16_ULPS} ulp and the cancellation bound"
        return
    scale = np.abs(r[ok]).astype(np.float64)
    if th is not None:
        scale = np.maximum(scale, np.abs(np.asarray(th, np.float64)[ok]))
        scale = np.maximum(scale, np.abs(np.asarray(t0, np.float64)[ok]))
    scale = np.maximum(scale, 2.0**-126)
    err = np.abs(g[ok].astype(np.float64) - r[ok].astype(np.float64))
    bad = err > FP32_RTOL * scale
    assert not bad.any(), f"{what}: {int(bad.sum())} elements beyond 1e-6 relative (max ratio {float((err / scale).max())})"


def run_and_check_full(w: W.Workload, steps=(0, 1, 2), rounds=10, accumulate=False, gdtype=None, flags=0,
                       draw_bits=32):
    """Generate w on the GPU, run simulate + gradient map for each step through
    the C ABI and compare every element with the oracle."""
    dev = torch.device("cuda")
    th, t0, sim, gs, go = W.generate(w, device=dev)
    if gdtype is not None:
        gs = [g.to(W.torch_dtype(gdtype)) for g in gs]
        go = [torch.empty_like(g) for g in gs]
    gdt = w.gdtype if gdtype is None else gdtype
    sess = session_for(w, th, t0, sim, rounds=rounds, flags=flags, draw_bits=draw_bits)
    hth = [to_host(x) for x in th]
    ht0 = [to_host(x) for x in t0]
    hgs = [to_host(x) for x in gs]
    for step in steps:
        if accumulate:
            for g in go:
                g.copy_(torch.randn(g.shape, device=dev).to(g.dtype))
        hgo_before = [to_host(x) for x in go] if accumulate else None
        sess.simulate_multi(step)
        sess.swap()
        sess.grad_map_multi(step, gs, go, accumulate=accumulate)
        sess.swap()
        scal = sess.tensor_scalars(step).cpu().numpy()
        torch.cuda.synchronize()
        cfg = orc_config(w, step, rounds, draw_bits)
        for k in range(len(w.tensors)):
            t = orc_tensor(w, k)
            ref = O.simulate(cfg, t, hth[k], ht0[k])
            # sigma_rel tensors: sigma_t comes from a reduction whose rounding order
            # differs between the two sides (1e-5 relative), so the forward is
            # compared within the float tolerance even with uniform noise.
            mode = O.NOISE_GAUSSIAN if w.tensors[k].sigma_rel > 0 else w.noise
            compare(to_host(sim[k]), ref.view(np.uint16 if w.dtype == O.BF16 else np.uint32), w.dtype, mode,
                    f32_of(hth[k]), f32_of(ht0[k]), what=f"{w.name} step {step} tensor {k} simulate")
            gref = O.gradmap(cfg, t, hgs[k], gdtype=gdt, accumulate=accumulate,
                             g_old=hgo_before[k] if accumulate else None)
            gv = np.uint16 if gdt == O.BF16 else np.uint32
            assert np.array_equal(to_host(go[k]).view(gv), gref.view(gv)), f"{w.name} step {step} tensor {k} gradmap"
            bits = sess.mask_bits(step, k).cpu().numpy().view(np.uint32)
            assert np.array_equal(bits, O.mask_bits(cfg, t)), f"{w.name} step {step} tensor {k} mask bits"
            s = O.scalars(cfg, t, hth[k], ht0[k])
            if w.alpha_mode != O.ALPHA_PER_ELEMENT:
                assert np.float32(scal[k, 0]) == np.float32(s["alpha"]), "alpha"
                assert np.float32(scal[k, 1]) == np.float32(s["c"]), "c"
            assert abs(float(scal[k, 2]) - s["sigma"]) <= 1e-5 * abs(s["sigma"]) + 1e-30, "sigma"
    assert sess.poll_errors() == 0
    sess.close()
