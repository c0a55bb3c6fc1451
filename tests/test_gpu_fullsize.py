"""Full-size parity: the 0.5B, 7B and vision-language lists at their stated
sizes, in the launch configuration the bench times, checked at sampled
elements against the CPU oracle (which evaluates elements one by one), and
through properties that hold at any size (binomial keep rate per tensor,
sigma_t against the oracle's two-pass statistics)."""

import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import workloads as W

from _parity import compare, f32_of, orc_config, orc_tensor, session_for, to_host

pytestmark = pytest.mark.gpu

SAMPLES = 768


def _popcount(words: torch.Tensor) -> int:
    w = words.to(torch.int64) & 0xFFFFFFFF
    c = torch.zeros_like(w)
    for b in range(32):
        c += (w >> b) & 1
    return int(c.sum())


def _check_workload(w: W.Workload, step: int = 0, draw_bits: int = 32):
    dev = torch.device("cuda")
    free, total = torch.cuda.mem_get_info()
    need = (2 if w.dtype == O.BF16 else 4) * w.numel * 3 + (2 if w.gdtype == O.BF16 else 4) * w.numel * 2
    if need > free * 0.9:
        pytest.skip(f"needs {need / 1e9:.1f} GB of device memory, {free / 1e9:.1f} GB free")
    th, t0, sim, gs, go = W.generate(w, device=dev)
    sess = session_for(w, th, t0, sim, draw_bits=draw_bits)
    sess.simulate_multi(step)
    sess.swap()
    sess.grad_map_multi(step, gs, go)
    sess.swap()
    scal = sess.tensor_scalars(step).cpu().numpy()
    torch.cuda.synchronize()
    cfg = orc_config(w, step, draw_bits=draw_bits)
    rng = np.random.default_rng(77)
    for k, spec in enumerate(w.tensors):
        n = spec.numel
        idx = np.unique(np.concatenate([np.arange(min(n, 16)), np.arange(max(0, n - 16), n),
                                        rng.integers(0, n, size=min(n, SAMPLES))]))
        it = torch.from_numpy(idx).to(dev)
        t = orc_tensor(w, k)
        if spec.sigma_rel > 0:
            sig = O.delta_stats(t, to_host(th[k]), to_host(t0[k]))["sigma"]
            assert abs(float(scal[k, 2]) - sig) <= 1e-5 * sig, f"tensor {k} sigma"
        else:
            sig = spec.sigma
        thv = f32_of(to_host(th[k][it]))
        t0v = f32_of(to_host(t0[k][it]))
        ref, kept = O.simulate_at(cfg, t, sig, idx, thv, t0v)
        mode = O.NOISE_GAUSSIAN if spec.sigma_rel > 0 else w.noise
        compare(to_host(sim[k][it]), ref, w.dtype, mode, thv, t0v, what=f"{w.name} tensor {k} ({spec.name})")
        gref = O.gradmap_at(cfg, t, idx, f32_of(to_host(gs[k][it])), gdtype=w.gdtype)
        gv = np.uint16 if w.gdtype == O.BF16 else np.uint32
        assert np.array_equal(to_host(go[k][it]).view(gv), gref.astype(gv)), f"tensor {k} gradmap"
        words = sess.mask_bits(step, k)
        wh = words.cpu().numpy().view(np.uint32)
        gbits = (wh[idx >> 5] >> (idx & 31).astype(np.uint32)) & 1
        assert np.array_equal(gbits.astype(np.uint8), kept), f"tensor {k} mask bits"
        p = float(np.float32(spec.keep_prob))
        if draw_bits == 16:
            p = math.floor(p * 65536) / 65536  # the 16-bit threshold
        if 0.0 < p < 1.0:
            kcount = _popcount(words)
            assert abs(kcount - n * p) <= 5 * math.sqrt(n * p * (1 - p)) + 1, f"tensor {k} keep rate"
    sess.close()
    del th, t0, sim, gs, go
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["dec_0p5b", "llama_7b", "vl_7b"])
def test_full_size_list_sampled(name):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    _check_workload(W.WORKLOADS[name]())


def test_flat_2_32_plus_ragged_bf16_sampled():
    """2^32 + 17 elements in one tensor: 64-bit element indexing end to end."""
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    w = W.flat_sweep(32, O.BF16, 0.3, 2, 1e-4)
    w.tensors[0].shape = ((1 << 32) + 17,)
    _check_workload(w, step=1)


def test_full_size_7b_list_draw16_sampled():
    """The 7B list with the 16-bit draw option, in the launch configuration
    `bench.py --draw-bits 16` times (the four-CTA work-list build with the
    statistics items), sampled against the oracle with the same option."""
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    _check_workload(W.llama_7b(), step=3, draw_bits=16)


@pytest.mark.parametrize("draw_bits", [32, 16])
def test_full_size_7b_list_fused_adamw_sampled(draw_bits):
    """The gradient map fused with AdamW on the whole 7B list in the launch
    configuration `bench.py --adamw` times (one call per optimizer step after
    the forward of its own SMAT step, warm moments): theta, m1 and m2 bit-exact
    against the oracle at sampled elements (each tensor's first and last 16
    and random ones), over two optimizer steps."""
    w = W.llama_7b()
    dev = torch.device("cuda")
    free, total = torch.cuda.mem_get_info()
    need = 2 * w.numel * 4 + 4 * w.numel * 2
    if need > free * 0.9:
        pytest.skip(f"needs {need / 1e9:.1f} GB of device memory, {free / 1e9:.1f} GB free")
    th, t0, sim, gs, _ = W.generate(w, device=dev, with_grad=True)
    gen = torch.Generator(device=dev).manual_seed(w.data_seed + 17)
    m1 = [torch.randn(t.numel, generator=gen, device=dev) * 1e-3 for t in w.tensors]
    m2 = [torch.rand(t.numel, generator=gen, device=dev) * 1e-6 for t in w.tensors]
    sess = session_for(w, th, t0, sim, draw_bits=draw_bits)
    rng = np.random.default_rng(91)
    picks = []
    for k, spec in enumerate(w.tensors):
        n = spec.numel
        idx = np.unique(np.concatenate([np.arange(min(n, 16)), np.arange(max(0, n - 16), n),
                                        rng.integers(0, n, size=min(n, SAMPLES // 4))]))
        it = torch.from_numpy(idx).to(dev)
        picks.append((idx, it, f32_of(to_host(th[k][it])), to_host(m1[k][it]), to_host(m2[k][it]),
                      f32_of(to_host(gs[k][it]))))
    hp = dict(lr=1e-5, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
    for t_opt, step in enumerate((3, 4), start=1):
        sess.simulate_multi(step)
        sess.grad_map_adamw_multi(step, gs, m1, m2, adam_step=t_opt, **hp)
        torch.cuda.synchronize()
        cfg = orc_config(w, step, draw_bits=draw_bits)
        for k in range(len(w.tensors)):
            idx, it, thv, a, b, gv = picks[k]
            bits, a, b = O.gradmap_adamw_at(cfg, orc_tensor(w, k), idx, gv, thv, a, b, adam_step=t_opt,
                                            gdtype=w.gdtype, **hp)
            got = to_host(th[k][it])
            assert np.array_equal(got.astype(np.uint32) if w.dtype == O.BF16 else got.view(np.uint32), bits), \
                f"step {step} tensor {k} theta"
            assert np.array_equal(to_host(m1[k][it]).view(np.uint32), a.view(np.uint32)), f"tensor {k} m1"
            assert np.array_equal(to_host(m2[k][it]).view(np.uint32), b.view(np.uint32)), f"tensor {k} m2"
            thv = f32_of(got)
            picks[k] = (idx, it, thv, a, b, gv)
    assert sess.poll_errors() == 0
    sess.close()
