"""The gradient map fused with an AdamW step (smat_grad_map_adamw_multi)
through the C ABI, against the oracle's definition (oracle.gradmap_adamw:
Eq. smat-gradient's stored gradient feeding one decoupled-weight-decay AdamW
step, each fp32 operation rounded in a fixed order). theta, m1 and m2 are
compared bit for bit over several optimizer steps, each after a forward of
its own SMAT step, on ragged lists (element path, chunk and unit
boundaries), every alpha mode, both draw layouts and round counts, fp32 and
bf16 parameters and gradients, and lists that mix the two parameter dtypes;
refused calls leave every buffer untouched."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300 import workloads as W

from _parity import orc_config, orc_tensor, session_for, to_host

pytestmark = pytest.mark.gpu

HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    yield
    torch.cuda.synchronize()


def _ragged(dtype, gdtype, alpha_mode, seed=0xADA3_0001):
    sizes = [0, 1, 7, 15, 16, 17, 33, 131_073, 262_144, 262_153, 600_003]
    keeps = [0.5, 0.9, 0.1, 0.7, 1.0, 0.0, 0.3, 0.5 + 2**-10, 0.9, 0.3, 0.7]
    specs = [W.TensorSpec(f"t{i}", (n,), "linear", keeps[i], 1e-3) for i, n in enumerate(sizes)]
    return W.Workload(f"adamw_{dtype}_{gdtype}_{alpha_mode}", specs, dtype, gdtype, 0.2, 1.0, alpha_mode,
                      O.NOISE_UNIFORM, 0.02, 1e-3, seed=seed)


def _moments(w, dev, seed):
    """Nonzero starting moments (m2 >= 0), as after earlier optimizer steps."""
    g = torch.Generator(device=dev).manual_seed(seed)
    m1 = [torch.randn(t.numel, generator=g, device=dev) * 1e-3 for t in w.tensors]
    m2 = [torch.rand(t.numel, generator=g, device=dev) * 1e-6 for t in w.tensors]
    return m1, m2


def _run(w, steps, rounds=10, draw_bits=32, hp=HP, zero_moments=False):
    dev = torch.device("cuda")
    th, t0, sim, gs, _ = W.generate(w, device=dev)
    if zero_moments:
        m1 = [torch.zeros(t.numel, device=dev) for t in w.tensors]
        m2 = [torch.zeros(t.numel, device=dev) for t in w.tensors]
    else:
        m1, m2 = _moments(w, dev, w.seed)
    sess = session_for(w, th, t0, sim, rounds=rounds, draw_bits=draw_bits)
    hth = [to_host(x) for x in th]
    h1 = [to_host(x) for x in m1]
    h2 = [to_host(x) for x in m2]
    hgs = [to_host(x) for x in gs]
    for t_opt, step in enumerate(steps, start=1):
        sess.simulate_multi(step)
        assert sess.swap() == 1
        assert sess.swap() == 0  # the model ran on theta~; the storage is switched back
        sess.grad_map_adamw_multi(step, gs, m1, m2, adam_step=t_opt, **hp)
        torch.cuda.synchronize()
        cfg = orc_config(w, step, rounds, draw_bits)
        for k in range(len(w.tensors)):
            t = orc_tensor(w, k)
            hth[k], h1[k], h2[k] = O.gradmap_adamw(cfg, t, hgs[k], hth[k], h1[k], h2[k], adam_step=t_opt,
                                                   gdtype=w.gdtype, **hp)
            tv = np.uint16 if w.dtype == O.BF16 else np.uint32
            what = f"{w.name} step {step} tensor {k}"
            assert np.array_equal(to_host(th[k]).view(tv), hth[k].view(tv)), what + " theta"
            assert np.array_equal(to_host(m1[k]).view(np.uint32), h1[k].view(np.uint32)), what + " m1"
            assert np.array_equal(to_host(m2[k]).view(np.uint32), h2[k].view(np.uint32)), what + " m2"
    assert sess.poll_errors() == 0
    sess.close()


@pytest.mark.parametrize("alpha_mode", [O.ALPHA_GLOBAL, O.ALPHA_PER_TENSOR, O.ALPHA_PER_ELEMENT])
@pytest.mark.parametrize("dtype,gdtype", [(O.F32, O.F32), (O.BF16, O.BF16), (O.BF16, O.F32), (O.F32, O.BF16)])
def test_fused_adamw_bit_exact_on_a_ragged_list(dtype, gdtype, alpha_mode):
    _run(_ragged(dtype, gdtype, alpha_mode), steps=(0, 1, 5))


@pytest.mark.parametrize("draw_bits,rounds", [(16, 10), (32, 7), (16, 7)])
def test_fused_adamw_draw_layouts_and_round_counts(draw_bits, rounds):
    _run(_ragged(O.BF16, O.BF16, O.ALPHA_PER_ELEMENT), steps=(2, 3), rounds=rounds, draw_bits=draw_bits)


def test_fused_adamw_from_zero_moments_and_without_decay():
    """The first optimizer step from zero moments (the update is then
    lr g / (|g| + eps') elementwise) and weight decay 0 (decay factor 1)."""
    hp = dict(HP, weight_decay=0.0, lr=3e-4)
    _run(_ragged(O.BF16, O.BF16, O.ALPHA_PER_TENSOR), steps=(4,), hp=hp, zero_moments=True)


def _mixed_list(dev, sizes, dtypes, offsets):
    """A list mixing fp32 and bf16 parameters; offsets (in elements) into larger
    buffers break the 32-byte alignment of some tensors."""
    g = torch.Generator(device=dev).manual_seed(77)
    bufs = []
    for n, dt, off in zip(sizes, dtypes, offsets):
        b0 = torch.randn(n + off, generator=g, device=dev) * 0.02
        b1 = b0 + torch.randn(n + off, generator=g, device=dev) * 1e-3
        bufs.append((b1.to(dt)[off:], b0.to(dt)[off:], torch.empty(n + off, dtype=dt, device=dev)[off:]))
    return bufs


def test_fused_adamw_mixed_dtypes_misaligned_and_offset_tensors():
    dev = torch.device("cuda")
    sizes = [100_003, 17, 262_160, 4096, 33]
    dtypes = [torch.float32, torch.bfloat16, torch.bfloat16, torch.float32, torch.bfloat16]
    offsets = [0, 1, 3, 8, 16]
    elem_offsets = [0, 5, 16, 2**36 + 3, 2**35]
    keeps = [0.7, 0.5, 0.9, 0.3, 1.0]
    bufs = _mixed_list(dev, sizes, dtypes, offsets)
    th = [b[0] for b in bufs]
    t0 = [b[1] for b in bufs]
    sim = [b[2] for b in bufs]
    gen = torch.Generator(device=dev).manual_seed(5)
    gs = [torch.randn(n, generator=gen, device=dev) for n in sizes]
    m1 = [torch.randn(n, generator=gen, device=dev) * 1e-3 for n in sizes]
    m2 = [torch.rand(n, generator=gen, device=dev) * 1e-6 for n in sizes]
    sess = S.SmatSession(th, t0, sim, keeps, [1e-3] * 5, elem_offsets=elem_offsets, seed=31, alpha_min=0.2,
                         alpha_max=1.0, alpha_mode=S.SMAT_ALPHA_PER_ELEMENT, noise=S.SMAT_NOISE_GAUSSIAN)
    hth = [to_host(x) for x in th]
    h1 = [to_host(x) for x in m1]
    h2 = [to_host(x) for x in m2]
    for t_opt, step in enumerate((0, 9), start=1):
        sess.simulate_multi(step)
        sess.grad_map_adamw_multi(step, gs, m1, m2, adam_step=t_opt, **HP)
        torch.cuda.synchronize()
        cfg = O.config(seed=31, step=step, alpha_mode=O.ALPHA_PER_ELEMENT, noise=O.NOISE_GAUSSIAN, alpha_min=0.2)
        for k in range(5):
            odt = O.F32 if dtypes[k] == torch.float32 else O.BF16
            t = O.tensor(k, sizes[k], odt, keep_prob=keeps[k], sigma=1e-3, elem_offset=elem_offsets[k])
            hth[k], h1[k], h2[k] = O.gradmap_adamw(cfg, t, to_host(gs[k]), hth[k], h1[k], h2[k], adam_step=t_opt,
                                                   gdtype=O.F32, **HP)
            tv = np.uint16 if odt == O.BF16 else np.uint32
            assert np.array_equal(to_host(th[k]).view(tv), hth[k].view(tv)), f"step {step} tensor {k} theta"
            assert np.array_equal(to_host(m1[k]).view(np.uint32), h1[k].view(np.uint32)), f"tensor {k} m1"
            assert np.array_equal(to_host(m2[k]).view(np.uint32), h2[k].view(np.uint32)), f"tensor {k} m2"
    assert sess.poll_errors() == 0
    sess.close()


def test_fused_adamw_matches_the_separate_gradient_map():
    """The gradient the fused call consumes is the one smat_grad_map_multi
    stores: AdamW with lr 0 and beta1 = beta2 = 0 leaves m1 = fl(1 * g) = g
    and m2 = g * g, so m1 after the fused call equals the separate map's
    output bit for bit (bf16 gradients: the stored value after rounding)."""
    w = _ragged(O.BF16, O.BF16, O.ALPHA_PER_ELEMENT, seed=0xADA3_0002)
    dev = torch.device("cuda")
    th, t0, sim, gs, go = W.generate(w, device=dev)
    m1 = [torch.full((t.numel,), 5.0, device=dev) for t in w.tensors]
    m2 = [torch.full((t.numel,), 5.0, device=dev) for t in w.tensors]
    sess = session_for(w, th, t0, sim)
    before = [to_host(x) for x in th]
    sess.simulate_multi(6)
    sess.grad_map_multi(6, gs, go)
    sess.grad_map_adamw_multi(6, gs, m1, m2, lr=0.0, beta1=0.0, beta2=0.0, eps=1.0, weight_decay=0.0)
    torch.cuda.synchronize()
    for k in range(len(w.tensors)):
        g = go[k].float()
        assert torch.equal(m1[k], g), k
        assert torch.equal(m2[k], g * g), k
        assert np.array_equal(to_host(th[k]), before[k]), k  # lr 0: theta unchanged
    sess.close()


def test_fused_adamw_refusals_leave_buffers_untouched():
    dev = torch.device("cuda")
    n = 5000
    gen = torch.Generator(device=dev).manual_seed(3)
    th = (torch.randn(n, generator=gen, device=dev) * 0.02).to(torch.bfloat16)
    t0 = (th.float() + 1e-3).to(torch.bfloat16)
    sim = torch.empty_like(th)
    g = torch.randn(n, generator=gen, device=dev)
    m1 = torch.full((n,), 2.0, device=dev)
    m2 = torch.full((n,), 3.0, device=dev)
    sess = S.SmatSession([th], [t0], [sim], [0.7], [1e-3], seed=9)
    th0 = th.clone()

    def refused(status, **kw):
        args = dict(step=4, g=g, a=m1, b=m2)
        args.update({k: kw.pop(k) for k in list(kw) if k in args})
        with pytest.raises(S.SmatError) as e:
            sess.grad_map_adamw_multi(args["step"], [args["g"]], [args["a"]], [args["b"]], **dict(HP, **kw))
        assert e.value.status == status, e.value.detail

    refused("SMAT_ERR_STATE")  # no forward yet
    sess.simulate_multi(4)
    refused("SMAT_ERR_STATE", step=3)  # not the last forward's step
    sess.swap()
    refused("SMAT_ERR_STATE")  # the simulated storage is active
    sess.swap()
    refused("SMAT_ERR_INVALID_ARG", beta1=1.0)
    refused("SMAT_ERR_INVALID_ARG", beta2=-0.1)
    refused("SMAT_ERR_INVALID_ARG", eps=0.0)
    refused("SMAT_ERR_INVALID_ARG", lr=float("nan"))
    refused("SMAT_ERR_INVALID_ARG", weight_decay=-1.0)
    refused("SMAT_ERR_INVALID_ARG", adam_step=0)
    refused("SMAT_ERR_INVALID_ARG", b=m1)  # m2 aliases m1
    refused("SMAT_ERR_INVALID_ARG", g=m1)  # g_sim aliases m1
    torch.cuda.synchronize()
    assert torch.equal(th, th0) and torch.all(m1 == 2.0) and torch.all(m2 == 3.0)
    sess.grad_map_adamw_multi(4, [g], [m1], [m2], **HP)
    torch.cuda.synchronize()
    assert not torch.equal(th, th0)
    assert sess.poll_errors() == 0
    sess.close()


def _same_f32(got, ref):
    """Bit-equal, except that any NaN matches any NaN (payloads differ between
    the CPU and the GPU)."""
    g, r = got.view(np.uint32), ref.view(np.uint32)
    nan = np.isnan(got.view(np.float32)) & np.isnan(ref.view(np.float32))
    return bool(np.all((g == r) | nan))


@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_fused_adamw_special_moments(dtype):
    """Moments of both zero signs (the shortcut around sqrt and the divides),
    subnormal, huge and non-finite moments and gradients, on both the vector
    and the element path."""
    dev = torch.device("cuda")
    n = 4096 + 13
    rng = np.random.default_rng(11)
    v1 = np.array([0.0, -0.0, 1e-40, -1e-40, 1e-3, -2.5e-7, 3e38, np.inf, -np.inf, np.nan], np.float32)
    v2 = np.array([0.0, -0.0, 1e-42, 1e-30, 1e-6, 3e38, np.inf, np.nan, 2.0], np.float32)
    h1 = v1[rng.integers(0, len(v1), n)]
    h2 = v2[rng.integers(0, len(v2), n)]
    gv = rng.standard_normal(n).astype(np.float32)
    gv[rng.integers(0, n, 64)] = np.array([0.0, -0.0, 1e-42, 3e38, np.inf, np.nan, -np.inf, 1e20], np.float32)[
        rng.integers(0, 8, 64)]
    tdt = torch.float32 if dtype == O.F32 else torch.bfloat16
    th = (torch.randn(n, device=dev) * 0.02).to(tdt)
    t0 = (th.float() + 1e-3).to(tdt)
    sim = torch.empty_like(th)
    g = torch.from_numpy(gv).to(dev)
    m1 = torch.from_numpy(h1.copy()).to(dev)
    m2 = torch.from_numpy(h2.copy()).to(dev)
    hth = to_host(th)
    sess = S.SmatSession([th], [t0], [sim], [0.6], [1e-3], seed=5, alpha_min=0.2, alpha_max=1.0,
                         alpha_mode=S.SMAT_ALPHA_PER_TENSOR, noise=S.SMAT_NOISE_UNIFORM)
    for t_opt, step in enumerate((0, 1), start=1):
        sess.simulate_multi(step)
        sess.grad_map_adamw_multi(step, [g], [m1], [m2], adam_step=t_opt, **HP)
        torch.cuda.synchronize()
        cfg = O.config(seed=5, step=step, alpha_mode=O.ALPHA_PER_TENSOR, noise=O.NOISE_UNIFORM, alpha_min=0.2,
                       alpha_max=1.0)
        t = O.tensor(0, n, dtype, keep_prob=0.6, sigma=1e-3)
        hth, h1, h2 = O.gradmap_adamw(cfg, t, gv, hth, h1, h2, adam_step=t_opt, **HP)
        assert _same_f32(to_host(m1), h1) and _same_f32(to_host(m2), h2), f"step {step} moments"
        got = to_host(th)
        if dtype == O.F32:
            assert _same_f32(got, hth), f"step {step} theta"
        else:
            ga, ra = O.bf16_to_f32(got), O.bf16_to_f32(hth)
            assert np.all((got == hth) | (np.isnan(ga) & np.isnan(ra))), f"step {step} theta"
    sess.close()
