"""In-place mode (Sec. 4.3): a tensor passed with sim == theta0 has one extra
buffer, holding theta0 until the forward overwrites it with theta~; theta0 is
copied back from host memory before the next forward. theta0 may also stay in
pinned host memory and be read there by the kernels (App. E keeps it on the
CPU). Both forwards and their gradient maps are compared element by element
with the CPU oracle (tolerances of tests/_parity.py) and with the two-buffer
mode; the state rules are enforced."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300 import workloads as W

from _parity import compare, f32_of, orc_config, orc_tensor, session_for, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


def _list(dtype, noise, rel):
    sizes = [70_001, 262_144 * 2 + 48, 17, 4096, 300_003]
    keeps = [0.7, 0.5 + 2**-10, 0.9, 1.0, 0.3]
    specs = [W.TensorSpec(f"t{i}", (n,), "linear", keeps[i], 0.0 if rel and i % 2 == 0 else 2e-3,
                          0.1 if rel and i % 2 == 0 else 0.0) for i, n in enumerate(sizes)]
    return W.Workload(f"inplace_{dtype}_{noise}_{rel}", specs, dtype, dtype, 0.3, 1.0, O.ALPHA_PER_TENSOR, noise,
                      0.02, 1e-3, seed=0x1A9_1ACE)


def _bits(t):
    return t.view(torch.int16 if t.dtype == torch.bfloat16 else torch.int32)


def _check_against_oracle(w, hth, ht0, sims, step, what, g_sim=None, g_out=None):
    """Every element of each tensor's theta~ (and mapped gradient) against the
    oracle at this step; sigma_rel tensors take the float tolerance since
    their sigma_t is a reduction whose rounding order differs."""
    cfg = orc_config(w, step)
    for k in range(len(w.tensors)):
        t = orc_tensor(w, k)
        ref = O.simulate(cfg, t, hth[k], ht0[k])
        mode = O.NOISE_GAUSSIAN if w.tensors[k].sigma_rel > 0 else w.noise
        compare(to_host(sims[k]), ref.view(np.uint16 if w.dtype == O.BF16 else np.uint32), w.dtype, mode,
                f32_of(hth[k]), f32_of(ht0[k]), what=f"{what} step {step} tensor {k}")
        if g_sim is not None:
            gv = np.uint16 if w.gdtype == O.BF16 else np.uint32
            gref = O.gradmap(cfg, t, to_host(g_sim[k]), gdtype=w.gdtype)
            assert np.array_equal(to_host(g_out[k]).view(gv), gref.view(gv)), f"{what} step {step} tensor {k} gradmap"


@pytest.mark.parametrize("chunk_log2", [12, 18])
@pytest.mark.parametrize("rel", [False, True])
@pytest.mark.parametrize("noise", [O.NOISE_UNIFORM, O.NOISE_GAUSSIAN, O.NOISE_LAPLACE])
@pytest.mark.parametrize("dtype", [O.BF16, O.F32])
def test_inplace_forward_matches_oracle_and_two_buffer_forward(dtype, noise, rel, chunk_log2):
    w = _list(dtype, noise, rel)
    dev = torch.device("cuda")
    th, t0, sim, gs, go = W.generate(w, device=dev)
    flags = S.SMAT_FLAG_CHUNK_LOG2(chunk_log2)
    ref = session_for(w, th, t0, sim, flags=flags)
    host_t0 = [x.cpu().pin_memory() for x in t0]
    buf = [x.clone() for x in t0]  # the single extra buffer: theta0, then theta~
    ip = session_for(w, th, buf, buf, flags=flags)
    hth = [to_host(x) for x in th]
    ht0 = [to_host(x) for x in t0]
    for step in (0, 5, 6):
        ref.simulate_multi(step)
        ip.simulate_multi(step)
        torch.cuda.synchronize()
        # gradient map: unaffected by the mode
        go2 = [torch.empty_like(g) for g in gs]
        for s, o in ((ref, go), (ip, go2)):
            s.swap()
            s.grad_map_multi(step, gs, o)
            s.swap()
        torch.cuda.synchronize()
        _check_against_oracle(w, hth, ht0, buf, step, "in-place", gs, go2)
        for a, b in zip(sim, buf):
            assert torch.equal(_bits(a), _bits(b)), f"step {step}"
        for a, b in zip(go, go2):
            assert torch.equal(_bits(a), _bits(b))
        ip.refill_theta0(host_t0)
        torch.cuda.synchronize()
        for a, b in zip(buf, t0):
            assert torch.equal(_bits(a), _bits(b))
    assert ref.poll_errors() == 0 and ip.poll_errors() == 0


def test_inplace_state_rules():
    w = _list(O.BF16, O.NOISE_GAUSSIAN, True)
    dev = torch.device("cuda")
    th, t0, sim, gs, go = W.generate(w, device=dev)
    buf = [x.clone() for x in t0]
    host_t0 = [x.cpu().pin_memory() for x in t0]
    ip = session_for(w, th, buf, buf)
    ip.simulate_multi(0)
    with pytest.raises(S.SmatError) as e:
        ip.simulate_multi(1)  # theta0 not refilled
    assert e.value.status == "SMAT_ERR_STATE"
    with pytest.raises(S.SmatError) as e:
        ip.tensor_scalars(1)  # statistics need theta0
    assert e.value.status == "SMAT_ERR_STATE"
    ip.swap()
    with pytest.raises(S.SmatError) as e:
        ip.refill_theta0(host_t0)  # the model reads these buffers now
    assert e.value.status == "SMAT_ERR_STATE"
    with pytest.raises(S.SmatError) as e:
        ip.mark_theta0_resident()
    assert e.value.status == "SMAT_ERR_STATE"
    ip.swap()
    with pytest.raises(ValueError):
        ip.refill_theta0(host_t0[:-1])
    ip.refill_theta0(host_t0)
    ip.simulate_multi(1)
    # a caller-side copy on its own stream, then the mark
    for b, h in zip(buf, host_t0):
        b.copy_(h, non_blocking=True)
    ip.mark_theta0_resident()
    ip.simulate_multi(2)
    torch.cuda.synchronize()
    assert ip.poll_errors() == 0


@pytest.mark.parametrize("rel", [False, True])
@pytest.mark.parametrize("noise", [O.NOISE_UNIFORM, O.NOISE_GAUSSIAN, O.NOISE_LAPLACE])
@pytest.mark.parametrize("dtype", [O.BF16, O.F32])
def test_theta0_read_from_pinned_host_memory(dtype, noise, rel):
    """theta0 may stay in pinned host memory (Sec. 4.3 keeps it there): the
    kernels read it directly, with the same results as from HBM."""
    w = _list(dtype, noise, rel)
    dev = torch.device("cuda")
    th, t0, sim, gs, go = W.generate(w, device=dev)
    ref = session_for(w, th, t0, sim)
    host_t0 = [x.cpu().pin_memory() for x in t0]
    sim2 = [torch.empty_like(x) for x in sim]
    hs = session_for(w, th, host_t0, sim2)
    hth = [to_host(x) for x in th]
    ht0 = [to_host(x) for x in t0]
    for step in (0, 4):
        ref.simulate_multi(step)
        hs.simulate_multi(step)
        torch.cuda.synchronize()
        _check_against_oracle(w, hth, ht0, sim2, step, "host theta0")
        for a, b in zip(sim, sim2):
            assert torch.equal(_bits(a), _bits(b)), f"step {step}"
    assert hs.poll_errors() == 0
