"""Periodic SMAT training (Sec. 4.3): t - 1 ordinary steps and one
simulated-loss step per period, storage switching around the simulated
step's forward and backward pass, the optimizer on the original storage.
The schedule's trajectory equals a hand-written loop whose simulated
weights and mapped gradients come from the oracle, and the in-place mode
(theta0 refilled from pinned host memory) follows the same trajectory as
the two-buffer mode."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300.schedule import PeriodicSmat

from _parity import to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


def _model(dtype, seed=0):
    torch.manual_seed(seed)
    m = torch.nn.Sequential(torch.nn.Linear(64, 256), torch.nn.GELU(), torch.nn.Linear(256, 64), torch.nn.GELU(),
                            torch.nn.Linear(64, 8))
    return m.to(device="cuda", dtype=dtype)


def _batch(step, dtype):
    g = torch.Generator(device="cuda").manual_seed(1000 + step)
    return torch.randn(32, 64, device="cuda", generator=g, dtype=dtype)


def _drift(params):
    with torch.no_grad():
        for k, p in enumerate(params):
            g = torch.Generator(device="cuda").manual_seed(77 + k)
            p.add_(torch.randn(p.shape, device="cuda", generator=g, dtype=p.dtype) * 1e-2)


def test_schedule_matches_oracle_driven_loop():
    period, steps, lr = 4, 10, 0.05
    keeps = [0.5, 1.0, 0.7, 1.0, 0.9, 1.0]
    sigmas = [2e-3] * 6
    cfg_kw = dict(seed=5, alpha_min=0.3, alpha_max=1.0, alpha_mode=S.SMAT_ALPHA_PER_TENSOR,
                  noise=S.SMAT_NOISE_UNIFORM)
    # the schedule
    ma = _model(torch.float32)
    pa = list(ma.parameters())
    theta0 = [p.detach().clone() for p in pa]
    _drift(pa)
    sched = PeriodicSmat(pa, keeps, sigmas, theta0=theta0, period=period, **cfg_kw)
    opt_a = torch.optim.SGD(pa, lr=lr)
    # the hand-written loop with the oracle's theta~ and mapped gradient
    mb = _model(torch.float32)
    pb = list(mb.parameters())
    _drift(pb)
    opt_b = torch.optim.SGD(pb, lr=lr)
    for step in range(steps):
        x = _batch(step, torch.float32)
        sched.before_forward(step)
        ma(x).square().mean().backward()
        sched.after_backward(step)
        opt_a.step()
        opt_a.zero_grad()

        smat = step % period == period - 1
        if smat:
            cfg = O.config(seed=5, step=step, alpha_mode=O.ALPHA_PER_TENSOR, noise=O.NOISE_UNIFORM, alpha_min=0.3)
            saved = [p.detach().clone() for p in pb]
            with torch.no_grad():
                for k, p in enumerate(pb):
                    t = O.tensor(k, p.numel(), O.F32, keep_prob=keeps[k], sigma=sigmas[k])
                    sim = O.simulate(cfg, t, to_host(p).ravel(), to_host(theta0[k]).ravel())
                    p.copy_(torch.from_numpy(sim.view(np.float32).reshape(p.shape)))
        mb(x).square().mean().backward()
        if smat:
            with torch.no_grad():
                for k, p in enumerate(pb):
                    t = O.tensor(k, p.numel(), O.F32, keep_prob=keeps[k], sigma=sigmas[k])
                    g = O.gradmap(cfg, t, to_host(p.grad).ravel())
                    p.grad.copy_(torch.from_numpy(g.view(np.float32).reshape(p.shape)))
                    p.copy_(saved[k])
        opt_b.step()
        opt_b.zero_grad()
        torch.cuda.synchronize()
        for a, b in zip(pa, pb):
            assert torch.equal(a.view(torch.int32), b.view(torch.int32)), f"step {step}"
    sched.close()


def test_inplace_schedule_follows_the_two_buffer_trajectory():
    period, steps = 4, 9
    kw = dict(seed=11, alpha_min=0.3, alpha_max=1.0, alpha_mode=S.SMAT_ALPHA_PER_TENSOR,
              noise=S.SMAT_NOISE_GAUSSIAN)
    models, scheds, opts = [], [], []
    for mode in ("device", "host"):
        m = _model(torch.bfloat16)
        ps = list(m.parameters())
        theta0 = [p.detach().clone() for p in ps]
        _drift(ps)
        keeps = [0.7 if p.dim() == 2 else 1.0 for p in ps]
        sig = [1e-3] * len(ps)
        rel = [0.1 if p.dim() == 2 else 0.0 for p in ps]
        if mode == "device":
            s = PeriodicSmat(ps, keeps, sig, rel, theta0=theta0, period=period, **kw)
        else:
            s = PeriodicSmat(ps, keeps, sig, rel, host_theta0=[t.cpu().pin_memory() for t in theta0], period=period,
                             **kw)
        models.append(m)
        scheds.append(s)
        opts.append(torch.optim.AdamW(ps, lr=1e-3, weight_decay=1e-3))
    for step in range(steps):
        x = _batch(step, torch.bfloat16)
        for m, s, o in zip(models, scheds, opts):
            s.before_forward(step)
            m(x).float().square().mean().backward()
            s.after_backward(step)
            o.step()
            o.zero_grad()
        torch.cuda.synchronize()
        for a, b in zip(models[0].parameters(), models[1].parameters()):
            assert torch.equal(a.view(torch.int16), b.view(torch.int16)), f"step {step}"
    assert scheds[1].session.poll_errors() == 0
    for s in scheds:
        s.close()


def test_schedule_argument_checks():
    m = _model(torch.float32)
    ps = list(m.parameters())
    t0 = [p.detach().clone() for p in ps]
    with pytest.raises(ValueError):
        PeriodicSmat(ps, [1.0] * len(ps), [0.0] * len(ps))
    with pytest.raises(ValueError):
        PeriodicSmat(ps, [1.0] * len(ps), [0.0] * len(ps), theta0=t0, host_theta0=[t.cpu() for t in t0])
    with pytest.raises(ValueError):
        PeriodicSmat(ps, [1.0] * len(ps), [0.0] * len(ps), host_theta0=[t.cpu() for t in t0])  # not pinned
    s = PeriodicSmat(ps, [1.0] * len(ps), [0.0] * len(ps), theta0=t0, period=4)
    assert [s.is_smat_step(i) for i in range(8)] == [False, False, False, True] * 2
    s.close()
