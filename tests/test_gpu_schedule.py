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


@pytest.mark.parametrize("period,inplace", [(4, False), (1, False), (3, True)])
def test_fused_adamw_schedule_matches_oracle_driven_loop(period, inplace):
    """optimizer_step with torch.optim.AdamW: ordinary steps are the
    optimizer's own; on simulated-loss steps the gradient map and the AdamW
    update run as one pass on the optimizer's moments. The trajectory (theta
    and both moments) equals a loop that runs the same optimizer on ordinary
    steps and, on simulated-loss steps, takes theta~ from the oracle and the
    fused update from the oracle (gradmap_adamw) on the restored theta. With
    period 1 the first step is a simulated-loss one, before the optimizer
    has any state."""
    steps = 8
    keeps = [0.5, 1.0, 0.7, 1.0, 0.9, 1.0]
    sigmas = [2e-3] * 6
    hp = dict(lr=1e-2, betas=(0.9, 0.99), eps=1e-6, weight_decay=0.05)
    cfg_kw = dict(seed=7, alpha_min=0.3, alpha_max=1.0, alpha_mode=S.SMAT_ALPHA_PER_TENSOR,
                  noise=S.SMAT_NOISE_UNIFORM)
    ma = _model(torch.float32)
    pa = list(ma.parameters())
    theta0 = [p.detach().clone() for p in pa]
    _drift(pa)
    if inplace:
        host = [t.detach().cpu().pin_memory() for t in theta0]
        sched = PeriodicSmat(pa, keeps, sigmas, host_theta0=host, period=period, **cfg_kw)
    else:
        sched = PeriodicSmat(pa, keeps, sigmas, theta0=theta0, period=period, **cfg_kw)
    opt_a = torch.optim.AdamW(pa, **hp)
    mb = _model(torch.float32)
    pb = list(mb.parameters())
    _drift(pb)
    opt_b = torch.optim.AdamW(pb, **hp)
    for step in range(steps):
        x = _batch(step, torch.float32)
        sched.before_forward(step)
        ma(x).square().mean().backward()
        sched.optimizer_step(step, opt_a)
        opt_a.zero_grad()

        smat = step % period == period - 1
        if smat:
            cfg = O.config(seed=7, step=step, alpha_mode=O.ALPHA_PER_TENSOR, noise=O.NOISE_UNIFORM, alpha_min=0.3)
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
                    st = opt_b.state[p]
                    if "step" not in st:
                        st["step"] = torch.tensor(0.0)
                        st["exp_avg"] = torch.zeros_like(p)
                        st["exp_avg_sq"] = torch.zeros_like(p)
                    t = O.tensor(k, p.numel(), O.F32, keep_prob=keeps[k], sigma=sigmas[k])
                    th, m1, m2 = O.gradmap_adamw(cfg, t, to_host(p.grad).ravel(), to_host(saved[k]).ravel(),
                                                 to_host(st["exp_avg"]).ravel(), to_host(st["exp_avg_sq"]).ravel(),
                                                 lr=hp["lr"], beta1=hp["betas"][0], beta2=hp["betas"][1],
                                                 eps=hp["eps"], weight_decay=hp["weight_decay"],
                                                 adam_step=int(float(st["step"])) + 1)
                    p.copy_(torch.from_numpy(th.reshape(p.shape)))
                    st["exp_avg"].copy_(torch.from_numpy(m1.reshape(p.shape)))
                    st["exp_avg_sq"].copy_(torch.from_numpy(m2.reshape(p.shape)))
                    st["step"] += 1
        else:
            opt_b.step()
        opt_b.zero_grad()
        torch.cuda.synchronize()
        for a, b in zip(pa, pb):
            assert torch.equal(a.view(torch.int32), b.view(torch.int32)), f"step {step} theta"
            sa, sb = opt_a.state[a], opt_b.state[b]
            assert torch.equal(sa["exp_avg"].view(torch.int32), sb["exp_avg"].view(torch.int32)), f"step {step} m1"
            assert torch.equal(sa["exp_avg_sq"].view(torch.int32), sb["exp_avg_sq"].view(torch.int32)), f"step {step}"
            assert float(sa["step"]) == float(sb["step"]) == step + 1
    sched.close()


def test_optimizer_step_falls_back_for_other_optimizers():
    """SGD (or an AdamW the fused path does not take, e.g. with amsgrad) goes
    through after_backward and the optimizer's own step: the same trajectory
    as the two-call loop."""
    keeps, sigmas = [0.5, 1.0, 0.7, 1.0, 0.9, 1.0], [2e-3] * 6
    kw = dict(seed=3, alpha_min=0.3, alpha_max=1.0, alpha_mode=S.SMAT_ALPHA_PER_TENSOR, noise=S.SMAT_NOISE_UNIFORM)
    runs = []
    for mode in ("two-call", "optimizer_step"):
        for make in (lambda ps: torch.optim.SGD(ps, lr=0.05), lambda ps: torch.optim.AdamW(ps, lr=1e-2, amsgrad=True)):
            m = _model(torch.float32)
            ps = list(m.parameters())
            t0 = [p.detach().clone() for p in ps]
            _drift(ps)
            sched = PeriodicSmat(ps, keeps, sigmas, theta0=t0, period=2, **kw)
            opt = make(ps)
            for step in range(5):
                sched.before_forward(step)
                m(_batch(step, torch.float32)).square().mean().backward()
                if mode == "two-call":
                    sched.after_backward(step)
                    opt.step()
                else:
                    sched.optimizer_step(step, opt)
                opt.zero_grad()
            torch.cuda.synchronize()
            runs.append([p.detach().clone() for p in ps])
            sched.close()
    for a, b in zip(runs[:2], runs[2:]):
        for x, y in zip(a, b):
            assert torch.equal(x.view(torch.int32), y.view(torch.int32))


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
