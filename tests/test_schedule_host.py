"""Host logic of the periodic schedule (Sec. 4.3: t - 1 ordinary steps, then
one simulated-loss step), checked on the CPU: the step rule and the argument
checks made before anything reaches the GPU."""

import types

import pytest
import torch

from paper_2609_33437_gb300.schedule import PeriodicSmat


@pytest.mark.parametrize("t", [1, 2, 4, 7])
def test_simulated_step_is_the_last_of_each_period(t):
    fake = types.SimpleNamespace(period=t)
    steps = [s for s in range(5 * t) if PeriodicSmat.is_smat_step(fake, s)]
    assert steps == [k * t + t - 1 for k in range(5)]  # one per period, at its end


def test_argument_checks_before_any_device_work():
    ps = [torch.nn.Parameter(torch.zeros(8))]
    with pytest.raises(ValueError):
        PeriodicSmat(ps, [1.0], [0.0])  # neither theta0 nor host_theta0
    with pytest.raises(ValueError):
        PeriodicSmat(ps, [1.0], [0.0], theta0=[torch.zeros(8)], host_theta0=[torch.zeros(8)])  # both
    with pytest.raises(ValueError):
        PeriodicSmat(ps, [1.0], [0.0], theta0=[torch.zeros(8)], period=0)


def test_fused_adamw_path_selection():
    """optimizer_step takes the fused map + AdamW pass only for one plain
    AdamW group holding exactly the schedule's fp32 parameters with one step
    count; everything else goes through the optimizer's own step."""
    ps = [torch.nn.Parameter(torch.zeros(8)), torch.nn.Parameter(torch.zeros(3))]
    fake = types.SimpleNamespace(params=ps)
    fus = lambda opt: PeriodicSmat._fusable(fake, opt)  # noqa: E731
    assert fus(torch.optim.AdamW(ps, lr=1e-3))
    assert not fus(torch.optim.SGD(ps, lr=1e-3))
    assert not fus(torch.optim.Adam(ps, lr=1e-3))  # coupled weight decay: not this update
    assert not fus(torch.optim.AdamW(ps, lr=1e-3, amsgrad=True))
    assert not fus(torch.optim.AdamW(ps, lr=1e-3, maximize=True))
    assert not fus(torch.optim.AdamW(ps, lr=torch.tensor(1e-3)))
    assert not fus(torch.optim.AdamW([{"params": ps[:1]}, {"params": ps[1:]}], lr=1e-3))  # two groups
    assert not fus(torch.optim.AdamW(ps[::-1], lr=1e-3))  # another order than the schedule's tensors
    assert not fus(torch.optim.AdamW(ps[:1], lr=1e-3))
    bf = [torch.nn.Parameter(torch.zeros(8, dtype=torch.bfloat16))]
    assert not PeriodicSmat._fusable(types.SimpleNamespace(params=bf), torch.optim.AdamW(bf, lr=1e-3))
    opt = torch.optim.AdamW(ps, lr=1e-3)
    opt.state[ps[0]]["step"] = torch.tensor(3.0)
    opt.state[ps[1]]["step"] = torch.tensor(2.0)
    assert not fus(opt)  # step counts differ
    opt.state[ps[1]]["step"] = torch.tensor(3.0)
    assert fus(opt)
