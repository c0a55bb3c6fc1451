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
