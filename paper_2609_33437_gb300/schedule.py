"""Periodic SMAT training (Sec. 4.3, "Periodic scheduling" and "Parameter
storage switching").

Each period of `period` steps (t = 4 in the paper) has t - 1 ordinary
expert-loss steps and one simulated-loss step, matching lambda = 1/t of the
SMAT objective; every step runs one forward and one backward pass. On the
simulated-loss step the parameters' storage is switched to theta~ (computed
by the library's forward, Eq. smat-state) for the forward and backward pass,
the gradient is mapped in place (g = alpha m (.) g~, Eq. smat-gradient) and
the original storage is restored before the optimizer update, which
therefore updates theta with the mapped gradient.

theta0 is kept either in its own device buffers (two buffers per parameter
besides theta: theta0 and theta~), or, as in the paper, in pinned host
memory with one device buffer per parameter (in-place mode): the buffer is
refilled with theta0 on a side stream right after each simulated-loss step,
so the copy overlaps the following ordinary steps, and the next
simulated-loss step waits for it.

Usage (a training loop with any optimizer):

    sched = PeriodicSmat(params, keep_probs, sigmas, theta0=..., period=4, ...)
    for step in range(n):
        sched.before_forward(step)
        loss_fn(model, batch).backward()
        sched.after_backward(step)
        opt.step(); opt.zero_grad()

or, with torch.optim.AdamW on fp32 parameters, the gradient map folded into
the optimizer's read of the gradient on simulated-loss steps:

        sched.before_forward(step)
        loss_fn(model, batch).backward()
        sched.optimizer_step(step, opt); opt.zero_grad()
"""

from typing import List, Optional, Sequence

import torch

from .smat import SmatSession


class PeriodicSmat:
    """Periodic simulated-merge schedule over a list of parameters.

    params: the trainable parameters (theta), contiguous CUDA tensors.
    keep_probs, sigmas, sigma_rels: per-parameter p_keep (1 outside the
      masked set), Perturb RMS, relative Perturb RMS (see SmatSession).
    theta0: device tensors of the shared initialisation (two-buffer mode), or
    host_theta0: pinned CPU tensors of it (in-place mode); exactly one.
    period: t; step s is a simulated-loss step when s % t == t - 1.
    Remaining keyword arguments (seed, alpha_min, alpha_max, alpha_mode,
    noise, philox_rounds, flags) go to SmatSession.
    """

    def __init__(self, params: List[torch.nn.Parameter], keep_probs: Sequence[float], sigmas: Sequence[float],
                 sigma_rels: Optional[Sequence[float]] = None, theta0: Optional[Sequence[torch.Tensor]] = None,
                 host_theta0: Optional[Sequence[torch.Tensor]] = None, period: int = 4, **cfg):
        if (theta0 is None) == (host_theta0 is None):
            raise ValueError("give exactly one of theta0 (device) and host_theta0 (pinned host)")
        if period < 1:
            raise ValueError("period must be >= 1")
        self.params = list(params)
        self.period = int(period)
        self.theta = [p.data for p in self.params]
        self.inplace = host_theta0 is not None
        if self.inplace:
            self.host_theta0 = list(host_theta0)
            for h, p in zip(self.host_theta0, self.params):
                if h.is_cuda or not h.is_pinned() or h.numel() != p.numel() or h.dtype != p.dtype:
                    raise ValueError("host_theta0: pinned CPU tensors shaped like the parameters")
            # the single extra buffer per parameter: theta0, then theta~ on simulated steps
            self.sims = [torch.empty_like(p.data) for p in self.params]
            for s, h in zip(self.sims, self.host_theta0):
                s.copy_(h)
            theta0_dev = self.sims
        else:
            self.sims = [torch.empty_like(p.data) for p in self.params]
            theta0_dev = list(theta0)
        self.session = SmatSession(self.theta, theta0_dev, self.sims, keep_probs, sigmas, sigma_rels, **cfg)
        self.copy_stream = torch.cuda.Stream(device=self.params[0].device) if self.inplace else None
        self.refilled = None  # event recorded after the last refill

    def is_smat_step(self, step: int) -> bool:
        return step % self.period == self.period - 1

    def _swap(self) -> int:
        active = self.session.swap()
        src = self.sims if active == 1 else self.theta
        for p, t in zip(self.params, src):
            p.data = t
        return active

    def before_forward(self, step: int):
        """On a simulated-loss step: theta~ for this step, then switch the
        parameters' storage to it."""
        if not self.is_smat_step(step):
            return
        if self.refilled is not None:
            torch.cuda.current_stream().wait_event(self.refilled)
        self.session.simulate_multi(step)
        self._swap()

    def after_backward(self, step: int):
        """On a simulated-loss step: map the gradients in place, restore the
        original storage (the optimizer updates theta), and in in-place mode
        start refilling theta0 on the side stream."""
        if not self.is_smat_step(step):
            return
        self.session.grad_map_multi(step, [p.grad for p in self.params], [p.grad for p in self.params])
        self._swap()
        self._refill_after()

    def _fusable(self, opt) -> bool:
        """The fused path takes one AdamW parameter group holding exactly this
        schedule's fp32 parameters, with a plain (non-capturable, non-fused,
        non-amsgrad, non-maximising) update and one step count for all."""
        if type(opt) is not torch.optim.AdamW or len(opt.param_groups) != 1:
            return False
        g = opt.param_groups[0]
        if [id(p) for p in g["params"]] != [id(p) for p in self.params]:
            return False
        if g.get("amsgrad") or g.get("maximize") or g.get("capturable") or g.get("fused") or g.get("differentiable"):
            return False
        if torch.is_tensor(g["lr"]) or any(p.dtype != torch.float32 for p in self.params):
            return False
        steps = {float(opt.state[p]["step"]) if "step" in opt.state[p] else 0.0 for p in self.params}
        return len(steps) == 1

    def optimizer_step(self, step: int, opt):
        """After the backward pass: on an ordinary step, opt.step(). On a
        simulated-loss step with an AdamW the fused path accepts (see
        _fusable), the storage is switched back and the gradient map and the
        AdamW update run as one pass (smat_grad_map_adamw_multi) on the
        optimizer's own moments; the mapped gradient is not written (p.grad
        keeps g~). Otherwise after_backward, then opt.step()."""
        if not self.is_smat_step(step):
            opt.step()
            return
        if not self._fusable(opt):
            self.after_backward(step)
            opt.step()
            return
        g = opt.param_groups[0]
        for p in self.params:
            st = opt.state[p]
            if "step" not in st:  # the optimizer's own lazy initialisation, done here first
                st["step"] = torch.tensor(0.0, dtype=torch.float32)
                st["exp_avg"] = torch.zeros_like(p, memory_format=torch.preserve_format)
                st["exp_avg_sq"] = torch.zeros_like(p, memory_format=torch.preserve_format)
        t = int(float(opt.state[self.params[0]]["step"])) + 1
        grads = [p.grad for p in self.params]
        self._swap()
        beta1, beta2 = g["betas"]
        self.session.grad_map_adamw_multi(step, grads, [opt.state[p]["exp_avg"] for p in self.params],
                                          [opt.state[p]["exp_avg_sq"] for p in self.params], lr=g["lr"],
                                          beta1=beta1, beta2=beta2, eps=g["eps"],
                                          weight_decay=g["weight_decay"], adam_step=t)
        for p in self.params:
            opt.state[p]["step"] += 1
        self._refill_after()

    def _refill_after(self):
        if self.inplace:
            # the copy may start once this stream is past the gradient map
            ready = torch.cuda.Event()
            ready.record()
            self.copy_stream.wait_event(ready)
            self.session.refill_theta0(self.host_theta0, stream=self.copy_stream)
            self.refilled = torch.cuda.Event()
            self.refilled.record(self.copy_stream)
            for s in self.sims:
                s.record_stream(self.copy_stream)

    def close(self):
        self.session.close()
