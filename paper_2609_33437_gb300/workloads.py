"""Synthetic workloads: tensor lists shaped like the paper's backbones and
seeded draws of theta0, theta = theta0 + delta and the incoming gradient.

This module holds no arithmetic of the simulated-merge transform; it only
describes parameter lists and draws inputs. Both the CUDA path's tests and
the oracle's tests take their inputs from here.

Lists (Sec. 5.1 backbones, shapes as stated for the synthetic stand-ins):
  tiny_flat   one fp32 tensor of 1,048,576 elements
  dec_0p5b    24-layer decoder, hidden 896, 14 heads (k/v 128 wide),
              MLP 4864, RMSNorm, embedding 151936 x 896 (218 tensors)
  llama_7b    32-layer decoder, hidden 4096, MLP 11008, RMSNorm,
              embedding and LM head 32000 x 4096 (291 tensors)
  vl_7b       CLIP ViT-L/14 tower + 2-layer projector + llama_7b (590 tensors)
  flat_sweep  one flat tensor, 2^16 .. 2^32 elements

Mask set (Sec. 4.1, "linear weights in Transformer attention and MLP blocks"):
tensors of kind 'linear' take the configured keep probability; embeddings,
LM head, norms, biases, patch/position/class embeddings and the projector
keep every coordinate (p_keep = 1) but are still perturbed.
"""

from dataclasses import dataclass, field
from typing import List, Optional

import torch

F32, BF16 = 0, 1


@dataclass
class TensorSpec:
    name: str
    shape: tuple
    kind: str          # 'linear' (in the mask set) or 'other'
    keep_prob: float
    sigma: float = 0.0
    sigma_rel: float = 0.0

    @property
    def numel(self) -> int:
        n = 1
        for s in self.shape:
            n *= s
        return n


@dataclass
class Workload:
    name: str
    tensors: List[TensorSpec]
    dtype: int                 # parameter storage dtype
    gdtype: int                # gradient dtype
    alpha_min: float
    alpha_max: float
    alpha_mode: int            # 0 global, 1 per tensor, 2 per element
    noise: int                 # 0 uniform, 1 Gaussian
    theta0_std: float
    delta_std: float
    seed: int = 0
    data_seed: int = 1234
    notes: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def numel(self) -> int:
        return sum(t.numel for t in self.tensors)

    def param_bytes(self) -> int:
        b = 2 if self.dtype == BF16 else 4
        return b * self.numel

    def grad_bytes(self) -> int:
        b = 2 if self.gdtype == BF16 else 4
        return b * self.numel


def _decoder(layers, hidden, kv_width, mlp, vocab, keep, sigma, sigma_rel, lm_head, prefix=""):
    t = []
    for i in range(layers):
        p = f"{prefix}layers.{i}."
        t.append(TensorSpec(p + "attn.q", (hidden, hidden), "linear", keep, sigma, sigma_rel))
        t.append(TensorSpec(p + "attn.k", (kv_width, hidden), "linear", keep, sigma, sigma_rel))
        t.append(TensorSpec(p + "attn.v", (kv_width, hidden), "linear", keep, sigma, sigma_rel))
        t.append(TensorSpec(p + "attn.o", (hidden, hidden), "linear", keep, sigma, sigma_rel))
        t.append(TensorSpec(p + "mlp.gate", (mlp, hidden), "linear", keep, sigma, sigma_rel))
        t.append(TensorSpec(p + "mlp.up", (mlp, hidden), "linear", keep, sigma, sigma_rel))
        t.append(TensorSpec(p + "mlp.down", (hidden, mlp), "linear", keep, sigma, sigma_rel))
        t.append(TensorSpec(p + "input_norm", (hidden,), "other", 1.0, sigma, sigma_rel))
        t.append(TensorSpec(p + "post_attn_norm", (hidden,), "other", 1.0, sigma, sigma_rel))
    t.insert(0, TensorSpec(prefix + "embed", (vocab, hidden), "other", 1.0, sigma, sigma_rel))
    if lm_head:
        t.append(TensorSpec(prefix + "lm_head", (vocab, hidden), "other", 1.0, sigma, sigma_rel))
    t.append(TensorSpec(prefix + "final_norm", (hidden,), "other", 1.0, sigma, sigma_rel))
    return t


def _vit_l14(keep, sigma):
    w, mlp = 1024, 4096
    t = [TensorSpec("vit.patch_embed", (w, 588), "other", 1.0, sigma),
         TensorSpec("vit.cls", (w,), "other", 1.0, sigma),
         TensorSpec("vit.pos_embed", (257, w), "other", 1.0, sigma),
         TensorSpec("vit.pre_ln.w", (w,), "other", 1.0, sigma),
         TensorSpec("vit.pre_ln.b", (w,), "other", 1.0, sigma)]
    for i in range(24):
        p = f"vit.layers.{i}."
        t += [TensorSpec(p + "ln1.w", (w,), "other", 1.0, sigma),
              TensorSpec(p + "ln1.b", (w,), "other", 1.0, sigma),
              TensorSpec(p + "attn.qkv", (3 * w, w), "linear", keep, sigma),
              TensorSpec(p + "attn.qkv.bias", (3 * w,), "other", 1.0, sigma),
              TensorSpec(p + "attn.out", (w, w), "linear", keep, sigma),
              TensorSpec(p + "attn.out.bias", (w,), "other", 1.0, sigma),
              TensorSpec(p + "ln2.w", (w,), "other", 1.0, sigma),
              TensorSpec(p + "ln2.b", (w,), "other", 1.0, sigma),
              TensorSpec(p + "mlp.fc1", (mlp, w), "linear", keep, sigma),
              TensorSpec(p + "mlp.fc1.bias", (mlp,), "other", 1.0, sigma),
              TensorSpec(p + "mlp.fc2", (w, mlp), "linear", keep, sigma),
              TensorSpec(p + "mlp.fc2.bias", (w,), "other", 1.0, sigma)]
    t += [TensorSpec("vit.post_ln.w", (w,), "other", 1.0, sigma),
          TensorSpec("vit.post_ln.b", (w,), "other", 1.0, sigma)]
    return t


def tiny_flat() -> Workload:
    """One flat fp32 tensor of 2^20 elements: theta0 ~ N(0, 0.02^2),
    delta ~ N(0, 1e-3^2), alpha ~ U[0.3, 1) per tensor, p_keep 0.9,
    Gaussian eps with sigma 1e-4, seed 0, step 0, incoming gradient N(0, 1)."""
    return Workload("tiny_flat_1Mi_f32", [TensorSpec("flat", (1048576,), "linear", 0.9, 1e-4)],
                    F32, F32, 0.3, 1.0, 1, 1, 0.02, 1e-3, data_seed=1235)


def dec_0p5b() -> Workload:
    """0.5B-class decoder in bf16, fp32 gradients: alpha ~ U[0.2, 1) per tensor,
    p_keep 0.5 on attention/MLP linears, sigma 1e-4 (Gaussian),
    theta0 ~ N(0, 0.02^2), delta ~ N(0, 5e-4^2)."""
    t = _decoder(24, 896, 128, 4864, 151936, 0.5, 1e-4, 0.0, lm_head=False)
    return Workload("dec_0p5b_bf16", t, BF16, F32, 0.2, 1.0, 1, 1, 0.02, 5e-4, data_seed=1236)


def llama_7b(noise: int = 1) -> Workload:
    """7B Llama-style decoder in bf16, bf16 gradients: alpha ~ U[0.3, 1) per
    tensor, p_keep 0.7 on linears, sigma_t = 0.1 std(delta_t) per tensor,
    theta0 ~ N(0, 0.02^2), delta ~ N(0, 3e-4^2)."""
    t = _decoder(32, 4096, 4096, 11008, 32000, 0.7, 0.0, 0.1, lm_head=True)
    name = "llama_7b_bf16" + ("" if noise == 1 else "_uniform_noise")
    return Workload(name, t, BF16, BF16, 0.3, 1.0, 1, noise, 0.02, 3e-4, data_seed=1237)


def vl_7b() -> Workload:
    """ViT-L/14 + projector + 7B decoder in bf16, bf16 gradients: p_keep 0.9 on
    vision linears, 0.3 on language linears, 1 elsewhere; sigma 5e-5
    (Gaussian); alpha ~ U[0.3, 1) per tensor."""
    sigma = 5e-5
    t = _vit_l14(0.9, sigma)
    t += [TensorSpec("proj.fc1", (4096, 1024), "other", 1.0, sigma),
          TensorSpec("proj.fc1.bias", (4096,), "other", 1.0, sigma),
          TensorSpec("proj.fc2", (4096, 4096), "other", 1.0, sigma),
          TensorSpec("proj.fc2.bias", (4096,), "other", 1.0, sigma)]
    t += _decoder(32, 4096, 4096, 11008, 32000, 0.3, sigma, 0.0, lm_head=True, prefix="lm.")
    return Workload("vl_7b_bf16", t, BF16, BF16, 0.3, 1.0, 1, 1, 0.02, 3e-4, data_seed=1238)


def flat_sweep(log2n: int, dtype: int, keep: float, alpha_mode: int, sigma: float) -> Workload:
    """One point of the flat-tensor sweep: n = 2^log2n, alpha ~ U[0, 1) per
    tensor (mode 1) or per element (mode 2), delta ~ N(0, 1e-3^2)."""
    t = [TensorSpec("flat", (1 << log2n,), "linear", keep, sigma)]
    return Workload(f"flat_2^{log2n}_{'bf16' if dtype == BF16 else 'f32'}_p{keep}_a{alpha_mode}_s{sigma}",
                    t, dtype, dtype, 0.0, 1.0, alpha_mode, 1, 0.02, 1e-3, data_seed=1239)


WORKLOADS = {"tiny_flat": tiny_flat, "dec_0p5b": dec_0p5b, "llama_7b": llama_7b, "vl_7b": vl_7b}


def scaled(w: Workload, max_numel: int) -> Workload:
    """The same list with every tensor's leading dimension cut so that the
    total stays near max_numel (shapes, kinds and per-tensor settings kept;
    sizes become ragged). For oracle-sized parity cases."""
    tot = w.numel
    if tot <= max_numel:
        return w
    f = max_numel / tot
    out = []
    for t in w.tensors:
        lead = max(1, int(t.shape[0] * f))
        shape = (lead,) + tuple(t.shape[1:])
        if len(shape) > 1 and lead * shape[1] > 3 * max(1, int(t.numel * f)):
            shape = (max(1, int(t.numel * f)),)
        out.append(TensorSpec(t.name, shape, t.kind, t.keep_prob, t.sigma, t.sigma_rel))
    return Workload(w.name + f"_scaled{max_numel}", out, w.dtype, w.gdtype, w.alpha_min, w.alpha_max,
                    w.alpha_mode, w.noise, w.theta0_std, w.delta_std, w.seed, w.data_seed, w.notes)


def torch_dtype(d: int):
    return torch.bfloat16 if d == BF16 else torch.float32


def generate_tensor(w: Workload, k: int, device, gen: Optional[torch.Generator] = None):
    """theta, theta0, g_sim of tensor k: theta0 and delta drawn in fp32, then
    theta0 = cast(theta0_f32), theta = cast(theta0_f32 + delta)."""
    spec = w.tensors[k]
    if gen is None:
        gen = torch.Generator(device=device)
        gen.manual_seed(w.data_seed * 100003 + k)
    n = spec.numel
    dt = torch_dtype(w.dtype)
    t0 = torch.randn(n, generator=gen, device=device, dtype=torch.float32).mul_(w.theta0_std)
    d = torch.randn(n, generator=gen, device=device, dtype=torch.float32).mul_(w.delta_std)
    theta = (t0 + d).to(dt)
    del d
    theta0 = t0.to(dt)
    del t0
    g = torch.randn(n, generator=gen, device=device, dtype=torch.float32).to(torch_dtype(w.gdtype))
    return theta, theta0, g


def generate(w: Workload, device="cpu", with_grad=True):
    """Lists theta, theta0, sim (uninitialised), g_sim, g_out for every tensor."""
    th, t0, sim, gs, go = [], [], [], [], []
    for k in range(len(w.tensors)):
        a, b, g = generate_tensor(w, k, device)
        th.append(a)
        t0.append(b)
        sim.append(torch.empty_like(a))
        if with_grad:
            gs.append(g)
            go.append(torch.empty_like(g))
        else:
            del g
    return th, t0, sim, gs, go
