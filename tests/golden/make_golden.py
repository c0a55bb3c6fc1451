"""Write tests/golden/oracle_regression.json: small fixed inputs and the CPU
oracle's outputs on them (calls only oracle/). Rerun only when the stream
specification changes on purpose; the commit that does so names the reason."""
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))
import oracle as O  # noqa: E402


def case(name, cfg, t, th, t0, gs, gdtype):
    sim = O.simulate(cfg, t, th, t0)
    g = O.gradmap(cfg, t, gs, gdtype=gdtype)
    bits = O.mask_bits(cfg, t)
    return {"name": name,
            "config": {f: getattr(cfg, f) for f, _ in O.OrcConfig._fields_},
            "tensor": {f: getattr(t, f) for f, _ in O.OrcTensor._fields_},
            "gdtype": gdtype,
            "theta_bits": np.asarray(th).view(np.uint16 if t.dtype == O.BF16 else np.uint32).tolist(),
            "theta0_bits": np.asarray(t0).view(np.uint16 if t.dtype == O.BF16 else np.uint32).tolist(),
            "gsim_bits": np.asarray(gs).view(np.uint16 if gdtype == O.BF16 else np.uint32).tolist(),
            "sim_bits": np.asarray(sim).view(np.uint16 if t.dtype == O.BF16 else np.uint32).tolist(),
            "g_bits": np.asarray(g).view(np.uint16 if gdtype == O.BF16 else np.uint32).tolist(),
            "mask_words": bits.tolist()}


def main():
    r = np.random.default_rng(20260)
    n = 77
    th = (r.standard_normal(n) * 0.02).astype(np.float32)
    t0 = (th + r.standard_normal(n) * 1e-3).astype(np.float32)
    gs = r.standard_normal(n).astype(np.float32)
    cases = [
        case("f32_uniform_per_tensor", O.config(seed=42, step=3, noise=O.NOISE_UNIFORM, alpha_min=0.2),
             O.tensor(5, n, O.F32, keep_prob=0.5, sigma=2e-3), th, t0, gs, O.F32),
        case("f32_gauss_per_element_offset", O.config(seed=7, step=1, noise=O.NOISE_GAUSSIAN,
                                                      alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=0.0),
             O.tensor(9, n, O.F32, keep_prob=0.9, sigma=1e-4, elem_offset=13), th, t0, gs, O.F32),
        case("bf16_sigma_rel_global", O.config(seed=2**40 + 5, step=2**31, noise=O.NOISE_GAUSSIAN,
                                               alpha_mode=O.ALPHA_GLOBAL, alpha_min=0.3),
             O.tensor(3, n, O.BF16, keep_prob=0.7, sigma_rel=0.1), O.f32_to_bf16(th), O.f32_to_bf16(t0),
             O.f32_to_bf16(gs), O.BF16),
        case("f32_laplace_per_tensor", O.config(seed=11, step=5, noise=O.NOISE_LAPLACE, alpha_min=0.3),
             O.tensor(6, n, O.F32, keep_prob=0.7, sigma=2e-3), th, t0, gs, O.F32),
        case("bf16_gauss_per_element_draw16", O.config(seed=19, step=4, noise=O.NOISE_GAUSSIAN,
                                                       alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=0.1,
                                                       draw_bits=16),
             O.tensor(12, n, O.BF16, keep_prob=0.3, sigma=1e-4, elem_offset=5), O.f32_to_bf16(th),
             O.f32_to_bf16(t0), O.f32_to_bf16(gs), O.BF16),
        case("f32_uniform_per_tensor_draw16", O.config(seed=23, step=0, noise=O.NOISE_UNIFORM, alpha_min=0.4,
                                                       draw_bits=16),
             O.tensor(14, n, O.F32, keep_prob=0.7, sigma=2e-3), th, t0, gs, O.F32),
    ]
    doc = {"about": "CPU-oracle outputs on fixed inputs; regression guard for the oracle "
                    "(written by tests/golden/make_golden.py, oracle/ only)",
           "cases": cases}
    with open(os.path.join(HERE, "oracle_regression.json"), "w") as f:
        json.dump(doc, f)


if __name__ == "__main__":
    main()
