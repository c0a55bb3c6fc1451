"""Pins of the CPU oracle against facts fixed outside it.

Each test checks the oracle against the paper's equations, a closed form, a
statistical law, an independent library routine or brute force. None of them
retypes the oracle's own formula. Chosen so that a plausible slip (a dropped
term, a swapped theta/theta0, a wrong sign, a wrong stream index or word) fails
at least one test.
"""

import json
import math
import os
import subprocess
import sys

import numpy as np
import pytest
import torch
from scipy import stats

import oracle as O

HERE = os.path.dirname(os.path.abspath(__file__))


def rng(seed):
    return np.random.default_rng(seed)


def f32(x):
    return np.asarray(x, np.float32)


# ----------------------------------------------------------------- Philox ---

def _triton_philox(ctrs, seeds, rounds):
    pytest.importorskip("triton")
    req = json.dumps({"ctr": [[int(v) for v in c] for c in ctrs],
                      "seed": [int(s) for s in seeds], "rounds": rounds})
    p = subprocess.run([sys.executable, os.path.join(HERE, "_triton_philox.py")], input=req,
                       capture_output=True, text=True, timeout=600)
    if p.returncode != 0:
        pytest.skip("triton interpreter unavailable: " + p.stderr[-300:])
    return np.array(json.loads(p.stdout), dtype=np.uint64).astype(np.uint32)


@pytest.mark.parametrize("rounds", [10, 7])
def test_philox_block_matches_triton_library(rounds):
    """Philox-4x32-R block (Salmon et al. SC'11) against Triton's Philox,
    including counter words and keys with all bits set."""
    r = rng(1)
    ctrs = r.integers(0, 2**32, size=(48, 4), dtype=np.uint64)
    ctrs[0] = 0
    ctrs[1] = 2**32 - 1
    seeds = r.integers(0, 2**63, size=48, dtype=np.uint64) * 2 + r.integers(0, 2, size=48, dtype=np.uint64)
    seeds[0] = 0
    seeds[1] = 2**64 - 1
    ref = _triton_philox(ctrs, seeds, rounds)
    for k in range(len(ctrs)):
        s = int(seeds[k])
        ours = O.philox(ctrs[k], [s & 0xFFFFFFFF, s >> 32], rounds)
        assert np.array_equal(ours, ref[k]), (k, ours, ref[k])


def test_stream_counter_layout_matches_triton_library():
    """W(stream, tid, j)[w] is word w of the Philox block at counter
    (j lo, j hi, stream << 28 | tid, step) under key (seed lo, seed hi)."""
    r = rng(2)
    seed, step = 0x0123456789ABCDEF, 77
    cfg = O.config(seed=seed, step=step)
    cases = []
    for _ in range(24):
        stream = int(r.integers(0, 5))
        tid = int(r.integers(0, 0x0FFFFFFF))
        j = int(r.integers(0, 2**40))
        cases.append((stream, tid, j))
    ref = _triton_philox([[j & 0xFFFFFFFF, j >> 32, (s << 28) | t, step] for s, t, j in cases],
                         [seed] * len(cases), 10)
    for k, (s, t, j) in enumerate(cases):
        got = O.stream_words(cfg, s, t, [j] * 4, [0, 1, 2, 3])
        assert np.array_equal(got, ref[k])


def test_philox_avalanche():
    """A one-bit counter change flips about half the output bits (a property of
    the published block function; catches a dropped round or mixing term)."""
    r = rng(3)
    flips = []
    for _ in range(400):
        c = r.integers(0, 2**32, size=4, dtype=np.uint64).astype(np.uint32)
        k = r.integers(0, 2**32, size=2, dtype=np.uint64).astype(np.uint32)
        w = int(r.integers(0, 4))
        b = int(r.integers(0, 32))
        c2 = c.copy()
        c2[w] ^= np.uint32(1 << b)
        a1, a2 = O.philox(c, k), O.philox(c2, k)
        flips.append(sum(bin(int(x ^ y)).count("1") for x, y in zip(a1, a2)))
    m = np.mean(flips)
    assert abs(m - 64.0) < 5 * 4.0 / math.sqrt(400) * 1.5, m


# ------------------------------------------------------------------- bf16 ---

def test_bf16_rounding_matches_torch():
    """Storage rounding = round-to-nearest-even, as torch's CPU float->bfloat16."""
    r = rng(4)
    x = np.concatenate([
        r.standard_normal(20000).astype(np.float32) * np.float32(0.02),
        (r.integers(0, 2**32, size=20000, dtype=np.uint64).astype(np.uint32)).view(np.float32),
        f32([0.0, -0.0, 1.0, -1.0, np.inf, -np.inf, 3.4028235e38, -3.4028235e38, 1e-45, -1e-45,
             1.1754942e-38, 1.00390625, 1.01171875, 1.0078125 + 2**-24]),
    ])
    # exact ties: low 16 bits = 0x8000
    ties = (r.integers(0, 2**16, size=2000, dtype=np.uint64).astype(np.uint32) << 16) | np.uint32(0x8000)
    x = np.concatenate([x, ties.view(np.float32)])
    ours = O.f32_to_bf16(x)
    ref = torch.from_numpy(x.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    nan = np.isnan(x)
    assert np.array_equal(ours[~nan], ref[~nan])
    assert np.all(np.isnan(O.bf16_to_f32(ours[nan])))


# ------------------------------------------------------------ identities ---

@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_identity_no_scale_mask_perturb(dtype):
    """alpha = 1, p_keep = 1, sigma = 0: theta~ is theta bit for bit
    (Eq. expert-displacement with alpha m = 1 and eps = 0)."""
    r = rng(5)
    n = 4099
    th = r.standard_normal(n).astype(np.float32) * np.float32(3.0)
    t0 = r.standard_normal(n).astype(np.float32) * np.float32(1e-3)
    th[:4] = f32([0.0, -0.0, 1e30, -1e-40])
    t0[:4] = f32([1e30, 5.0, -1e30, 7.0])
    if dtype == O.BF16:
        th, t0 = O.f32_to_bf16(th), O.f32_to_bf16(t0)
    cfg = O.config(alpha_min=1.0, alpha_max=1.0, step=3)
    t = O.tensor(11, n, dtype=dtype, keep_prob=1.0, sigma=0.0)
    out = O.simulate(cfg, t, th, t0)
    assert out.tobytes() == np.asarray(th).tobytes()


@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_all_dropped_without_noise_is_theta0(dtype):
    """p_keep = 0, sigma = 0: every coordinate is masked, theta~ = theta0."""
    r = rng(6)
    n = 1000
    th = r.standard_normal(n).astype(np.float32)
    t0 = r.standard_normal(n).astype(np.float32)
    if dtype == O.BF16:
        th, t0 = O.f32_to_bf16(th), O.f32_to_bf16(t0)
    t = O.tensor(3, n, dtype=dtype, keep_prob=0.0, sigma=0.0)
    out = O.simulate(O.config(), t, th, t0)
    assert out.tobytes() == np.asarray(t0).tobytes()


def test_no_mask_closed_form():
    """Mask off (p_keep = 1), fixed alpha = 0.75, no noise: theta~ = theta0 +
    0.75 (theta - theta0) rounded once (Eq. smat-state), computed here in
    float64 from the fp32 difference."""
    r = rng(7)
    n = 5000
    th = r.standard_normal(n).astype(np.float32)
    t0 = r.standard_normal(n).astype(np.float32)
    cfg = O.config(alpha_min=0.75, alpha_max=0.75)
    t = O.tensor(1, n, keep_prob=1.0)
    out = O.simulate(cfg, t, th, t0)
    d = (th - t0).astype(np.float64)
    ref = (t0.astype(np.float64) + 0.75 * d).astype(np.float32)
    assert np.array_equal(out, ref)


def test_masked_closed_form_and_kept_set():
    """alpha = 0.5, p_keep = 0.25 (rescale 4): kept coordinates are
    theta0 + 2 (theta - theta0), dropped ones theta0 (Eq. smat-mask rescaling);
    the kept set is the one mask_bits reports."""
    r = rng(8)
    n = 8192
    th = r.standard_normal(n).astype(np.float32)
    t0 = r.standard_normal(n).astype(np.float32)
    cfg = O.config(alpha_min=0.5, alpha_max=0.5, step=9)
    t = O.tensor(21, n, keep_prob=0.25)
    out = O.simulate(cfg, t, th, t0)
    kept = O.unpack_bits(O.mask_bits(cfg, t), n).astype(bool)
    d = (th - t0).astype(np.float64)
    ref = np.where(kept, (t0.astype(np.float64) + 2.0 * d).astype(np.float32), t0)
    assert np.array_equal(out, ref)
    assert 0.2 < kept.mean() < 0.3


def test_scalars_inverse_keep_and_threshold():
    """1 / p_keep is the Eq. smat-mask rescale 1 / (1 - p); the threshold is
    floor(p_keep 2^32)."""
    for pk in (0.0, 0.1, 0.3, 0.5, 0.7, 0.9, 1.0, 2.0**-20):
        s = O.scalars(O.config(), O.tensor(5, 10, keep_prob=pk))
        assert s["T"] == math.floor(float(np.float32(pk)) * 2**32)
        if pk > 0:
            assert s["inv_keep"] == float(np.float32(1.0 / float(np.float32(pk))))


# ---------------------------------------------------------- Mask (Eq. 4) ---

@pytest.mark.parametrize("pk", [0.1, 0.3, 0.5, 0.7, 0.9])
def test_keep_rate_binomial(pk):
    """Empirical keep rate within a 5-sigma binomial bound of p_keep."""
    n = 200_000
    t = O.tensor(1234, n, keep_prob=pk)
    k = O.unpack_bits(O.mask_bits(O.config(seed=5, step=1), t), n).sum()
    p = float(np.float32(pk))
    assert abs(k - n * p) <= 5 * math.sqrt(n * p * (1 - p))


def test_keep_threshold_low_24_bits_on_ties():
    """kept <=> U < floor(p_keep 2^32) with U uniform on 32 bits: masks at nested
    keep probabilities are nested (one uniform per coordinate), and between
    p = 128/256 and p = 129/256 lie exactly the coordinates whose high byte is
    128. At p = 1/2 + 2^-10 the low 24 bits of the threshold are 2^22, so a
    quarter of those must be kept: treating the tie as always kept (rate 1) or
    always dropped (rate 0) fails."""
    n = 2_000_000
    cfg = O.config(seed=11)

    def kept(pk):
        return O.unpack_bits(O.mask_bits(cfg, O.tensor(77, n, keep_prob=pk)), n).astype(bool)

    lo, mid, hi = kept(0.5), kept(0.5 + 2.0**-10), kept(129 / 256)
    assert np.all(lo <= mid) and np.all(mid <= hi)
    ties = hi & ~lo
    m = int(ties.sum())
    assert abs(m - n / 256) < 5 * math.sqrt(n / 256)
    rate = mid[ties].mean()
    assert abs(rate - 0.25) < 5 * math.sqrt(0.25 * 0.75 / m)


def test_mask_has_no_lag_correlation():
    """Coordinates are masked independently (Eq. smat-mask): for lags inside and
    across the 4- and 16-element draw groups, P(both kept) = p^2."""
    n = 400_000
    pk = 0.5
    m = O.unpack_bits(O.mask_bits(O.config(seed=3), O.tensor(9, n, keep_prob=pk)), n).astype(np.float64)
    for lag in (1, 2, 3, 4, 5, 8, 12, 15, 16, 17, 32, 64):
        both = (m[:-lag] * m[lag:]).mean()
        se = math.sqrt(0.25 * 0.75 / (n - lag))
        assert abs(both - 0.25) < 6 * se, lag


def test_masks_differ_across_tensors_steps_seeds():
    n = 4096
    base = O.mask_bits(O.config(seed=1, step=2), O.tensor(5, n, keep_prob=0.5))
    for cfg, tid in ((O.config(seed=1, step=3), 5), (O.config(seed=2, step=2), 5), (O.config(seed=1, step=2), 6)):
        other = O.mask_bits(cfg, O.tensor(tid, n, keep_prob=0.5))
        agree = np.mean(O.unpack_bits(base, n) == O.unpack_bits(other, n))
        assert 0.45 < agree < 0.55


def test_mask_moments_over_steps():
    """E[m_k] = 1 and E[m_k^2] = 1 / (1 - p_k) (proof of Prop. moments, App. C),
    m = kept / p_keep, over many steps."""
    n, steps, pk = 512, 600, 0.3
    acc1 = np.zeros(n)
    acc2 = np.zeros(n)
    for s in range(steps):
        kept = O.unpack_bits(O.mask_bits(O.config(seed=4, step=s), O.tensor(2, n, keep_prob=pk)), n)
        m = kept / pk
        acc1 += m
        acc2 += m * m
    tot = n * steps
    e1, e2 = acc1.sum() / tot, acc2.sum() / tot
    sd1 = math.sqrt((1 / pk - 1) / tot)
    sd2 = math.sqrt((1 / pk**3 - 1 / pk**2) / tot)
    assert abs(e1 - 1.0) < 5 * sd1
    assert abs(e2 - 1 / pk) < 5 * sd2


# ------------------------------------------------------- Scale and noise ---

def test_alpha_uniform_per_tensor_and_global():
    """Scale: alpha ~ U[alpha_min, alpha_max) (Sec. 4.1); one scalar for every
    tensor in global mode, independent draws per tensor in per-tensor mode."""
    amin, amax = 0.3, 1.0
    al = []
    for s in range(3000):
        al.append(O.scalars(O.config(seed=8, step=s, alpha_min=amin, alpha_max=amax), O.tensor(4, 1))["alpha"])
    al = np.array(al)
    assert al.min() >= amin and al.max() < amax
    assert stats.kstest((al - amin) / (amax - amin), "uniform").pvalue > 1e-4
    g = O.config(seed=8, step=0, alpha_mode=O.ALPHA_GLOBAL)
    ga = {O.scalars(g, O.tensor(tid, 1))["alpha"] for tid in range(20)}
    assert len(ga) == 1
    pt = O.config(seed=8, step=0, alpha_mode=O.ALPHA_PER_TENSOR)
    pa = {O.scalars(pt, O.tensor(tid, 1))["alpha"] for tid in range(20)}
    assert len(pa) == 20


def _alpha_per_element(cfg, tid, n, elem_offset=0):
    """Per-element alpha of n coordinates, read through the gradient map: with
    p_keep = 1 every coordinate is kept and rescaled by 1, so g~ = 1 maps to
    alpha_i itself (Eq. smat-gradient)."""
    t = O.tensor(tid, n, keep_prob=1.0, elem_offset=elem_offset)
    return O.gradmap(cfg, t, np.ones(n, np.float32)).astype(np.float64)


@pytest.mark.parametrize("amin,amax", [(0.0, 1.0), (0.3, 0.8)])
def test_alpha_per_element_law(amin, amax):
    """Scale per coordinate (Sec. 4.1, reading R4): alpha_i ~ U[alpha_min,
    alpha_max), independent across coordinates (lags inside and across the
    4-coordinate draw blocks) and independent of the same coordinate's Mask and
    Perturb draws."""
    n = 1 << 18
    cfg = O.config(seed=31, step=3, alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=amin, alpha_max=amax,
                   noise=O.NOISE_GAUSSIAN)
    a = _alpha_per_element(cfg, 40, n)
    assert a.min() >= amin and a.max() < amax
    assert stats.kstest((a - amin) / (amax - amin), "uniform").pvalue > 1e-4
    assert abs(a.mean() - (amin + amax) / 2) < 5 * (amax - amin) / math.sqrt(12 * n)
    se = 1 / math.sqrt(n)
    for lag in (1, 2, 3, 4, 5, 8, 16):
        assert abs(np.corrcoef(a[:-lag], a[lag:])[0, 1]) < 5 * se, lag
    # Mask of the same coordinates at p_keep = 1/2
    kept = O.unpack_bits(O.mask_bits(cfg, O.tensor(40, n, keep_prob=0.5)), n).astype(np.float64)
    assert abs(np.corrcoef(a, kept)[0, 1]) < 5 * se
    # Perturb of the same coordinates
    z = O.noise_z(cfg, O.tensor(40, n, keep_prob=1.0, sigma=1.0), np.arange(n))
    assert abs(np.corrcoef(a, z)[0, 1]) < 5 * se
    assert abs(np.corrcoef(a, np.abs(z))[0, 1]) < 5 * se
    # and the kept rescaled coordinates carry alpha_i / p_keep
    g = O.gradmap(cfg, O.tensor(40, n, keep_prob=0.5), np.ones(n, np.float32)).astype(np.float64)
    on = kept.astype(bool)
    assert np.array_equal(g[on], (a[on].astype(np.float32) * np.float32(2.0)).astype(np.float64))
    assert np.all(g[~on] == 0.0)


def _packed_field24(words12, k):
    """The 24-bit field of element k (0..15) of a 16-element group from the
    group's twelve words: quad q = k // 4 reads words 3q, 3q + 1, 3q + 2; its
    first three elements take their top 24 bits, the fourth their low bytes."""
    q, r = k >> 2, k & 3
    A, B, C = (int(words12[3 * q + m]) for m in range(3))
    if r < 3:
        return (A, B, C)[r] >> 8
    return (A & 255) | ((B & 255) << 8) | ((C & 255) << 16)


def test_alpha_per_element_stream_layout_matches_triton_library():
    """Coordinate gidx's alpha comes from the 24-bit field of gidx in the
    ALPHA_E stream (stream 2): the twelve words of blocks 3 (gidx div 16) + b,
    b = 0, 1, 2, of Triton's Philox serve the group's sixteen coordinates,
    three words per quad of four (reading R22). (alpha_i - alpha_min) /
    (alpha_max - alpha_min) equals that field times 2^-24 to within the fp32
    rounding of the affine map. Covers element offsets and draw-block indices
    at and above 2^32 (counter word 1); the noise field has the same packing
    (R18) and shares the oracle's routine."""
    seed, step, tid, amin, amax = 0x0DDB1A5E5BADDEC0, 6, 0x0ABCDEF, 0.25, 0.875
    cfg = O.config(seed=seed, step=step, alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=amin, alpha_max=amax)
    cases = [(0, 40), (13, 19), ((1 << 36) - 6, 12), (3 << 36, 8)]
    groups = sorted({(off + i) >> 4 for off, n in cases for i in range(n)})
    ctrs = []
    for g in groups:
        for b in range(3):
            j = 3 * g + b
            ctrs.append([j & 0xFFFFFFFF, j >> 32, (2 << 28) | tid, step])
    assert any((3 * g) >> 32 for g in groups)
    words = _triton_philox(ctrs, [seed] * len(ctrs), 10)
    w12 = {g: np.concatenate([words[3 * n + b] for b in range(3)]) for n, g in enumerate(groups)}
    back, exp, wrong = [], [], []
    for off, n in cases:
        a = _alpha_per_element(cfg, tid, n, elem_offset=off)
        for i in range(n):
            gidx = off + i
            k = gidx & 15
            back.append((a[i] - amin) / (amax - amin))
            exp.append(_packed_field24(w12[gidx >> 4], k) * 2.0**-24)
            wrong.append(_packed_field24(w12[gidx >> 4], (k & 12) | ((k + 1) & 3)) * 2.0**-24)
    back, exp, wrong = np.array(back), np.array(exp), np.array(wrong)
    assert np.all(np.abs(back - exp) <= 2.0**-22), np.max(np.abs(back - exp))
    # another coordinate's field is an unrelated uniform
    assert np.mean(np.abs(back - wrong) <= 2.0**-22) < 0.1


def test_uniform_noise_law():
    """Perturb: eps ~ U[-sqrt3 sigma, sqrt3 sigma] (Sec. 4.1): with theta0 = 0 and
    every coordinate dropped, theta~ = eps exactly; mean 0, variance sigma^2,
    support inside the interval, KS against the uniform law."""
    n, sigma = 200_000, 2e-3
    t = O.tensor(8, n, keep_prob=0.0, sigma=sigma)
    z = np.zeros(n, np.float32)
    eps = O.simulate(O.config(seed=6, noise=O.NOISE_UNIFORM), t, z, z).astype(np.float64)
    a = math.sqrt(3.0) * sigma
    assert np.all(np.abs(eps) <= a * (1 + 1e-6))
    assert abs(eps.mean()) < 5 * sigma / math.sqrt(n)
    assert abs(eps.var() / sigma**2 - 1) < 5 * math.sqrt(0.8 / n)
    assert stats.kstest(eps / a, "uniform", args=(-1, 2)).pvalue > 1e-4


def test_erfinv_matches_scipy_library():
    """The Gaussian transform's erfinv (double, by Newton on erf / erfc)
    against scipy.special.erfinv, including the extreme inputs
    +-(1 - 2^-24) that sym() can produce."""
    from scipy.special import erfinv as sp_erfinv
    r = rng(30)
    k = r.integers(0, 2**24, size=20000)
    v = (2.0 * k + 1 - 2**24) * 2.0**-24
    v = np.concatenate([v, [1 - 2.0**-24, -(1 - 2.0**-24), 2.0**-24, -(2.0**-24), 0.5 + 2.0**-24, 0.75, -0.999]])
    ours = O.erfinv(v)
    ref = sp_erfinv(v)
    assert np.allclose(ours, ref, rtol=1e-13, atol=0)
    assert np.array_equal(np.sign(ours), np.sign(v))


def test_gaussian_noise_law():
    """Gaussian Perturb (eps ~ N(0, sigma^2)): KS against N(0, 1), unit
    variance, symmetric, and neighbouring coordinates uncorrelated (one
    independent word per coordinate)."""
    n, sigma = 200_000, 1e-4
    t = O.tensor(8, n, keep_prob=0.0, sigma=sigma)
    z = np.zeros(n, np.float32)
    eps = O.simulate(O.config(seed=6, noise=O.NOISE_GAUSSIAN), t, z, z).astype(np.float64) / sigma
    assert stats.kstest(eps, "norm").pvalue > 1e-4
    assert abs(eps.var() - 1) < 5 * math.sqrt(2.0 / n)
    assert abs(eps.mean()) < 5 / math.sqrt(n)
    for lag in (1, 2, 3, 4, 16):
        assert abs(np.corrcoef(eps[:-lag], eps[lag:])[0, 1]) < 5 / math.sqrt(n), lag


def test_gaussian_z_matches_noise_of_simulate():
    """eps = fl(sqrt2 sigma) * fl(erfinv(v)) equals sigma z, z = sqrt2 erfinv(v),
    to within fp32 rounding."""
    n = 4096
    sigma = 1.0
    t = O.tensor(8, n, keep_prob=0.0, sigma=sigma)
    z = np.zeros(n, np.float32)
    cfg = O.config(seed=9, noise=O.NOISE_GAUSSIAN)
    eps = O.simulate(cfg, t, z, z).astype(np.float64)
    zz = O.gauss_z(cfg, t, np.arange(n))
    assert np.allclose(eps, zz, rtol=3 * 2.0**-24, atol=0)


def test_laplace_transform_closed_forms():
    """Laplace inverse-CDF transform z(v) = -sign(v) ln(1 - |v|): z(+-1/2) =
    +-ln 2, z(1 - 2^-k) = k ln 2 (both exact in double), z(0) = 0, exactly odd
    and strictly increasing over the noise grid sym24(u)."""
    k = np.arange(1, 25)
    v = np.concatenate([[0.5, -0.5, 0.0], 1 - 2.0**-k])
    z = O.laplace(v)
    assert z[0] == math.log(2) and z[1] == -math.log(2) and z[2] == 0.0
    assert np.allclose(z[3:], k * math.log(2), rtol=1e-15, atol=0)
    u = np.arange(0, 1 << 24, 4099, dtype=np.int64)
    g = (2 * u + 1 - (1 << 24)).astype(np.float64) * 2.0**-24
    zg = O.laplace(g)
    assert np.array_equal(O.laplace(-g), -zg)
    assert np.all(np.diff(zg) > 0)


def test_laplace_law_on_the_noise_grid():
    """Over all 2^24 values of sym24(u), z(v) is Laplace(0, 1): its CDF is
    within the grid's 2^-24 steps of 1/2 e^x (x < 0) / 1 - 1/2 e^-x, its mean
    is 0 and its variance 2 (matched RMS: eps = (sigma / sqrt2) z has variance
    sigma^2)."""
    u = np.arange(1 << 24, dtype=np.int64)
    v = (2 * u + 1 - (1 << 24)).astype(np.float64) * 2.0**-24
    z = O.laplace(v)  # increasing in u
    x = np.array([-6.0, -2.0, -0.5, -0.1, 0.0, 0.1, 0.5, 2.0, 6.0])
    emp = np.searchsorted(z, x, side="right") / z.size
    cdf = np.where(x < 0, 0.5 * np.exp(x), 1 - 0.5 * np.exp(-x))
    assert np.max(np.abs(emp - cdf)) <= 2.0**-23
    assert abs(z.mean()) < 1e-12
    assert abs(z.var() - 2.0) < 1e-4


def test_laplace_noise_law_in_simulate():
    """Laplace Perturb through the full forward: RMS sigma, the Laplace
    kurtosis 6 (uniform: 1.8, Gaussian: 3), KS against Laplace(0, 1/sqrt2) of
    eps / sigma, and the unit variates of noise_z match eps / sigma."""
    n, sigma = 200_000, 1e-4
    t = O.tensor(8, n, keep_prob=0.0, sigma=sigma)
    zero = np.zeros(n, np.float32)
    cfg = O.config(seed=6, noise=O.NOISE_LAPLACE)
    eps = O.simulate(cfg, t, zero, zero).astype(np.float64) / sigma
    assert abs(eps.var() - 1) < 5 * math.sqrt(5.0 / n)
    kurt = np.mean(eps**4) / eps.var() ** 2
    assert abs(kurt - 6.0) < 0.3
    assert stats.kstest(eps, "laplace", args=(0.0, 1 / math.sqrt(2))).pvalue > 1e-4
    z = O.noise_z(cfg, t, np.arange(n))
    assert np.allclose(eps, z, rtol=4 * 2.0**-24, atol=1e-12)


# ------------------------------------------- Prop. moments (App. C) ---

def test_state_moments_proposition():
    """Prop. moments (App. C), global alpha: mean theta0 + abar Delta; covariance
    v_a Delta Delta^T + s_a Diag(Delta^2 p/(1-p)) + sigma^2 I (p the drop
    probability), checked coordinate-wise and on off-diagonal pairs."""
    r = rng(10)
    n, steps = 24, 6000
    amin, pk, sigma = 0.2, 0.6, 0.05
    t0 = r.standard_normal(n).astype(np.float32)
    delta = (r.standard_normal(n) * 0.5 + np.sign(r.standard_normal(n))).astype(np.float32)
    th = (t0 + delta).astype(np.float32)
    D = (th - t0).astype(np.float64)
    X = np.zeros((steps, n))
    for s in range(steps):
        cfg = O.config(seed=12, step=s, alpha_mode=O.ALPHA_GLOBAL, alpha_min=amin, alpha_max=1.0)
        X[s] = O.simulate(cfg, O.tensor(3, n, keep_prob=pk, sigma=sigma), th, t0)
    abar = (1 + amin) / 2
    va = (1 - amin) ** 2 / 12
    sa = abar**2 + va
    p_drop = 1 - pk
    mean_ref = t0 + abar * D
    var_ref = va * D**2 + sa * D**2 * p_drop / (1 - p_drop) + sigma**2
    mean = X.mean(0)
    C = np.cov(X.T, bias=True)
    assert np.all(np.abs(mean - mean_ref) < 5 * np.sqrt(var_ref / steps))
    # variance: standard error of a sample variance <= sqrt((m4 - var^2) / steps)
    m4 = ((X - mean) ** 4).mean(0)
    assert np.all(np.abs(np.diag(C) - var_ref) < 5 * np.sqrt((m4 - np.diag(C) ** 2) / steps) + 1e-12)
    # off-diagonal: only the shared alpha correlates coordinates
    Xc = X - mean
    for (k, l) in ((0, 1), (2, 7), (5, 19), (10, 11)):
        prod = Xc[:, k] * Xc[:, l]
        ref = va * D[k] * D[l]
        assert abs(prod.mean() - ref) < 5 * prod.std() / math.sqrt(steps), (k, l)


def test_state_moments_proposition_per_element_alpha():
    """Prop. moments (App. C) with alpha drawn per coordinate (reading R4):
    the mean is still theta0 + abar Delta and each coordinate's variance is
    v_a Delta^2 + s_a Delta^2 p/(1-p) + sigma^2, but coordinates no longer
    share a scale, so every off-diagonal covariance is 0 (the shared-alpha
    term v_a Delta_k Delta_l of the global mode vanishes)."""
    r = rng(32)
    n, steps = 24, 6000
    amin, pk, sigma = 0.2, 0.6, 0.05
    t0 = r.standard_normal(n).astype(np.float32)
    delta = (r.standard_normal(n) * 0.5 + np.sign(r.standard_normal(n))).astype(np.float32)
    th = (t0 + delta).astype(np.float32)
    D = (th - t0).astype(np.float64)
    X = np.zeros((steps, n))
    for s in range(steps):
        cfg = O.config(seed=13, step=s, alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=amin, alpha_max=1.0)
        X[s] = O.simulate(cfg, O.tensor(3, n, keep_prob=pk, sigma=sigma), th, t0)
    abar = (1 + amin) / 2
    va = (1 - amin) ** 2 / 12
    sa = abar**2 + va
    p_drop = 1 - pk
    mean_ref = t0 + abar * D
    var_ref = va * D**2 + sa * D**2 * p_drop / (1 - p_drop) + sigma**2
    mean = X.mean(0)
    assert np.all(np.abs(mean - mean_ref) < 5 * np.sqrt(var_ref / steps))
    var = X.var(0)
    m4 = ((X - mean) ** 4).mean(0)
    assert np.all(np.abs(var - var_ref) < 5 * np.sqrt((m4 - var**2) / steps) + 1e-12)
    Xc = X - mean
    for (k, l) in ((0, 1), (2, 3), (4, 7), (5, 19), (10, 11), (15, 16)):
        prod = Xc[:, k] * Xc[:, l]
        assert abs(prod.mean()) < 5 * prod.std() / math.sqrt(steps), (k, l)
    # the shared-alpha covariance of the global mode is far outside that band
    big = max(((k, l) for k in range(n) for l in range(k + 1, n)), key=lambda kl: abs(D[kl[0]] * D[kl[1]]))
    prod = Xc[:, big[0]] * Xc[:, big[1]]
    assert abs(va * D[big[0]] * D[big[1]]) > 5 * prod.std() / math.sqrt(steps)


# ---------------------------------------------- gradient (Eq. smat-gradient) ---

@pytest.mark.parametrize("mode", [O.ALPHA_PER_TENSOR, O.ALPHA_PER_ELEMENT])
def test_gradient_map_matches_finite_differences(mode):
    """With the draws fixed, the gradient of L(theta~(theta)) w.r.t. theta is
    alpha m (.) grad L(theta~) (Eq. smat-gradient). L = 1/2 sum w theta~^2,
    central differences in double."""
    r = rng(13)
    n = 61
    th = r.standard_normal(n)
    t0 = r.standard_normal(n)
    w = r.standard_normal(n)
    cfg = O.config(seed=21, step=4, alpha_mode=mode, alpha_min=0.2, alpha_max=1.0, noise=O.NOISE_GAUSSIAN)
    t = O.tensor(6, n, keep_prob=0.7, sigma=0.01)

    def loss(x):
        y = O.simulate_f64(cfg, t, 0.01, x, t0)
        return 0.5 * np.sum(w * y * y)

    y = O.simulate_f64(cfg, t, 0.01, th, t0)
    g = O.gradmap_f64(cfg, t, w * y)
    h = 1e-6
    fd = np.zeros(n)
    for k in range(n):
        e = np.zeros(n)
        e[k] = h
        fd[k] = (loss(th + e) - loss(th - e)) / (2 * h)
    assert np.allclose(g, fd, rtol=1e-6, atol=1e-8)
    kept = O.unpack_bits(O.mask_bits(O.config(seed=21, step=4, alpha_mode=mode), t), n).astype(bool)
    assert np.all(g[~kept] == 0.0) and np.all(g[kept] != 0.0)


def test_gradient_fp32_agrees_with_real_arithmetic():
    r = rng(14)
    n = 3000
    gs = r.standard_normal(n).astype(np.float32)
    cfg = O.config(seed=2, step=1, alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=0.0, alpha_max=1.0)
    t = O.tensor(4, n, keep_prob=0.3)
    g32 = O.gradmap(cfg, t, gs).astype(np.float64)
    g64 = O.gradmap_f64(cfg, t, gs.astype(np.float64))
    assert np.allclose(g32, g64, rtol=2 * 2**-24, atol=0)


def test_gradient_zero_when_alpha_zero():
    """alpha = 0: no coordinate contributes, the mapped gradient is 0 (Sec. 4.2)."""
    n = 777
    gs = rng(15).standard_normal(n).astype(np.float32)
    cfg = O.config(alpha_min=0.0, alpha_max=0.0)
    out = O.gradmap(cfg, O.tensor(1, n, keep_prob=0.5), gs)
    assert np.all(out == 0.0)


def test_gradient_of_ones_is_rescaled_mask():
    """g~ = 1 maps to c on kept coordinates and 0 elsewhere, c = alpha / p_keep."""
    n = 5000
    cfg = O.config(seed=3, step=5)
    t = O.tensor(17, n, keep_prob=0.7)
    g = O.gradmap(cfg, t, np.ones(n, np.float32))
    c = O.scalars(cfg, t)["c"]
    kept = O.unpack_bits(O.mask_bits(cfg, t), n).astype(bool)
    assert np.all(g[kept] == np.float32(c)) and np.all(g[~kept] == 0.0)


def test_gradient_accumulate_adds():
    r = rng(16)
    n = 1000
    gs = r.standard_normal(n).astype(np.float32)
    go = r.standard_normal(n).astype(np.float32)
    cfg = O.config(seed=3)
    t = O.tensor(2, n, keep_prob=0.5)
    plain = O.gradmap(cfg, t, gs)
    acc = O.gradmap(cfg, t, gs, accumulate=True, g_old=go)
    assert np.array_equal(acc, (go + plain).astype(np.float32))


# ---------------------------------------------------- consistency checks ---

def test_forward_kept_set_equals_gradient_kept_set():
    """The gradient map regenerates the forward's mask (App. D): the kept flags of
    the forward are exactly the nonzero pattern of the mapped ones."""
    n = 3000
    r = rng(17)
    th = r.standard_normal(n).astype(np.float32)
    t0 = r.standard_normal(n).astype(np.float32)
    cfg = O.config(seed=5, step=2, noise=O.NOISE_GAUSSIAN)
    t = O.tensor(99, n, keep_prob=0.4, sigma=1e-3)
    _, kept = O.simulate_at(cfg, t, 1e-3, np.arange(n), th, t0)
    g = O.gradmap(cfg, t, np.ones(n, np.float32))
    assert np.array_equal(kept.astype(bool), g != 0)


@pytest.mark.parametrize("split", [1, 15, 16, 17, 1000, 2999])
def test_shard_invariance(split):
    """Element offsets make any contiguous sharding produce the same bits."""
    n = 3000
    r = rng(18)
    th = r.standard_normal(n).astype(np.float32)
    t0 = r.standard_normal(n).astype(np.float32)
    cfg = O.config(seed=7, step=1, alpha_mode=O.ALPHA_PER_ELEMENT, noise=O.NOISE_GAUSSIAN)
    full = O.simulate(cfg, O.tensor(4, n, keep_prob=0.6, sigma=1e-2), th, t0)
    a = O.simulate(cfg, O.tensor(4, split, keep_prob=0.6, sigma=1e-2), th[:split], t0[:split])
    b = O.simulate(cfg, O.tensor(4, n - split, keep_prob=0.6, sigma=1e-2, elem_offset=split),
                   th[split:], t0[split:])
    assert np.array_equal(full, np.concatenate([a, b]))


def test_simulate_at_matches_full_tensor():
    n = 2000
    r = rng(19)
    th = O.f32_to_bf16(r.standard_normal(n).astype(np.float32) * 0.02)
    t0 = O.f32_to_bf16(r.standard_normal(n).astype(np.float32) * 0.02)
    cfg = O.config(seed=5, noise=O.NOISE_GAUSSIAN)
    t = O.tensor(12, n, dtype=O.BF16, keep_prob=0.7, sigma_rel=0.1)
    full = O.simulate(cfg, t, th, t0)
    sig = O.delta_stats(t, th, t0)["sigma"]
    idx = r.choice(n, 300, replace=False)
    bits, _ = O.simulate_at(cfg, t, sig, idx, O.bf16_to_f32(th[idx]), O.bf16_to_f32(t0[idx]))
    assert np.array_equal(bits.astype(np.uint16), full[idx])


@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
@pytest.mark.parametrize("mode", [O.ALPHA_GLOBAL, O.ALPHA_PER_TENSOR, O.ALPHA_PER_ELEMENT])
@pytest.mark.parametrize("noise", [O.NOISE_UNIFORM, O.NOISE_GAUSSIAN, O.NOISE_LAPLACE])
def test_at_index_evaluation_matches_full_tensor(dtype, mode, noise):
    """The sampled evaluations (simulate_at, gradmap_at: what the full-size GPU
    checks compare against) give the bits of the whole-tensor forward and
    gradient map at every sampled index, with an element offset, mask ties in
    range, and with and without accumulation."""
    r = rng(41 + 3 * mode + noise)
    n, off = 3001, (1 << 33) + 7
    th = r.standard_normal(n).astype(np.float32) * np.float32(0.02)
    t0 = r.standard_normal(n).astype(np.float32) * np.float32(0.02)
    gs = r.standard_normal(n).astype(np.float32)
    go = r.standard_normal(n).astype(np.float32)
    if dtype == O.BF16:
        th, t0, gs, go = O.f32_to_bf16(th), O.f32_to_bf16(t0), O.f32_to_bf16(gs), O.f32_to_bf16(go)
    f = (lambda x: O.bf16_to_f32(x)) if dtype == O.BF16 else (lambda x: x)
    cfg = O.config(seed=77, step=9, alpha_mode=mode, noise=noise, alpha_min=0.1, alpha_max=0.9)
    t = O.tensor(31, n, dtype=dtype, keep_prob=0.5 + 2.0**-10, sigma=3e-3, elem_offset=off)
    idx = np.sort(r.choice(n, 700, replace=False))
    bits_t = np.uint16 if dtype == O.BF16 else np.uint32
    full = O.simulate(cfg, t, th, t0).view(bits_t)
    bits, kept = O.simulate_at(cfg, t, 3e-3, idx, f(th)[idx], f(t0)[idx])
    assert np.array_equal(bits.astype(bits_t), full[idx])
    mb = O.unpack_bits(O.mask_bits(cfg, t), n)
    assert np.array_equal(kept, mb[idx])
    for acc in (False, True):
        gfull = O.gradmap(cfg, t, gs, gdtype=dtype, accumulate=acc, g_old=go if acc else None).view(bits_t)
        gat = O.gradmap_at(cfg, t, idx, f(gs)[idx], gdtype=dtype, accumulate=acc,
                           gold_vals=f(go)[idx] if acc else None)
        assert np.array_equal(gat.astype(bits_t), gfull[idx]), acc


def test_delta_stats_match_numpy():
    """sigma_t = sigma_rel * population std of theta - theta0."""
    r = rng(20)
    n = 100_003
    t0 = O.f32_to_bf16(r.standard_normal(n).astype(np.float32) * 0.02)
    d = r.standard_normal(n).astype(np.float32) * 3e-4 + 1e-4
    th = O.f32_to_bf16(O.bf16_to_f32(t0) + d)
    t = O.tensor(1, n, dtype=O.BF16, sigma_rel=0.1)
    s = O.delta_stats(t, th, t0)
    dd = (O.bf16_to_f32(th) - O.bf16_to_f32(t0)).astype(np.float64)
    assert math.isclose(s["mean"], dd.mean(), rel_tol=1e-12)
    assert math.isclose(s["sigma"], float(np.float32(0.1 * dd.std())), rel_tol=1e-6)


def test_paper_default_settings_fixture():
    """The paper's stated SMAT settings (tests/golden/paper_settings.json) give
    the intended Mask keep rate and Perturb RMS."""
    with open(os.path.join(HERE, "golden", "paper_settings.json")) as f:
        gold = json.load(f)
    for name, s in gold["settings"].items():
        pk = 1.0 - s["mask_drop_p"]
        n = 100_000
        t = O.tensor(1, n, keep_prob=pk, sigma=s["perturb_rms"])
        cfg = O.config(seed=1, alpha_min=s["alpha_min"], alpha_max=1.0, noise=O.NOISE_UNIFORM)
        k = O.unpack_bits(O.mask_bits(cfg, t), n).sum()
        assert abs(k - n * pk) <= 5 * math.sqrt(n * pk * (1 - pk)), name
        z = np.zeros(n, np.float32)
        eps = O.simulate(cfg, O.tensor(1, n, keep_prob=0.0, sigma=s["perturb_rms"]), z, z)
        assert abs(np.sqrt(np.mean(eps.astype(np.float64) ** 2)) / s["perturb_rms"] - 1) < 0.01, name


def test_oracle_regression_fixture():
    """The oracle still reproduces its committed outputs (guards against an
    unintended change of the stream specification)."""
    with open(os.path.join(HERE, "golden", "oracle_regression.json")) as f:
        doc = json.load(f)
    for c in doc["cases"]:
        cfg = O.OrcConfig(**c["config"])
        t = O.OrcTensor(**c["tensor"])
        pd = np.uint16 if t.dtype == O.BF16 else np.uint32
        gd = np.uint16 if c["gdtype"] == O.BF16 else np.uint32
        th = np.array(c["theta_bits"], pd)
        t0 = np.array(c["theta0_bits"], pd)
        gs = np.array(c["gsim_bits"], gd)
        if t.dtype == O.F32:
            th, t0 = th.view(np.float32), t0.view(np.float32)
        if c["gdtype"] == O.F32:
            gs = gs.view(np.float32)
        sim = np.asarray(O.simulate(cfg, t, th, t0)).view(pd)
        g = np.asarray(O.gradmap(cfg, t, gs, gdtype=c["gdtype"])).view(gd)
        assert sim.tolist() == c["sim_bits"], c["name"]
        assert g.tolist() == c["g_bits"], c["name"]
        assert O.mask_bits(cfg, t).tolist() == c["mask_words"], c["name"]


# ------------------------------------------- merging (Eq. merged-state) ---

def _dyadic(r, n, scale=2.0**-6):
    """Small multiples of 2^-10: differences, sums and products by the
    coefficients below are exact in fp32, so results equal exact rationals."""
    return (r.integers(-64, 65, n) * scale / 16).astype(np.float32)


def test_merge_ta_wa_closed_forms_and_identities():
    """TA: theta0 + gamma sum_j Delta_j, WA: theta0 + (1/K) sum_j Delta_j
    (Sec. 3.1), against exact rational arithmetic on dyadic inputs; gamma = 0
    gives theta0; permuting the experts changes nothing (exact sums)."""
    r = rng(30)
    n, K = 257, 4
    t0 = _dyadic(r, n)
    ex = [_dyadic(r, n) for _ in range(K)]
    exact_sum = sum(e.astype(np.float64) - t0 for e in ex)
    ta, _ = O.merge(O.MERGE_TA, t0, ex, gamma=0.5)
    assert np.array_equal(ta.astype(np.float64), t0 + 0.5 * exact_sum)
    wa, _ = O.merge(O.MERGE_WA, t0, ex)
    assert np.array_equal(wa.astype(np.float64), t0 + exact_sum / K)
    z, _ = O.merge(O.MERGE_TA, t0, ex, gamma=0.0)
    assert np.array_equal(z, t0)
    perm, _ = O.merge(O.MERGE_TA, t0, ex[::-1], gamma=0.5)
    assert np.array_equal(perm, ta)


def test_merge_dare_masks_are_the_smat_mask_stream():
    """DARE (Yu et al.) drops each coordinate of Delta_j with probability p and
    rescales the rest by 1/(1-p); expert j's mask is the SMAT Mask stream at
    step j: with one expert at a time, the kept set equals mask_bits at that
    step, the keep rate is binomial, p = 0 is TA exactly, and the merge is
    unbiased over seeds."""
    r = rng(31)
    n, K, p = 20_000, 3, 0.3
    t0 = _dyadic(r, n)
    ex = [_dyadic(r, n) + np.float32(1.0) for _ in range(K)]  # Delta never 0
    for j in range(K):
        one = [t0.copy() for _ in range(K)]
        one[j] = ex[j]
        out, _ = O.merge(O.MERGE_DARE_TA, t0, one, gamma=1.0, p_drop=p, seed=77, tensor_id=5)
        kept = out != t0
        bits = O.unpack_bits(O.mask_bits(O.config(seed=77, step=j), O.tensor(5, n, keep_prob=np.float32(1 - p))), n)
        assert np.array_equal(kept, bits.astype(bool)), j
        assert abs(kept.sum() - n * (1 - p)) < 5 * math.sqrt(n * p * (1 - p))
    d0, _ = O.merge(O.MERGE_DARE_TA, t0, ex, gamma=0.7, p_drop=0.0, seed=1)
    ta, _ = O.merge(O.MERGE_TA, t0, ex, gamma=0.7)
    assert np.array_equal(d0, ta)
    m = 600
    small = [e[:64] for e in ex]
    mean = np.mean([O.merge(O.MERGE_DARE_TA, t0[:64], small, gamma=1.0, p_drop=0.5, seed=s)[0].astype(np.float64)
                    for s in range(m)], axis=0)
    target = O.merge(O.MERGE_TA, t0[:64], small, gamma=1.0)[0].astype(np.float64)
    spread = np.sqrt(sum((e[:64].astype(np.float64) - t0[:64]) ** 2 for e in ex) / m)  # sd of the mean, p = 0.5
    assert np.all(np.abs(mean - target) < 5 * spread + 1e-6)


def test_merge_ties_hand_example():
    """TIES (Yadav et al.): trim, elect sign, disjoint mean, worked by hand.
    Delta_1 = (1, -2, 3, 0.5), Delta_2 = (2, 1, -1, -0.5), Delta_3 = (-4, 1, -1,
    0.5). No trimming: sums (-1, 0, 1, 0.5), merged (-4, 0, 3, 0.5). Retention
    0.5 (r = 2 of 4): thresholds 2, 1, 1 (ties kept: Delta_2 keeps 2, 1, -1),
    trimmed sums (-2, 0, 1, 0), merged (-4, 0, 3, 0)."""
    t0 = np.zeros(4, np.float32)
    ex = [np.array([1, -2, 3, 0.5], np.float32), np.array([2, 1, -1, -0.5], np.float32),
          np.array([-4, 1, -1, 0.5], np.float32)]
    out, _ = O.merge(O.MERGE_TIES, t0, ex, gamma=1.0, retention=1.0)
    assert np.array_equal(out, np.array([-4, 0, 3, 0.5], np.float32))
    out, thr = O.merge(O.MERGE_TIES, t0, ex, gamma=1.0, retention=0.5)
    assert np.array_equal(out, np.array([-4, 0, 3, 0], np.float32))
    assert np.array_equal(thr.view(np.float32), np.array([2, 1, 1], np.float32))
    out, _ = O.merge(O.MERGE_TIES, t0 + np.float32(0.25), [e + np.float32(0.25) for e in ex], gamma=0.5,
                     retention=1.0)
    assert np.array_equal(out, np.array([-1.75, 0.25, 1.75, 0.5], np.float32))


def test_merge_ties_threshold_is_the_rth_largest_magnitude():
    """The trim threshold equals the ceil(k n)-th largest |Delta| of numpy's
    sort, and exactly the entries at or above it survive."""
    r = rng(32)
    n, K = 1001, 3
    t0 = (r.standard_normal(n) * 0.02).astype(np.float32)
    ex = [(t0 + r.standard_normal(n).astype(np.float32) * np.float32(1e-3)).astype(np.float32) for _ in range(K)]
    for k in (0.1, 0.3, 0.5, 1.0):
        _, thr = O.merge(O.MERGE_TIES, t0, ex, retention=k)
        for j in range(K):
            d = np.abs(ex[j] - t0)
            ref = np.sort(d)[::-1][min(n, max(1, math.ceil(k * n))) - 1]
            assert thr.view(np.float32)[j] == ref


def test_merge_ties_degenerate_cases():
    """TIES reduces to simpler merges in degenerate cases. One expert with no
    trimming is TA with that expert: its own sign is elected and the mean of
    one value is that value. Four identical experts give the same, exactly,
    since 4 Delta and 4 Delta / 4 are exact in fp32. Two opposite experts
    cancel: the sum is 0, no sign is elected and theta0 is kept. A NaN Delta
    makes the elected sum NaN, so theta0 is kept. A +inf among positive
    Deltas elects + and the mean is +inf."""
    r = rng(33)
    n = 513
    t0 = _dyadic(r, n)
    x = _dyadic(r, n)
    ta, _ = O.merge(O.MERGE_TA, t0, [x], gamma=0.5)
    one, _ = O.merge(O.MERGE_TIES, t0, [x], gamma=0.5, retention=1.0)
    assert np.array_equal(one.view(np.uint32), ta.view(np.uint32))
    four, _ = O.merge(O.MERGE_TIES, t0, [x] * 4, gamma=0.5, retention=1.0)
    assert np.array_equal(four.view(np.uint32), ta.view(np.uint32))
    z = np.zeros(n, np.float32)
    cancel, _ = O.merge(O.MERGE_TIES, z, [x, -x], gamma=0.5, retention=1.0)
    assert np.array_equal(cancel.view(np.uint32), z.view(np.uint32))
    z4 = np.zeros(4, np.float32)
    nan = np.array([np.nan, 1, 1, 1], np.float32)
    out, _ = O.merge(O.MERGE_TIES, z4, [nan, np.ones(4, np.float32)], gamma=0.5, retention=1.0)
    assert np.array_equal(out, np.array([0, 0.5, 0.5, 0.5], np.float32))
    inf = np.array([np.inf, 2, 2, 2], np.float32)
    out, _ = O.merge(O.MERGE_TIES, z4, [inf, np.ones(4, np.float32)], gamma=0.5, retention=1.0)
    assert np.array_equal(out, np.array([np.inf, 0.75, 0.75, 0.75], np.float32))


# ------------------------------------------------------- 16-bit draw option ---

def _draw16(words4, gidx):
    """Element gidx's 16-bit draw from the four words of block gidx >> 3:
    half gidx & 1 (low half first) of word (gidx & 7) >> 1."""
    w = int(words4[(gidx & 7) >> 1])
    return (w >> 16) if gidx & 1 else (w & 0xFFFF)


def test_draw16_layout_matches_triton_library():
    """The 16-bit draw option (draw_bits = 16, the 16-bit layout of the
    hot-path contract): element gidx's draw in the MASK, NOISE and ALPHA_E
    streams is half gidx & 1 (low half first) of word (gidx & 7) >> 1 of
    Triton's Philox block j = gidx >> 3 of that stream. Checked through the
    oracle's outputs: the keep bits (kept iff the draw is below floor(p 2^16)),
    uniform noise (eps / (sqrt3 sigma) = (2D + 1 - 2^16) 2^-16) and per-element
    alpha ((alpha - alpha_min) / (alpha_max - alpha_min) = D 2^-16), each up to
    fp32 rounding; element offsets with block indices at and above 2^32."""
    seed, step, tid, p, sigma, amin, amax = 0x5EED5EED12345678, 9, 0x0345678, 0.37, 1e-3, 0.2, 0.9
    cases = [(0, 40), (5, 11), ((1 << 35) - 7, 16), (5 << 35, 8)]
    need = sorted({(s, (off + i) >> 3) for s in (0, 1, 2) for off, n in cases for i in range(n)})
    assert any(j >> 32 for _, j in need)
    words = _triton_philox([[j & 0xFFFFFFFF, j >> 32, (s << 28) | tid, step] for s, j in need],
                           [seed] * len(need), 10)
    W = {key: words[k] for k, key in enumerate(need)}
    T16 = math.floor(p * 65536)
    for off, n in cases:
        gid = [off + i for i in range(n)]
        cfg = O.config(seed=seed, step=step, draw_bits=16, noise=O.NOISE_UNIFORM)
        t = O.tensor(tid, n, keep_prob=p, elem_offset=off)
        kept = O.unpack_bits(O.mask_bits(cfg, t), n).astype(bool)
        assert np.array_equal(kept, [_draw16(W[(0, g >> 3)], g) < T16 for g in gid]), off
        # every coordinate dropped and theta0 = 0: theta~ = eps
        t0 = O.tensor(tid, n, keep_prob=0.0, sigma=sigma, elem_offset=off)
        z = np.zeros(n, np.float32)
        eps = O.simulate(cfg, t0, z, z).astype(np.float64) / (math.sqrt(3.0) * float(np.float32(sigma)))
        v = np.array([(2 * _draw16(W[(1, g >> 3)], g) + 1 - 65536) * 2.0**-16 for g in gid])
        assert np.all(np.abs(eps - v) <= 4e-7 * np.abs(v)), (off, np.max(np.abs(eps - v)))
        v_nb = np.array([(2 * _draw16(W[(1, (g ^ 1) >> 3)], g ^ 1) + 1 - 65536) * 2.0**-16 for g in gid])
        assert np.mean(np.abs(eps - v_nb) <= 4e-7 * np.abs(v_nb)) < 0.2
        # the threshold itself: p = D_k / 2^16 (exact in fp32) drops element k
        # (the compare is strict) and keeps every draw below D_k
        dk = _draw16(W[(0, gid[3] >> 3)], gid[3])
        te = O.tensor(tid, n, keep_prob=float(np.float32(dk / 65536)), elem_offset=off)
        ke = O.unpack_bits(O.mask_bits(cfg, te), n).astype(bool)
        assert not ke[3]
        assert np.array_equal(ke, [_draw16(W[(0, g >> 3)], g) < dk for g in gid])
        assert O.unpack_bits(O.mask_bits(cfg, O.tensor(tid, n, keep_prob=1.0, elem_offset=off)), n).all()
        cfa = O.config(seed=seed, step=step, draw_bits=16, alpha_mode=O.ALPHA_PER_ELEMENT,
                       alpha_min=amin, alpha_max=amax)
        back = (_alpha_per_element(cfa, tid, n, elem_offset=off) - amin) / (amax - amin)
        d = np.array([_draw16(W[(2, g >> 3)], g) * 2.0**-16 for g in gid])
        assert np.all(np.abs(back - d) <= 2.0**-22), (off, np.max(np.abs(back - d)))


@pytest.mark.parametrize("p", [0.3, 0.25, 0.9])
def test_draw16_keep_rate_and_gradient_support(p):
    """16-bit draws: the keep rate is floor(p 2^16) / 2^16 (a binomial 5-sigma
    bound over 2^18 coordinates), the 32-bit layout's keep decisions are a
    different, independent draw, and the gradient map (Eq. smat-gradient) is
    zero exactly on the dropped coordinates."""
    n = 1 << 18
    cfg16 = O.config(seed=41, step=2, draw_bits=16)
    t = O.tensor(77, n, keep_prob=p)
    k16 = O.unpack_bits(O.mask_bits(cfg16, t), n).astype(bool)
    q = math.floor(p * 65536) / 65536
    assert abs(k16.mean() - q) < 5 * math.sqrt(q * (1 - q) / n)
    k32 = O.unpack_bits(O.mask_bits(O.config(seed=41, step=2), t), n).astype(bool)
    agree = np.mean(k16 == k32)
    assert abs(agree - (q * q + (1 - q) * (1 - q))) < 5 * math.sqrt(0.25 / n)
    g = O.gradmap(cfg16, t, np.ones(n, np.float32))
    assert np.array_equal(g != 0, k16)


def test_draw16_gaussian_and_alpha_laws():
    """16-bit draws: Gaussian Perturb is N(0, sigma^2) up to the 2^-16 grid
    (KS against N(0, 1), unit variance, symmetric, |z| at most
    sqrt2 erfinv(1 - 2^-16)); per-element alpha is U[alpha_min, alpha_max)
    (KS) and independent of the neighbouring coordinate."""
    from scipy.special import erfinv as sp_erfinv
    n, sigma = 200_000, 1e-4
    t = O.tensor(8, n, keep_prob=0.0, sigma=sigma)
    z = np.zeros(n, np.float32)
    eps = O.simulate(O.config(seed=6, noise=O.NOISE_GAUSSIAN, draw_bits=16), t, z, z).astype(np.float64) / sigma
    assert stats.kstest(eps, "norm").pvalue > 1e-4
    assert abs(eps.var() - 1) < 5 * math.sqrt(2.0 / n)
    assert abs(eps.mean()) < 5 / math.sqrt(n)
    assert np.max(np.abs(eps)) <= math.sqrt(2.0) * sp_erfinv(1 - 2.0**-16) * (1 + 1e-6)
    eps32 = O.simulate(O.config(seed=6, noise=O.NOISE_GAUSSIAN), t, z, z).astype(np.float64) / sigma
    assert abs(np.corrcoef(eps, eps32)[0, 1]) < 5 / math.sqrt(n)
    amin, amax = 0.3, 0.8
    cfa = O.config(seed=32, step=1, draw_bits=16, alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=amin, alpha_max=amax)
    a = _alpha_per_element(cfa, 90, n)
    assert np.all((a >= amin) & (a < amax))
    assert stats.kstest((a - amin) / (amax - amin), "uniform").pvalue > 1e-4
    assert abs(np.corrcoef(a[:-1], a[1:])[0, 1]) < 5 / math.sqrt(n)


# ------------------------------------- gradient map fused with AdamW (Sec. 4.3) ---

def test_gradmap_adamw_matches_torch_adamw_on_the_mapped_gradient():
    """The fused step equals torch.optim.AdamW (a library routine, float64)
    applied with the gradient the gradient map stores (Eq. smat-gradient:
    alpha m (.) g~, dropped coordinates 0), step after step, within fp32
    rounding; moments likewise. Per-element alpha, a Mask, weight decay, bf16
    gradients."""
    n, steps = 4096, 5
    lr, b1, b2, eps, wd = 1e-3, 0.9, 0.95, 1e-8, 0.1
    rg = rng(70)
    t = O.tensor(12, n, dtype=O.F32, keep_prob=0.7)
    th = (rg.standard_normal(n) * 0.02).astype(np.float32)
    m1 = np.zeros(n, np.float32)
    m2 = np.zeros(n, np.float32)
    p = torch.tensor(th.astype(np.float64), requires_grad=True)
    f = lambda v: float(np.float32(v))  # noqa: E731  (the hyperparameters cross the ABI as fp32)
    opt = torch.optim.AdamW([p], lr=f(lr), betas=(f(b1), f(b2)), eps=f(eps), weight_decay=f(wd))
    for k in range(1, steps + 1):
        cfg = O.config(seed=8, step=10 + k, alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=0.3)
        gs = O.f32_to_bf16((rg.standard_normal(n) * 0.5).astype(np.float32))
        g = O.bf16_to_f32(O.gradmap(cfg, t, gs, gdtype=O.BF16)).astype(np.float64)
        th, m1, m2 = O.gradmap_adamw(cfg, t, gs, th, m1, m2, lr, b1, b2, eps, wd, adam_step=k, gdtype=O.BF16)
        p.grad = torch.tensor(g)
        opt.step()
        st = opt.state[p]
        ref = p.detach().numpy()
        # fp32 rounding, step after step: m1 may cancel towards 0 (an absolute
        # floor at fp32 resolution of its terms), m2 is a sum of positives
        assert np.allclose(m1, st["exp_avg"].numpy(), rtol=2e-6, atol=1e-7), k
        assert np.allclose(m2, st["exp_avg_sq"].numpy(), rtol=1e-6, atol=0), k
        # theta: a few fp32 ulps of theta per step, and of the update near 0
        assert np.all(np.abs(th.astype(np.float64) - ref) <= 2e-6 * np.abs(ref) + 5e-5 * lr), k


def test_gradmap_adamw_first_step_and_weight_decay_closed_forms():
    """Step 1 from zero moments without weight decay moves each coordinate by
    -lr g / (|g| + eps) (the bias corrections cancel); with g~ = 0 the step is
    the decoupled decay theta (1 - lr wd) alone and the moments stay 0."""
    n, lr, eps = 2048, 3e-4, 1e-8
    rg = rng(71)
    t = O.tensor(13, n, dtype=O.F32, keep_prob=1.0)
    cfg = O.config(seed=9, step=1, alpha_mode=O.ALPHA_GLOBAL, alpha_min=1.0, alpha_max=1.0)  # alpha = 1: g = g~
    th = (rg.standard_normal(n) * 0.02).astype(np.float32)
    gs = (rg.standard_normal(n)).astype(np.float32)
    z = np.zeros(n, np.float32)
    b1, b2 = 0.875, 0.984375  # exact in fp32
    th1, m1, m2 = O.gradmap_adamw(cfg, t, gs, th, z, z, lr, b1, b2, eps, 0.0, adam_step=1)
    g = gs.astype(np.float64)
    exp = th.astype(np.float64) - np.float64(np.float32(lr)) * g / (np.abs(g) + eps)
    assert np.all(np.abs(th1 - exp) <= 2e-7 * np.abs(exp) + 1e-6 * lr)
    assert np.allclose(m1, (1 - b1) * g, rtol=1e-7) and np.allclose(m2, (1 - b2) * g * g, rtol=3e-7)
    wd = 0.05
    th2, a, b = O.gradmap_adamw(cfg, t, z, th, z, z, lr, 0.9, 0.999, eps, wd, adam_step=3)
    assert np.array_equal(th2, th * np.float32(1.0 - lr * wd))
    assert not a.any() and not b.any()


@pytest.mark.parametrize("dtype,gdtype", [(O.BF16, O.BF16), (O.F32, O.F32), (O.BF16, O.F32)])
def test_gradmap_adamw_at_equals_the_whole_tensor(dtype, gdtype):
    """The sampled form (which the full-size GPU check uses) equals the
    whole-tensor form at every sampled index: per-element alpha, a keep rate
    just above a tie boundary, an element offset above 2^33, warm moments."""
    n = 5000
    rg = rng(83)
    t = O.tensor(21, n, dtype=dtype, keep_prob=0.5 + 2**-10, elem_offset=2**33 + 7)
    cfg = O.config(seed=4, step=6, alpha_mode=O.ALPHA_PER_ELEMENT, alpha_min=0.2)
    th32 = (rg.standard_normal(n) * 0.02).astype(np.float32)
    gs32 = rg.standard_normal(n).astype(np.float32)
    th = O.f32_to_bf16(th32) if dtype == O.BF16 else th32
    gs = O.f32_to_bf16(gs32) if gdtype == O.BF16 else gs32
    m1 = (rg.standard_normal(n) * 1e-3).astype(np.float32)
    m2 = (rg.random(n) * 1e-6).astype(np.float32)
    hp = dict(lr=1e-3, weight_decay=0.01, adam_step=4, gdtype=gdtype)
    th_all, m1_all, m2_all = O.gradmap_adamw(cfg, t, gs, th, m1, m2, **hp)
    idx = np.sort(rg.choice(n, 700, replace=False))
    thv = O.bf16_to_f32(th[idx]) if dtype == O.BF16 else th[idx]
    gv = O.bf16_to_f32(gs[idx]) if gdtype == O.BF16 else gs[idx]
    bits, a, b = O.gradmap_adamw_at(cfg, t, idx, gv, thv, m1[idx], m2[idx], **hp)
    ref = th_all[idx].view(np.uint16).astype(np.uint32) if dtype == O.BF16 else th_all[idx].view(np.uint32)
    assert np.array_equal(bits, ref)
    assert np.array_equal(a.view(np.uint32), m1_all[idx].view(np.uint32))
    assert np.array_equal(b.view(np.uint32), m2_all[idx].view(np.uint32))
