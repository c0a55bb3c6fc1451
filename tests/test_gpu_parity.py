"""GPU parity: the CUDA path through the C ABI against the CPU oracle, element
by element, on seeded inputs spanning several chunks and ragged tails.
Tolerances are those of tests/_parity.py (bit-exact masks and gradient map;
bit-exact uniform-noise forward; Gaussian forward within 1e-6 relative in fp32
and 1 ulp in bf16)."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300 import workloads as W

from _parity import compare, f32_of, orc_config, orc_tensor, run_and_check_full, session_for, to_host

pytestmark = pytest.mark.gpu

@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    yield
    torch.cuda.synchronize()


# ------------------------------------------------------------------ Philox ---

@pytest.mark.parametrize("rounds", [10, 7])
def test_device_philox_matches_oracle_and_curand(rounds):
    g = torch.Generator().manual_seed(3)
    n = 4096
    ctr = torch.randint(-2**31, 2**31 - 1, (n, 4), generator=g, dtype=torch.int64).to(torch.int32)
    ctr[0] = 0
    ctr[1] = -1
    for seed in (0, 0x0123456789ABCDEF, 2**64 - 1):
        out, ref = S.debug_philox(ctr.cuda(), seed, rounds, with_curand=(rounds == 10))
        out = out.cpu().numpy().view(np.uint32)
        c = ctr.numpy().view(np.uint32)
        for i in list(range(64)) + list(range(n - 8, n)):
            exp = O.philox(c[i], [seed & 0xFFFFFFFF, seed >> 32], rounds)
            assert np.array_equal(out[i], exp), (seed, i)
        if ref is not None:
            assert np.array_equal(out, ref.cpu().numpy().view(np.uint32)), "cuRAND curand_Philox4x32_10 differs"


# ---------------------------------------------------------- whole workloads ---

def test_tiny_flat_f32_gaussian_steps_0_1_2():
    """1 Mi fp32 tensor, Gaussian eps, per-tensor alpha, p_keep 0.9: forward
    within 1e-6 relative, gradient map and masks exact, three steps."""
    run_and_check_full(W.tiny_flat())


@pytest.mark.parametrize("name", ["dec_0p5b", "llama_7b", "vl_7b"])
def test_scaled_backbone_lists(name):
    """Every tensor of the list (shapes cut to ~3M elements total, ragged)."""
    w = W.scaled(W.WORKLOADS[name](), 3_000_000)
    run_and_check_full(w, steps=(0, 2))


@pytest.mark.parametrize("noise", [O.NOISE_UNIFORM, O.NOISE_GAUSSIAN, O.NOISE_LAPLACE])
@pytest.mark.parametrize("alpha_mode", [O.ALPHA_GLOBAL, O.ALPHA_PER_TENSOR, O.ALPHA_PER_ELEMENT])
@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_modes_small_ragged_list(dtype, alpha_mode, noise):
    # work chunks are 2^18 elements (gradient-map units 2^17): sizes around both
    sizes = [0, 1, 3, 15, 16, 17, 31, 33, 255, 131_073, 262_144, 262_145, 600_003]
    keeps = [0.5, 0.9, 0.1, 0.7, 1.0, 0.0, 0.3, 0.5, 0.7, 0.9, 0.3, 0.5 + 2**-10, 0.7]
    specs = [W.TensorSpec(f"t{i}", (n,), "linear", keeps[i], 2e-3 if i % 4 else 0.0) for i, n in enumerate(sizes)]
    w = W.Workload(f"ragged_{dtype}_{alpha_mode}_{noise}", specs, dtype, dtype, 0.2, 1.0, alpha_mode, noise, 0.02, 1e-3,
                   seed=0x1234_5678_9ABC)
    run_and_check_full(w, steps=(0, 7))


@pytest.mark.parametrize("chunk_log2", [12, 16, 18])
@pytest.mark.parametrize("noise", [O.NOISE_UNIFORM, O.NOISE_GAUSSIAN, O.NOISE_LAPLACE])
def test_forced_chunk_sizes_ragged_list(chunk_log2, noise):
    """The work-chunk size (chosen per list; forced here) changes no result:
    ragged tensors around 2^12, 2^16, 2^17 (gradient-map unit) and 2^18
    boundaries, bf16, elementwise against the oracle."""
    sizes = [5, 4096, 4097, 65_536 + 17, 131_072, 262_144, 262_161, 600_003, 33]
    keeps = [0.7, 0.5, 0.3, 0.7, 0.9, 0.1, 0.7, 0.5 + 2**-10, 1.0]
    specs = [W.TensorSpec(f"t{i}", (n,), "linear", keeps[i], 2e-3 if i % 3 else 0.0) for i, n in enumerate(sizes)]
    w = W.Workload(f"chunks_{chunk_log2}_{noise}", specs, O.BF16, O.BF16, 0.3, 1.0, O.ALPHA_PER_TENSOR, noise, 0.02,
                   1e-3, seed=0x5EED_0018)
    run_and_check_full(w, steps=(0, 3), flags=S.SMAT_FLAG_CHUNK_LOG2(chunk_log2))


def test_philox_7_rounds_and_accumulate_and_f32_grads_on_bf16_params():
    specs = [W.TensorSpec("a", (70_001,), "linear", 0.7, 1e-3), W.TensorSpec("b", (9,), "other", 1.0, 1e-3)]
    w = W.Workload("r7", specs, O.BF16, O.BF16, 0.3, 1.0, 1, O.NOISE_UNIFORM, 0.02, 1e-3, seed=5)
    run_and_check_full(w, steps=(1,), rounds=7, accumulate=True, gdtype=O.F32)


@pytest.mark.parametrize("sig", [0.0, 1e-4])
@pytest.mark.parametrize("am", [O.ALPHA_PER_TENSOR, O.ALPHA_PER_ELEMENT])
@pytest.mark.parametrize("dt", [O.F32, O.BF16])
def test_sweep_grid_at_2_16(dt, am, sig):
    """Every setting of the flat-tensor sweep (2 dtypes x 5 keep probabilities
    x alpha per tensor or per element, U[0, 1) x sigma 0 or 1e-4, Gaussian) on
    a 2^16-element tensor, element by element."""
    for p in (0.1, 0.3, 0.5, 0.7, 0.9):
        run_and_check_full(W.flat_sweep(16, dt, p, am, sig), steps=(0,))


def test_sweep_points_2_18_and_2_20_small_chunks():
    """Larger sweep points: 2^18 in both dtypes; 2^20 fp32 with per-element
    alpha and noise on 2^12-element work chunks (256 chunks, each its own
    rare-element queue)."""
    for dt in (O.F32, O.BF16):
        for p, am, sig in ((0.1, 1, 0.0), (0.5, 2, 1e-4), (0.9, 1, 1e-4), (0.3, 2, 0.0)):
            run_and_check_full(W.flat_sweep(18, dt, p, am, sig), steps=(0,))
    run_and_check_full(W.flat_sweep(20, O.F32, 0.7, O.ALPHA_PER_ELEMENT, 1e-4), steps=(0, 1),
                       flags=S.SMAT_FLAG_CHUNK_LOG2(12))


# ------------------------------------------------------------------ edges ---

def _one(n, dtype=torch.bfloat16, keep=0.5, sigma=1e-3, offset_elems=0, elem_offset=0, noise=O.NOISE_UNIFORM,
         amin=0.2, amax=1.0, pad=0):
    """A single tensor, optionally starting offset_elems into a larger buffer
    (breaking 32-byte alignment) and with guard padding after it."""
    dev = torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(n + offset_elems)
    tot = n + offset_elems + pad
    base0 = (torch.randn(tot, generator=g, device=dev) * 0.02).to(dtype)
    base1 = (base0.float() + torch.randn(tot, generator=g, device=dev) * 1e-3).to(dtype)
    simbuf = torch.full((tot,), 7.0, dtype=dtype, device=dev)
    th = base1[offset_elems:offset_elems + n]
    t0 = base0[offset_elems:offset_elems + n]
    sim = simbuf[offset_elems:offset_elems + n]
    sess = S.SmatSession([th], [t0], [sim], [keep], [sigma], elem_offsets=[elem_offset], seed=9, alpha_min=amin,
                         alpha_max=amax, alpha_mode=S.SMAT_ALPHA_PER_TENSOR, noise=noise)
    return sess, th, t0, sim, simbuf


@pytest.mark.parametrize("offset_elems", [1, 3, 8, 16])
@pytest.mark.parametrize("elem_offset", [0, 5, 16, 2**36 + 3])
def test_misaligned_and_offset_tensors_take_the_element_path(offset_elems, elem_offset):
    n = 5003
    sess, th, t0, sim, simbuf = _one(n, offset_elems=offset_elems, elem_offset=elem_offset, pad=64)
    sess.simulate_multi(3)
    torch.cuda.synchronize()
    cfg = O.config(seed=9, step=3, alpha_mode=O.ALPHA_PER_TENSOR, noise=O.NOISE_UNIFORM, alpha_min=0.2)
    t = O.tensor(0, n, O.BF16, keep_prob=0.5, sigma=1e-3, elem_offset=elem_offset)
    ref = O.simulate(cfg, t, to_host(th), to_host(t0))
    compare(to_host(sim), ref, O.BF16, O.NOISE_UNIFORM, what="misaligned")
    sb = to_host(simbuf)
    assert np.all(sb[:offset_elems] == to_host(torch.tensor([7.0], dtype=torch.bfloat16))[0])
    assert np.all(sb[offset_elems + n:] == to_host(torch.tensor([7.0], dtype=torch.bfloat16))[0])
    bits = sess.mask_bits(3, 0).cpu().numpy().view(np.uint32)
    assert np.array_equal(bits, O.mask_bits(cfg, t))


def test_guard_canaries_around_every_output():
    """Outputs stay inside their tensors: guard bytes after each sim / grad
    buffer keep their sentinel."""
    dev = torch.device("cuda")
    sizes = [17, 4096, 65537, 131072 + 5]
    pad = 128
    th, t0, simbufs, sims, gs, gobufs, gos = [], [], [], [], [], [], []
    for n in sizes:
        th.append((torch.randn(n, device=dev) * 0.02).to(torch.bfloat16))
        t0.append((torch.randn(n, device=dev) * 0.02).to(torch.bfloat16))
        sb = torch.full((n + pad,), -3.0, dtype=torch.bfloat16, device=dev)
        simbufs.append(sb)
        sims.append(sb[:n])
        gs.append(torch.randn(n, device=dev).to(torch.bfloat16))
        gb = torch.full((n + pad,), -5.0, dtype=torch.bfloat16, device=dev)
        gobufs.append(gb)
        gos.append(gb[:n])
    sess = S.SmatSession(th, t0, sims, [0.7] * 4, [1e-3] * 4, seed=1, alpha_mode=S.SMAT_ALPHA_PER_ELEMENT,
                         noise=S.SMAT_NOISE_GAUSSIAN)
    sess.simulate_multi(0)
    sess.grad_map_multi(0, gs, gos)
    torch.cuda.synchronize()
    for n, sb, gb in zip(sizes, simbufs, gobufs):
        assert torch.all(sb[n:] == -3.0)
        assert torch.all(gb[n:] == -5.0)


def test_identity_and_all_dropped_on_gpu():
    n = 70_000
    sess, th, t0, sim, _ = _one(n, keep=1.0, sigma=0.0, amin=1.0, amax=1.0)
    sess.simulate_multi(0)
    torch.cuda.synchronize()
    assert np.array_equal(to_host(sim), to_host(th))
    sess, th, t0, sim, _ = _one(n, keep=0.0, sigma=0.0)
    sess.simulate_multi(0)
    torch.cuda.synchronize()
    assert np.array_equal(to_host(sim), to_host(t0))


def test_shard_invariance_on_gpu():
    """Two halves with elem_offset give the bits of the whole tensor."""
    dev = torch.device("cuda")
    n, split = 300_017, 123_456
    th = (torch.randn(n, device=dev) * 0.02).to(torch.bfloat16)
    t0 = (torch.randn(n, device=dev) * 0.02).to(torch.bfloat16)
    full = torch.empty_like(th)
    a = torch.empty(split, dtype=torch.bfloat16, device=dev)
    b = torch.empty(n - split, dtype=torch.bfloat16, device=dev)
    kw = dict(seed=4, alpha_mode=S.SMAT_ALPHA_PER_ELEMENT, noise=S.SMAT_NOISE_GAUSSIAN)
    S.SmatSession([th], [t0], [full], [0.6], [1e-3], tensor_ids=[5], **kw).simulate_multi(2)
    # tensor ids are unique within a context, so each half is its own context with the same id
    S.SmatSession([th[:split].contiguous()], [t0[:split].contiguous()], [a], [0.6], [1e-3], tensor_ids=[5],
                  elem_offsets=[0], **kw).simulate_multi(2)
    S.SmatSession([th[split:].contiguous()], [t0[split:].contiguous()], [b], [0.6], [1e-3], tensor_ids=[5],
                  elem_offsets=[split], **kw).simulate_multi(2)
    torch.cuda.synchronize()
    assert torch.equal(torch.cat([a, b]).view(torch.int16), full.view(torch.int16))


def test_tensor_order_and_grouping_invariance():
    """Results depend on each tensor's id, not on its position in the list or
    on which other tensors share the launch: the list in reverse order, and
    split into two contexts, give the same bits (forward, with sigma_rel
    statistics fused, and gradient map)."""
    dev = torch.device("cuda")
    sizes = [70_001, 262_144 + 7, 17, 300_000, 4096]
    th = [(torch.randn(n, device=dev) * 0.02).to(torch.bfloat16) for n in sizes]
    t0 = [(x.float() + torch.randn(x.numel(), device=dev) * 1e-3).to(torch.bfloat16) for x in th]
    gs = [torch.randn(n, device=dev).to(torch.bfloat16) for n in sizes]
    keeps = [0.7, 0.5, 1.0, 0.3, 0.9]
    sig = [1e-3, 0.0, 2e-3, 0.0, 1e-3]
    rel = [0.0, 0.1, 0.0, 0.1, 0.0]
    kw = dict(seed=21, alpha_min=0.3, alpha_mode=S.SMAT_ALPHA_PER_TENSOR, noise=S.SMAT_NOISE_GAUSSIAN)

    def run(order_groups):
        sims = [torch.empty_like(x) for x in th]
        gos = [torch.empty_like(g) for g in gs]
        for idx in order_groups:
            s = S.SmatSession([th[i] for i in idx], [t0[i] for i in idx], [sims[i] for i in idx],
                              [keeps[i] for i in idx], [sig[i] for i in idx], [rel[i] for i in idx],
                              tensor_ids=[100 + i for i in idx], **kw)
            s.simulate_multi(3)
            s.swap()
            s.grad_map_multi(3, [gs[i] for i in idx], [gos[i] for i in idx])
            s.swap()
            assert s.poll_errors() == 0
        torch.cuda.synchronize()
        return sims, gos

    ref = run([[0, 1, 2, 3, 4]])
    for groups in ([[4, 3, 2, 1, 0]], [[3, 0], [4, 2, 1]]):
        got = run(groups)
        for a, b in zip(ref[0] + ref[1], got[0] + got[1]):
            assert torch.equal(a.view(torch.int16), b.view(torch.int16)), groups


def test_inplace_gradient_map():
    dev = torch.device("cuda")
    n = 100_003
    sess, th, t0, sim, _ = _one(n, keep=0.7)
    g = torch.randn(n, device=dev).to(torch.bfloat16)
    g0 = to_host(g)
    sess.simulate_multi(4)
    sess.grad_map_multi(4, [g], [g])
    torch.cuda.synchronize()
    cfg = O.config(seed=9, step=4, alpha_mode=O.ALPHA_PER_TENSOR, noise=O.NOISE_UNIFORM, alpha_min=0.2)
    ref = O.gradmap(cfg, O.tensor(0, n, O.BF16, keep_prob=0.7, sigma=1e-3), g0, gdtype=O.BF16)
    assert np.array_equal(to_host(g), ref)


def test_gradient_map_needs_the_forward_of_its_step():
    """The gradient map regenerates the mask of the forward that produced
    theta~ (Eq. smat-gradient; App. D): a map for a step that no forward on
    this context ran, or for an earlier forward's step, is refused with
    SMAT_ERR_STATE before any device work, and g_out stays untouched."""
    n = 5000
    sess, th, t0, sim, _ = _one(n, keep=0.7)
    dev = torch.device("cuda")
    g = torch.randn(n, device=dev).to(torch.bfloat16)
    go = torch.full((n,), 7.0, dtype=torch.bfloat16, device=dev)
    for bad in (0, 3):
        with pytest.raises(S.SmatError) as e:
            sess.grad_map_multi(bad, [g], [go])  # no forward yet
        assert e.value.status == "SMAT_ERR_STATE"
    sess.simulate_multi(3)
    with pytest.raises(S.SmatError) as e:
        sess.grad_map_multi(2, [g], [go])
    assert e.value.status == "SMAT_ERR_STATE" and "step 3" in e.value.detail
    torch.cuda.synchronize()
    assert torch.all(go == 7.0)
    sess.grad_map_multi(3, [g], [go])
    sess.grad_map_multi(3, [g], [go], accumulate=True)  # accumulation over one forward
    sess.simulate_multi(4)
    with pytest.raises(S.SmatError):
        sess.grad_map_multi(3, [g], [go])
    sess.grad_map_multi(4, [g], [go])
    torch.cuda.synchronize()
    cfg = O.config(seed=9, step=4, alpha_mode=O.ALPHA_PER_TENSOR, noise=O.NOISE_UNIFORM, alpha_min=0.2)
    ref = O.gradmap(cfg, O.tensor(0, n, O.BF16, keep_prob=0.7, sigma=1e-3), to_host(g), gdtype=O.BF16)
    assert np.array_equal(to_host(go), ref)
    assert sess.poll_errors() == 0


def test_swap_state_and_errors():
    sess, th, t0, sim, _ = _one(1000)
    assert sess.active == 0
    sess.simulate_multi(0)
    assert sess.swap() == 1
    with pytest.raises(S.SmatError) as e:
        sess.simulate_multi(1)
    assert "SMAT_ERR_STATE" in str(e.value)
    assert sess.swap() == 0
    sess.simulate_multi(1)
    with pytest.raises(S.SmatError):
        sess.mask_bits(0, 3)


def test_parameter_switching_toy_mlp_step():
    """Storage switching (Sec. 4.3) on a 2-layer MLP: forward/backward read
    theta~ after swap(); the mapped gradient equals alpha m (.) grad at theta~
    (Eq. smat-gradient, oracle); the optimizer sees the original storage."""
    dev = torch.device("cuda")
    torch.manual_seed(0)
    model = torch.nn.Sequential(torch.nn.Linear(64, 128), torch.nn.GELU(), torch.nn.Linear(128, 8)).to(dev)
    params = list(model.parameters())
    theta0 = [p.detach().clone() for p in params]
    with torch.no_grad():
        for p in params:
            p.add_(torch.randn_like(p) * 1e-2)
    theta_before = [p.detach().clone() for p in params]
    keeps = [0.5 if p.dim() == 2 else 1.0 for p in params]
    sp = S.SmatParameters(params, theta0, keeps, [2e-3] * len(params), seed=3, alpha_min=0.2,
                          alpha_mode=S.SMAT_ALPHA_GLOBAL, noise=S.SMAT_NOISE_UNIFORM)
    step = 6
    sp.simulate(step)
    assert sp.swap() == 1
    for p, s in zip(params, sp.sims):
        assert p.data.data_ptr() == s.data_ptr()
    x = torch.randn(32, 64, device=dev)
    loss = model(x).square().mean()
    loss.backward()
    g_sim = [p.grad.detach().clone() for p in params]
    sp.grad_map(step)
    assert sp.swap() == 0
    torch.cuda.synchronize()
    cfg = O.config(seed=3, step=step, alpha_mode=O.ALPHA_GLOBAL, noise=O.NOISE_UNIFORM, alpha_min=0.2)
    for k, p in enumerate(params):
        assert p.data.data_ptr() == sp.theta[k].data_ptr()
        assert torch.equal(p.data, theta_before[k])
        t = O.tensor(k, p.numel(), O.F32, keep_prob=keeps[k], sigma=2e-3)
        ref = O.gradmap(cfg, t, to_host(g_sim[k]).ravel())
        assert np.array_equal(to_host(p.grad).ravel().view(np.uint32), ref.view(np.uint32))
        sim_ref = O.simulate(cfg, t, to_host(theta_before[k]).ravel(), to_host(theta0[k]).ravel())
        assert np.array_equal(to_host(sp.sims[k]).ravel().view(np.uint32), sim_ref.view(np.uint32))
    torch.optim.SGD(params, lr=0.1).step()


def _sprinkle(x: np.ndarray, rng, dtype, frac=0.01):
    """Signed zeros, infinities, NaN, subnormals and the largest finite values
    written over a fraction of the elements (as storage bits)."""
    n = x.size
    idx = rng.choice(n, size=max(8, int(frac * n)), replace=False)
    if dtype == O.BF16:
        specials = np.array([0x0000, 0x8000, 0x7F80, 0xFF80, 0x7FC0, 0x0001, 0x8003, 0x7F7F, 0xFF7F], np.uint16)
        xv = x.view(np.uint16)
    else:
        specials = np.array([0x00000000, 0x80000000, 0x7F800000, 0xFF800000, 0x7FC00000, 0x00000001, 0x80000005,
                             0x7F7FFFFF, 0xFF7FFFFF], np.uint32)
        xv = x.view(np.uint32)
    xv[idx] = specials[rng.integers(0, len(specials), size=len(idx))]
    return x


@pytest.mark.parametrize("alpha_mode", [O.ALPHA_PER_TENSOR, O.ALPHA_PER_ELEMENT])
@pytest.mark.parametrize("noise", [O.NOISE_UNIFORM, O.NOISE_GAUSSIAN])
@pytest.mark.parametrize("dtype", [O.BF16, O.F32])
def test_special_values_in_theta_theta0_and_gradients(dtype, noise, alpha_mode):
    """Signed zeros, infinities, NaN, subnormals and the largest finite values
    in theta, theta0 and g~ (vector and element paths): the forward follows
    the same IEEE operations as the oracle (NaN wherever the oracle's is NaN;
    otherwise the usual tolerances) and the gradient map equals the oracle's
    with any NaN equal to any NaN (dropped coordinates are +0 whatever g~)."""
    rng = np.random.default_rng(1000 + 10 * dtype + noise + 100 * alpha_mode)
    dev = torch.device("cuda")
    sizes = [70_001, 4099]
    tdt = torch.bfloat16 if dtype == O.BF16 else torch.float32
    hs = []
    for n in sizes:
        t0 = (rng.standard_normal(n) * 0.02).astype(np.float32)
        th = (t0 + rng.standard_normal(n) * 1e-3).astype(np.float32)
        g = rng.standard_normal(n).astype(np.float32)
        if dtype == O.BF16:
            t0, th, g = O.f32_to_bf16(t0), O.f32_to_bf16(th), O.f32_to_bf16(g)
        hs.append((_sprinkle(th, rng, dtype), _sprinkle(t0, rng, dtype), _sprinkle(g, rng, dtype)))

    def dev_t(a):
        t = torch.from_numpy(a.view(np.int16) if dtype == O.BF16 else a).to(dev)
        return t.view(tdt)

    th = [dev_t(h[0]) for h in hs]
    t0 = [dev_t(h[1]) for h in hs]
    gs = [dev_t(h[2]) for h in hs]
    sim = [torch.empty_like(x) for x in th]
    go = [torch.empty_like(x) for x in th]
    keeps, sig = [0.7, 0.3], 2e-3
    sess = S.SmatSession(th, t0, sim, keeps, [sig, sig], seed=321, alpha_min=0.3, alpha_max=1.0,
                         alpha_mode=alpha_mode, noise=noise)
    sess.simulate_multi(2)
    sess.swap()
    sess.grad_map_multi(2, gs, go)
    sess.swap()
    torch.cuda.synchronize()
    cfg = O.config(seed=321, step=2, alpha_mode=alpha_mode, noise=noise, alpha_min=0.3, alpha_max=1.0)
    sv = np.uint16 if dtype == O.BF16 else np.uint32
    for k, n in enumerate(sizes):
        t = O.tensor(k, n, dtype=dtype, keep_prob=keeps[k], sigma=sig)
        ref = O.simulate(cfg, t, hs[k][0], hs[k][1])
        compare(to_host(sim[k]), ref.view(sv), dtype, noise, f32_of(hs[k][0]), f32_of(hs[k][1]),
                what=f"special values tensor {k}")
        gref = f32_of(O.gradmap(cfg, t, hs[k][2], gdtype=dtype))
        gg = f32_of(to_host(go[k]))
        assert np.array_equal(np.isnan(gg), np.isnan(gref)), f"tensor {k}: gradient NaN pattern"
        ok = ~np.isnan(gref)
        assert np.array_equal(gg[ok].view(np.uint32), gref[ok].view(np.uint32)), f"tensor {k}: gradient bits"
    assert sess.poll_errors() == 0
    sess.close()
