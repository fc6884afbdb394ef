"""GPU parity: the CUDA library (through its C ABI) against the CPU oracle.

Every case runs the library's kernels on seeded inputs and the oracle on the
same inputs (host generator), then compares every state of every replica
with the tolerance of ``parity_util`` (1e-5 relative, RMS floor).
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from parity_util import (TOL, compare, host_grads, oracle_run, rel_err, sample_indices,
                         state_names, workload_dict)
from synth import generators as G
from synth import workloads as W

pytestmark = pytest.mark.gpu

SEED_G, SEED_I = 1234, 5678


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2510_05361_gb300 as P
    P.load()
    return P


def to_dev(g_np, gdt):
    t = torch.from_numpy(np.ascontiguousarray(g_np)).cuda()
    return t.to(torch.bfloat16) if gdt == "bf16" else t


def gpu_run(P, w, T, fused=True, lr=None, t0=0, eng=None, x0=None):
    lay = W.layout(w["shapes"])
    n = lay["n_padded"]
    opt = w["opt"]
    lr = opt.get("lr", 1e-3) if lr is None else lr
    idx = np.arange(n)
    if eng is None:
        eng = P.MTDAO(opt, w["M"], w["shapes"])
        if x0 is None:
            x0 = G.init_params(w, lay, SEED_I, idx)
        eng.set_params(torch.from_numpy(x0).cuda())
    for t in range(t0, t0 + T):
        g = to_dev(host_grads(w, lay, SEED_G, t, idx), w["grad_dtype"])
        due = eng.sync_due()
        if fused:
            eng.step(g, lr, due)
        else:
            eng.step(g, lr, 0)
            eng.sync(due)
    torch.cuda.synchronize()
    return eng


def gpu_states(eng, opt):
    out = {}
    for s, name in enumerate(state_names(opt)):
        out[name] = eng.state_view(s).cpu().numpy()
    return out


RAGGED = [1, 7, 300, 4099, 2560, 13]


@pytest.mark.parametrize("gdt", ["f32", "bf16"])
@pytest.mark.parametrize("N", [1, 2, 3, 4])
@pytest.mark.parametrize("base", ["adam", "adopt", "sgdm"])
@pytest.mark.parametrize("M", [2, 3, 4, 5, 6, 7, 8, 12, 16, 32, 64])
def test_step_and_sync_parity_matrix(P, base, N, gdt, M):
    betas = W.SWEEP_BETAS[:N]
    w = workload_dict(RAGGED, M, base=base, betas=betas, beta2=0.9999 if base == "adopt" else 0.999,
                      px=5, pu=[3, 4, 2, 6][:N], pv=4, lr=2.0 ** -8 if base == "adopt" else 1e-3,
                      gdt=gdt)
    T = 13
    eng = gpu_run(P, w, T)
    lay = W.layout(w["shapes"])
    ref = oracle_run(w["opt"], M, np.arange(lay["n_padded"]), T, lay, w, SEED_G, SEED_I)
    compare(gpu_states(eng, w["opt"]), ref)
    eng.close()


@pytest.mark.parametrize("M", [1, 2, 5, 8])
def test_replica_counts(P, M):
    w = workload_dict([5000, 123], M, betas=(0.9, 0.999), px=4, pu=2, pv=3)
    eng = gpu_run(P, w, 9)
    lay = W.layout(w["shapes"])
    ref = oracle_run(w["opt"], M, np.arange(lay["n_padded"]), 9, lay, w, SEED_G, SEED_I)
    compare(gpu_states(eng, w["opt"]), ref)
    eng.close()


@pytest.mark.parametrize("gdt", ["f32", "bf16"])
@pytest.mark.parametrize("M", [2, 3, 4, 5, 6, 7, 8, 9, 12, 16, 17, 24, 32, 33, 64, 100, 128, 200, 256])
def test_fused_sync_is_bitwise_equal_to_separate_sync(P, M, gdt):
    for base in ("adam", "adopt", "sgdm"):
        w = workload_dict(RAGGED, M, base=base, betas=(0.9, 0.99, 0.5), px=3, pu=[2, 3, 4], pv=2,
                          beta2=0.9999 if base == "adopt" else 0.999, gdt=gdt)
        a = gpu_run(P, w, 8, fused=True)
        b = gpu_run(P, w, 8, fused=False)
        sa, sb = gpu_states(a, w["opt"]), gpu_states(b, w["opt"])
        for k in sa:
            assert np.array_equal(sa[k].view(np.uint32), sb[k].view(np.uint32)), (base, k)
        a.close()
        b.close()


@pytest.mark.parametrize("M", range(2, 71))
def test_fused_equals_separate_for_every_replica_count(P, M):
    """Every M from 2 to 70 crosses each switch between averaging paths:
    lane groups (M <= 8), the block-staged fused step (9..64; one or two
    float4 positions per thread at 16/17, four-column or one-column means at
    32/33), step + average above 64, and the standalone average in registers
    (M <= 14) or streamed.  Fused and separate averaging agree bit for bit,
    and the averaged states equal the oracle within the tolerance."""
    w = workload_dict([700, 300, 24], M, base="adam", betas=(0.9, 0.99), px=2, pu=[3, 2], pv=3, gdt="f32")
    a = gpu_run(P, w, 6, fused=True)
    b = gpu_run(P, w, 6, fused=False)
    sa, sb = gpu_states(a, w["opt"]), gpu_states(b, w["opt"])
    for k in sa:
        assert np.array_equal(sa[k].view(np.uint32), sb[k].view(np.uint32)), k
    lay = W.layout(w["shapes"])
    ref = oracle_run(w["opt"], M, np.arange(lay["n_padded"]), 6, lay, w, SEED_G, SEED_I)
    compare(sa, ref)
    a.close()
    b.close()


@pytest.mark.parametrize("M", [3, 4, 5, 7, 8, 12, 16, 32])
@pytest.mark.parametrize("gdt", ["f32", "bf16"])
@pytest.mark.parametrize("base", ["adam", "sgdm"])
def test_global_norm_clip_parity(P, base, gdt, M):
    # sigma = 1 gives ||g|| ~ 90 >> rho = 1: clipping is active every step
    w = workload_dict([5000, 3001, 17], M, base=base, betas=(0.9, 0.999), clip="global_norm",
                      rho=1.0, px=3, pu=2, pv=3, sigma=1.0, gdt=gdt)
    eng = gpu_run(P, w, 10)
    lay = W.layout(w["shapes"])
    ref = oracle_run(w["opt"], M, np.arange(lay["n_padded"]), 10, lay, w, SEED_G, SEED_I)
    compare(gpu_states(eng, w["opt"]), ref)
    eng.close()


@pytest.mark.parametrize("gdt", ["f32", "bf16"])
def test_grad_sqnorm(P, gdt):
    w = workload_dict([70000, 3, 1000], 3, sigma=0.5, gdt=gdt)
    lay = W.layout(w["shapes"])
    g = host_grads(w, lay, SEED_G, 0, np.arange(lay["n_padded"]))
    eng = P.MTDAO(w["opt"], 3, w["shapes"])
    out = torch.zeros(3, dtype=torch.float64, device="cuda")
    gd = to_dev(g, gdt)
    P.mtdao_grad_sqnorm(eng.h, gd.data_ptr(), P.BF16 if gdt == "bf16" else P.F32, out.data_ptr())
    got = out.cpu().numpy()
    expect = np.sum(g.astype(np.float64) ** 2, axis=1)
    assert np.max(np.abs(got - expect) / expect) < 1e-6
    again = torch.zeros_like(out)
    P.mtdao_grad_sqnorm(eng.h, gd.data_ptr(), P.BF16 if gdt == "bf16" else P.F32, again.data_ptr())
    assert torch.equal(out, again)           # deterministic
    eng.close()


@pytest.mark.parametrize("M,gdt", [(4, "f32"), (8, "bf16")])
def test_grad_sqnorm_and_nonfinite_count_at_scale(P, M, gdt):
    """2^26 elements per replica: every thread of the norm kernels walks
    hundreds of strided positions (16-byte loads: 4 f32 or 8 bf16 values).
    The sum of squares matches an fp64 sum taken by torch on the device
    (1e-6 relative, as the oracle's norm tests) and is reproducible; the
    non-finite count finds planted values exactly."""
    from synth.device import DeviceInputs
    shapes = [1 << 26]
    w = workload_dict(shapes, M, sigma=0.5, gdt=gdt)
    lay = W.layout(shapes)
    g = DeviceInputs(w, lay, SEED_G, SEED_I).grads(0)
    eng = P.MTDAO(w["opt"], M, shapes)
    dt = P.BF16 if gdt == "bf16" else P.F32
    out = torch.zeros(M, dtype=torch.float64, device="cuda")
    again = torch.zeros_like(out)
    P.mtdao_grad_sqnorm(eng.h, g.data_ptr(), dt, out.data_ptr())
    P.mtdao_grad_sqnorm(eng.h, g.data_ptr(), dt, again.data_ptr())
    expect = (g.double() ** 2).sum(dim=1)
    assert torch.equal(out, again)
    assert float(((out - expect).abs() / expect).max()) < 1e-6
    g[M - 1, 12345] = float("nan")
    g[0, (1 << 26) - 3] = float("inf")
    g[0, 7] = float("-inf")
    cnt = torch.zeros(M, dtype=torch.float64, device="cuda")
    P.mtdao_grad_nonfinite(eng.h, g.data_ptr(), dt, cnt.data_ptr())
    want = [0.0] * M
    want[0] += 2
    want[M - 1] += 1
    assert cnt.cpu().tolist() == want
    eng.close()


@pytest.mark.parametrize("gdt", ["f32", "bf16"])
def test_grad_sqnorm_extreme_range(P, gdt):
    """Sums of squares whose terms leave fp32's range: replica 0 holds a few
    finite values whose squares overflow fp32 (1.5e19 squares to 2.25e38,
    four of them to more than the largest float; 3e30 and -1e38 overflow
    outright), replica 1 is scaled to ~1e-25 (every square underflows
    fp32), replica 2 is ordinary.  Each must match the fp64 sum within
    1e-6 relative, as the oracle's norm (fp64) does."""
    M = 3
    w = workload_dict([70000, 3, 1000], M, sigma=0.5, gdt=gdt)
    lay = W.layout(w["shapes"])
    g = host_grads(w, lay, SEED_G, 0, np.arange(lay["n_padded"]))
    g[0, [4, 5, 6, 7]] = np.float32(1.5e19)
    g[0, 100] = np.float32(-1.5e19)
    g[0, 2000] = np.float32(3e30)
    g[0, 3001] = np.float32(-1e38)
    g[1] *= np.float32(2e-25)
    if gdt == "bf16":
        g = G.round_bf16(g)
    assert np.all(np.isfinite(g))
    eng = P.MTDAO(w["opt"], M, w["shapes"])
    out = torch.zeros(M, dtype=torch.float64, device="cuda")
    gd = to_dev(g, gdt)
    P.mtdao_grad_sqnorm(eng.h, gd.data_ptr(), P.BF16 if gdt == "bf16" else P.F32, out.data_ptr())
    got = out.cpu().numpy()
    expect = np.sum(g.astype(np.float64) ** 2, axis=1)
    assert np.all(np.isfinite(got)), got
    assert np.max(np.abs(got - expect) / expect) < 1e-6, (got, expect)
    eng.close()


@pytest.mark.parametrize("gdt", ["f32", "bf16"])
@pytest.mark.parametrize("base", ["adam", "sgdm"])
def test_global_norm_clip_parity_with_huge_gradients(P, base, gdt):
    """clip(g, rho) when a replica's gradient holds finite values whose fp32
    squares overflow a four-term sum (1.5e19 each): the norm is formed in
    range, the clip factor is the oracle's tiny one rather than 0, and every
    state matches the oracle (the states themselves stay within fp32)."""
    M = 4
    w = workload_dict([5000, 3001, 17], M, base=base, betas=(0.9, 0.999), clip="global_norm",
                      rho=1.0, px=3, pu=2, pv=3, sigma=1.0, gdt=gdt)
    lay = W.layout(w["shapes"])
    n = lay["n_padded"]
    idx = np.arange(n)
    lr = w["opt"]["lr"]
    eng = P.MTDAO(w["opt"], M, w["shapes"])
    x0 = G.init_params(w, lay, SEED_I, idx)
    eng.set_params(torch.from_numpy(x0).cuda())
    from oracle.oracle import Oracle
    o = Oracle(w["opt"], M, n, x0=x0.astype(np.float64))
    T = 6
    for t in range(T):
        g = host_grads(w, lay, SEED_G, t, idx)
        if t in (1, 4):
            g[1, 8:12] = np.float32(1.5e19)
            g[2, 5003] = np.float32(-1.5e19)
            if gdt == "bf16":
                g = G.round_bf16(g)             # what the device sees after its bf16 rounding
        eng.step(to_dev(g, gdt), lr, eng.sync_due())
        o.step(t, lr, g.astype(np.float64))
    o.settle(T)
    torch.cuda.synchronize()
    compare(gpu_states(eng, w["opt"]), o.states())
    eng.close()


@pytest.mark.parametrize("gdt", ["f32", "bf16"])
def test_grad_nonfinite_counts(P, gdt):
    """mtdao_grad_nonfinite counts exactly the NaN / +-Inf values planted in
    each replica's gradient (counts known by construction); the largest
    finite values, subnormals and -0 are not counted."""
    M = 5
    w = workload_dict(RAGGED + [70000], M, gdt=gdt)
    lay = W.layout(w["shapes"])
    n = lay["n_padded"]
    g = host_grads(w, lay, SEED_G, 0, np.arange(n))
    rng = np.random.default_rng(31)
    extremes = {(0, 1): 3.0e38, (1, 2): -3.0e38, (2, 3): 1e-45, (3, 4): -0.0, (4, 5): 1e-39}
    for (m, i), v in extremes.items():
        g[m, i] = np.float32(v)
    expected = []
    for m in range(M):
        k = [0, 1, 7, 300, 4099][m]
        pos = rng.choice(np.arange(8, n), size=k, replace=False)
        g[m, pos] = rng.choice(np.array([np.nan, np.inf, -np.inf], np.float32), size=k)
        expected.append(float(k))
    gd = to_dev(g, gdt)
    dt = P.BF16 if gdt == "bf16" else P.F32
    eng = P.MTDAO(w["opt"], M, w["shapes"])
    out = torch.full((M,), -1.0, dtype=torch.float64, device="cuda")
    P.mtdao_grad_nonfinite(eng.h, gd.data_ptr(), dt, out.data_ptr())
    assert out.cpu().numpy().tolist() == expected
    clean = to_dev(host_grads(w, lay, SEED_G, 1, np.arange(n)), gdt)
    P.mtdao_grad_nonfinite(eng.h, clean.data_ptr(), dt, out.data_ptr())
    assert out.cpu().numpy().tolist() == [0.0] * M
    eng.close()


@pytest.mark.parametrize("clip", ["elementwise", "none"])
@pytest.mark.parametrize("gdt", ["f32", "bf16"])
@pytest.mark.parametrize("M", [2, 4, 8])
def test_adopt_clip_parity(P, clip, M, gdt):
    w = workload_dict(RAGGED, M, base="adopt", betas=(0.95, 0.999), beta2=0.9999, clip=clip,
                      px=6, pu=3, pv=3, lr=2.0 ** -8, gdt=gdt)
    eng = gpu_run(P, w, 20)
    lay = W.layout(w["shapes"])
    ref = oracle_run(w["opt"], M, np.arange(lay["n_padded"]), 20, lay, w, SEED_G, SEED_I)
    compare(gpu_states(eng, w["opt"]), ref)
    eng.close()


@pytest.mark.parametrize("M", [3, 4, 8])
@pytest.mark.parametrize("clip", ["elementwise", "none"])
def test_adopt_original_ordering_parity(P, clip, M):
    """adopt_prev_v (original ADOPT order): step 0 only initialises v."""
    w = workload_dict(RAGGED, M, base="adopt", betas=(0.95, 0.999), beta2=0.9999, clip=clip,
                      px=5, pu=3, pv=4, lr=2.0 ** -8)
    w["opt"]["adopt_prev_v"] = True
    eng = gpu_run(P, w, 17)
    lay = W.layout(w["shapes"])
    ref = oracle_run(w["opt"], M, np.arange(lay["n_padded"]), 17, lay, w, SEED_G, SEED_I)
    compare(gpu_states(eng, w["opt"]), ref)
    eng.close()


@pytest.mark.parametrize("M", [3, 4, 8])
@pytest.mark.parametrize("base", ["adopt", "adam", "sgdm"])
def test_alg2_literal_phase_parity(P, base, M):
    w = workload_dict(RAGGED, M, base=base, betas=(0.95, 0.5), beta2=0.9999 if base == "adopt" else 0.999,
                      px=4, pu=[3, 2], pv=5, phase="alg2_literal", lr=2.0 ** -8)
    eng = gpu_run(P, w, 14)
    lay = W.layout(w["shapes"])
    ref = oracle_run(w["opt"], M, np.arange(lay["n_padded"]), 14, lay, w, SEED_G, SEED_I)
    compare(gpu_states(eng, w["opt"]), ref)
    eng.close()


def test_sync_kernel_parity_and_invariants(P):
    M, shapes = 4, [20000, 11]
    w = workload_dict(shapes, M, betas=(0.9, 0.99))
    eng = P.MTDAO(w["opt"], M, shapes)
    n = eng.n_padded
    rng = np.random.default_rng(3)
    vals = {}
    for s in range(eng.n_states):
        arr = rng.standard_normal((M, n)).astype(np.float32)
        if s == eng.n_states - 1:
            arr = np.abs(arr)
        vals[s] = arr
        eng.state_view(s).copy_(torch.from_numpy(arr).cuda())
    eng.sync(0b1011)                       # x, u1, v
    torch.cuda.synchronize()
    for s in range(eng.n_states):
        got = eng.state_view(s).cpu().numpy()
        if (0b1011 >> s) & 1:
            expect = np.broadcast_to(vals[s].astype(np.float64).mean(0), (M, n))
            # s_0 + fl(sum_m fl(s_m - s_0)) / M: M-1 differences, M-2 additions,
            # one division and one addition, each within u = 2^-24 of operands
            # bounded by 2 max_m |s_m|  ->  |error| <= (2M + 1) u max_m |s_m|
            bound = (2 * M + 1) * 2.0 ** -24 * np.abs(vals[s]).max(axis=0)
            assert np.all(np.abs(got - expect) <= bound[None, :])
            assert rel_err(got, expect) <= 1e-5
            assert np.all(got == got[0:1])
        else:
            assert np.array_equal(got, vals[s])
    before = {s: eng.state_view(s).cpu().numpy().copy() for s in range(eng.n_states)}
    eng.sync(0b1011)                       # idempotent: replicas now agree
    torch.cuda.synchronize()
    for s in range(eng.n_states):
        assert np.array_equal(eng.state_view(s).cpu().numpy(), before[s])
    eng.close()


@pytest.mark.parametrize("path", ["sync", "stats", "fused"])
@pytest.mark.parametrize("M", [2, 3, 4, 8, 12, 16, 300])
def test_mean_of_nonfinite_values(P, M, path):
    """The worker mean of values that hold infinities is the infinity when
    they have one sign only, NaN when both signs or a NaN occur (the mean
    sum_m s_m / M of the method), in the plain and the diagnostics average
    and in the fused step (u_1 = beta u_1 with a zero gradient keeps the
    values' classes).  Finite columns keep the compensated mean."""
    if path == "fused" and M > 256:
        pytest.skip("the fused average covers M <= 256")
    shapes = [1024]
    w = workload_dict(shapes, M, betas=(0.9, 0.99))
    eng = P.MTDAO(w["opt"], M, shapes)
    n = eng.n_padded
    rng = np.random.default_rng(M)
    vals = rng.standard_normal((M, n)).astype(np.float32)
    vals[M - 1, 0] = np.inf                  # one +inf
    vals[M // 2, 1] = -np.inf                # one -inf
    vals[0, 2], vals[M - 1, 2] = np.inf, -np.inf
    vals[1 % M, 3] = np.nan
    vals[:, 4] = np.inf                      # every replica +inf
    vals[0, 5] = -np.inf                     # the reference replica
    u1 = 1
    eng.state_view(u1).copy_(torch.from_numpy(vals).cuda())
    with np.errstate(invalid="ignore"):          # inf - inf in the reference mean is the point
        if path == "sync":
            eng.sync(1 << u1)
            expect = vals.astype(np.float64).mean(0)
        elif path == "stats":
            eng.sync_stats(1 << u1)
            expect = vals.astype(np.float64).mean(0)
        else:
            g = torch.zeros((M, n), device="cuda")
            eng.step(g, 1e-3, 1 << u1)
            beta = w["opt"]["beta1"][0]
            expect = (beta * vals.astype(np.float64)).mean(0)
    torch.cuda.synchronize()
    got = eng.state_view(u1).cpu().numpy()
    ref = np.broadcast_to(expect.astype(np.float32), (M, n))
    assert np.array_equal(np.isnan(got), np.isnan(ref))
    assert np.array_equal(np.isposinf(got), np.isposinf(ref))
    assert np.array_equal(np.isneginf(got), np.isneginf(ref))
    assert np.all(got == got[0:1]) or np.all(np.isnan(got) == np.isnan(got[0:1]))
    fin = np.isfinite(ref)
    assert np.allclose(got[fin], ref[fin], rtol=1e-5, atol=1e-6)
    eng.close()


@pytest.mark.parametrize("M", [1, 3, 4, 6, 8])
def test_sync_identity_on_identical_replicas(P, M):
    w = workload_dict([777, 4096], M, betas=(0.9,))
    eng = P.MTDAO(w["opt"], M, w["shapes"])
    rng = np.random.default_rng(M)
    for s in range(eng.n_states):
        row = rng.standard_normal(eng.n_padded).astype(np.float32)
        eng.state_view(s).copy_(torch.from_numpy(np.tile(row, (M, 1))).cuda())
    before = {s: eng.state_view(s).cpu().numpy().copy() for s in range(eng.n_states)}
    eng.sync((1 << eng.n_states) - 1)
    torch.cuda.synchronize()
    for s in range(eng.n_states):
        assert np.array_equal(eng.state_view(s).cpu().numpy().view(np.uint32),
                              before[s].view(np.uint32))
    eng.close()


@pytest.mark.parametrize("M,gdt", [(4, "f32"), (8, "bf16"), (3, "bf16")])
@pytest.mark.parametrize("memory", ["pinned", "pageable"])
def test_host_gradient_path_is_bitwise_equal(P, memory, M, gdt):
    """Pinned host gradients are read by the kernel over the host link;
    pageable ones go through the staging copy.  Both equal the device path."""
    w = workload_dict(RAGGED, M, betas=(0.9, 0.999), px=3, pu=3, pv=3, gdt=gdt)
    lay = W.layout(w["shapes"])
    idx = np.arange(lay["n_padded"])
    a = gpu_run(P, w, 7)
    b = P.MTDAO(w["opt"], M, w["shapes"])
    b.set_params(torch.from_numpy(G.init_params(w, lay, SEED_I, idx)).cuda())
    dt = P.BF16 if gdt == "bf16" else P.F32
    for t in range(7):
        g = np.ascontiguousarray(host_grads(w, lay, SEED_G, t, idx))
        if gdt == "bf16":
            g = np.ascontiguousarray(G.to_bf16_bits(g))          # the bf16 bit patterns
        if memory == "pinned":
            gt = torch.from_numpy(g.view(np.int16) if gdt == "bf16" else g).pin_memory()
            b.step_host(gt.data_ptr(), 1e-3, dtype=dt)
        else:
            b.step_host(g.ctypes.data, 1e-3, dtype=dt)
        torch.cuda.current_stream().synchronize()
    sa, sb = gpu_states(a, w["opt"]), gpu_states(b, w["opt"])
    for k in sa:
        assert np.array_equal(sa[k], sb[k]), k
    a.close()
    b.close()


def test_checkpoint_resume_is_bitwise_equal(P):
    w = workload_dict(RAGGED, 4, betas=(0.9, 0.999), px=4, pu=3, pv=4)
    full = gpu_run(P, w, 10)
    first = gpu_run(P, w, 6)
    saved = {s: first.state_view(s).cpu().numpy().copy() for s in range(first.n_states)}
    step = first.t
    first.close()
    resumed = P.MTDAO(w["opt"], 4, w["shapes"])
    for s, arr in saved.items():
        for m in range(4):
            row = np.ascontiguousarray(arr[m])
            P.mtdao_copy_state_from_host(resumed.h, s, m, row.ctypes.data)
    resumed.t = step
    gpu_run(P, w, 4, t0=6, eng=resumed)
    sf, sr = gpu_states(full, w["opt"]), gpu_states(resumed, w["opt"])
    for k in sf:
        assert np.array_equal(sf[k], sr[k]), k
    full.close()
    resumed.close()


NONFINITE_VARIANTS = {
    "adam": dict(base="adam"),
    "adam_clip": dict(base="adam", clip="global_norm", rho=1.0),
    "adopt": dict(base="adopt", beta2=0.9999),
    "adopt_prev_v": dict(base="adopt", beta2=0.9999, clip="elementwise"),
    "sgdm": dict(base="sgdm"),
}


@pytest.mark.parametrize("M", [4, 12])
@pytest.mark.parametrize("t_plant", [0, 2])
@pytest.mark.parametrize("sync", ["plain", "fused_every2", "fused_every1"])
@pytest.mark.parametrize("gdt", ["f32", "bf16"])
@pytest.mark.parametrize("variant", sorted(NONFINITE_VARIANTS))
def test_nonfinite_gradients_propagate_like_the_oracle(P, variant, gdt, sync, t_plant, M):
    """NaN, +Inf and -Inf gradients planted in three of M replicas at
    step 0 or 2, with no average, the fused average every second step, or
    every step: the NaN/Inf positions of every state equal the oracle's and
    the finite values agree within the tolerance.  The original ADOPT order
    (step 0 only sets v = g_0^2, Algorithm 2 read as the original method)
    must leave u and x finite when step 0's gradient is not.  An infinite
    state stays infinite at the next steps (beta * inf = inf), M = 12 runs
    the fused average of the block-staged kernel."""
    period = {"plain": 0, "fused_every2": 2, "fused_every1": 1}[sync]
    kw = dict(NONFINITE_VARIANTS[variant])
    w = workload_dict([1000, 37], M, betas=(0.9, 0.99), px=period, pu=period, pv=period, gdt=gdt,
                      lr=2.0 ** -8 if kw["base"] == "adopt" else 1e-3, **kw)
    if variant == "adopt_prev_v":
        w["opt"]["adopt_prev_v"] = True
    lay = W.layout(w["shapes"])
    n = lay["n_padded"]
    idx = np.arange(n)
    lr = w["opt"]["lr"]
    eng = P.MTDAO(w["opt"], M, w["shapes"])
    x0 = G.init_params(w, lay, SEED_I, idx)
    eng.set_params(torch.from_numpy(x0).cuda())
    from oracle.oracle import Oracle
    o = Oracle(w["opt"], M, n, x0=x0.astype(np.float64))
    T = 4
    for t in range(T):
        g = host_grads(w, lay, SEED_G, t, idx)
        if t == t_plant:
            g[0, 5] = np.nan
            g[1, 9] = np.inf
            g[2, lay["offsets"][1] + 3] = -np.inf
        eng.step(to_dev(g, gdt), lr, eng.sync_due())
        o.step(t, lr, g.astype(np.float64))
    o.settle(T)
    torch.cuda.synchronize()
    got, ref = gpu_states(eng, w["opt"]), o.states()
    compare(got, ref)                    # includes: non-finite positions are equal
    # NaN and each sign of Inf where the oracle has them, averages included
    # (the mean of values holding infinities of one sign is that infinity)
    for k in ref:
        assert np.array_equal(np.isnan(got[k]), np.isnan(ref[k])), k
        assert np.array_equal(np.isposinf(got[k]), np.isposinf(ref[k])), k
        assert np.array_equal(np.isneginf(got[k]), np.isneginf(ref[k])), k
    eng.close()


def test_original_adopt_step0_moves_nothing_but_v(P):
    """Original ADOPT order, step 0 with non-finite gradients: v = g_0^2
    (NaN or Inf where g_0 is), u and x bit-identical to their initial
    values on every replica, averaged or not."""
    for period in (0, 1):
        w = workload_dict([1000, 37], 4, base="adopt", betas=(0.9, 0.99), beta2=0.9999, px=period,
                          pu=period, pv=period, clip="elementwise")
        w["opt"]["adopt_prev_v"] = True
        lay = W.layout(w["shapes"])
        idx = np.arange(lay["n_padded"])
        eng = P.MTDAO(w["opt"], 4, w["shapes"])
        x0 = G.init_params(w, lay, SEED_I, idx)
        eng.set_params(torch.from_numpy(x0).cuda())
        g = host_grads(w, lay, SEED_G, 0, idx)
        g[0, 5], g[1, 9], g[2, 40] = np.nan, np.inf, -np.inf
        eng.step(to_dev(g, "f32"), 2.0 ** -8, eng.sync_due())
        torch.cuda.synchronize()
        st = gpu_states(eng, w["opt"])
        assert np.array_equal(st["x"], np.broadcast_to(x0, st["x"].shape))
        for j in (1, 2):
            assert not np.any(st["u%d" % j]), j
        want = (g.astype(np.float32) ** 2)
        if period == 1:
            # averaged at the end of step 0: a column with a non-finite
            # replica value is non-finite on every replica, the others hold
            # the replica mean of g_0^2
            nonfin = ~np.isfinite(want).all(axis=0)
            assert np.array_equal(~np.isfinite(st["v"]), np.broadcast_to(nonfin, st["v"].shape))
            mean = want[:, ~nonfin].astype(np.float64).mean(axis=0)
            assert np.allclose(st["v"][:, ~nonfin], mean[None, :], rtol=1e-6, atol=0)
        else:
            assert np.array_equal(st["v"], want, equal_nan=True)
        eng.close()


def test_error_codes(P, monkeypatch):
    w = workload_dict([1024], 2, betas=(0.9,))
    eng = P.MTDAO(w["opt"], 2, w["shapes"])
    g = torch.zeros(2 * eng.n_padded + 4, device="cuda")
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_step(eng.h, g.data_ptr() + 4, P.F32, 1e-3, 0)
    assert e.value.code == P.ERR_ALIGN
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_step(eng.h, g.data_ptr(), 7, 1e-3, 0)
    assert e.value.code == P.ERR_INVALID
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_step(eng.h, g.data_ptr(), P.F32, 1e-3, 1 << eng.n_states)
    assert e.value.code == P.ERR_INVALID
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_sync(eng.h, 1 << 5)
    assert e.value.code == P.ERR_INVALID
    # double outputs must be 8-byte aligned; refused before any launch
    outs = torch.zeros(64, dtype=torch.float64, device="cuda")
    bad = outs.data_ptr() + 4
    for call in (lambda: P.mtdao_grad_sqnorm(eng.h, g.data_ptr(), P.F32, bad),
                 lambda: P.mtdao_grad_nonfinite(eng.h, g.data_ptr(), P.F32, bad),
                 lambda: P.mtdao_sync_stats(eng.h, 1, bad)):
        with pytest.raises(P.MTDAOError) as e:
            call()
        assert e.value.code == P.ERR_ALIGN
    P.mtdao_track_anchor(eng.h, 1)
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_pseudo_grad_stats(eng.h, 0, bad)
    assert e.value.code == P.ERR_ALIGN
    P.mtdao_track_anchor(eng.h, 0)
    torch.cuda.synchronize()
    assert eng.t == 0
    eng.close()
    free0 = torch.cuda.mem_get_info()[0]
    for k in (1, 2, 3, 4):
        monkeypatch.setenv("MTDAO_FAULT_ALLOC", str(k))
        with pytest.raises(P.MTDAOError) as e:
            P.mtdao_create(P.make_config(w["opt"]), 2, [1 << 20])
        assert e.value.code == P.ERR_OOM
        assert "failed" in P.mtdao_last_error(None)
    monkeypatch.delenv("MTDAO_FAULT_ALLOC")
    torch.cuda.synchronize()
    assert abs(torch.cuda.mem_get_info()[0] - free0) < (64 << 20)


def test_device_generator_matches_host_generator(P):
    from synth.device import DeviceInputs
    for name in ("tiny", "gpt2_small", "decoder_350m", "decoder_1b"):
        w = W.get(name)
        w["M"] = min(w["M"], 2)
        w["shapes"] = w["shapes"][:3] + [1001]
        lay = W.layout(w["shapes"])
        dev = DeviceInputs(w, lay, SEED_G, SEED_I)
        idx = sample_indices(lay, 5000, seed=1)
        for t in (0, 7):
            got = dev.grads(t)
            if w["grad_dtype"] == "bf16":
                got = got.float()
            got = got.cpu().numpy()[:, idx]
            expect = host_grads(w, lay, SEED_G, t, idx)
            assert np.array_equal(got.view(np.uint32), expect.view(np.uint32)), name
        x0 = dev.init_params().cpu().numpy()[idx]
        assert np.array_equal(x0, G.init_params(w, lay, SEED_I, idx))


def test_zero_size_and_single_element_tensors(P):
    for shapes in ([0, 5, 0, 300, 0], [1]):
        w = workload_dict(shapes, 2, betas=(0.9, 0.999), px=2, pu=3, pv=2)
        eng = gpu_run(P, w, 7)
        lay = W.layout(w["shapes"])
        ref = oracle_run(w["opt"], 2, np.arange(lay["n_padded"]), 7, lay, w, SEED_G, SEED_I)
        compare(gpu_states(eng, w["opt"]), ref)
        eng.close()


@pytest.mark.parametrize("base,M", [("adam", 4), ("adopt", 8), ("sgdm", 2), ("adam", 3)])
def test_padding_canaries_are_untouched(P, base, M):
    """Canary values planted in the parameters' alignment padding (between
    tensors and at the end) survive steps, fused and standalone averages bit
    for bit, u and v stay zero there, and the tensors' own elements are
    bit-identical to a run without canaries: no kernel reads or writes
    across a tensor boundary."""
    w = workload_dict(RAGGED, M, base=base, betas=(0.9, 0.99), px=3, pu=[2, 4], pv=2,
                      beta2=0.9999 if base == "adopt" else 0.999)
    lay = W.layout(w["shapes"])
    n = lay["n_padded"]
    inside = G.in_tensor_mask(np.arange(n), lay["offsets"], lay["numels"])
    assert (~inside).sum() > 0
    x0 = G.init_params(w, lay, SEED_I, np.arange(n))
    x0c = x0.copy()
    x0c[~inside] = np.float32(1234.5)
    runs = []
    for start in (x0, x0c):
        eng = gpu_run(P, w, 9, x0=start)
        eng.sync(0b1)                                     # one standalone average too
        torch.cuda.synchronize()
        runs.append(gpu_states(eng, w["opt"]))
        eng.close()
    plain, canary = runs
    assert np.all(canary["x"][:, ~inside] == np.float32(1234.5))
    for name, a in canary.items():
        if name != "x":
            assert np.all(a[:, ~inside] == 0), name
        assert np.array_equal(a[:, inside].view(np.uint32), plain[name][:, inside].view(np.uint32)), name


def test_handle_streams_are_respected(P):
    """A handle created on a side stream, switched to another stream with
    mtdao_set_stream half-way, and two handles stepping concurrently on two
    streams all give the bits of the same run on the default stream: every
    launch and copy goes to the handle's stream."""
    w = workload_dict(RAGGED, 4, betas=(0.9, 0.99), px=3, pu=[2, 5], pv=4)
    lay = W.layout(w["shapes"])
    n = lay["n_padded"]
    T = 9
    x0 = torch.from_numpy(G.init_params(w, lay, SEED_I, np.arange(n))).cuda()
    gs = [to_dev(host_grads(w, lay, SEED_G, t, np.arange(n)), "f32") for t in range(T)]
    torch.cuda.synchronize()

    def run(eng, stream_for_step):
        for t in range(T):
            with torch.cuda.stream(stream_for_step(t)):
                eng.step(gs[t], 1e-3)
        return eng

    base = P.MTDAO(w["opt"], 4, w["shapes"])
    base.set_params(x0)
    run(base, lambda t: torch.cuda.current_stream())
    torch.cuda.synchronize()
    ref = gpu_states(base, w["opt"])
    base.close()

    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    eng = P.MTDAO(w["opt"], 4, w["shapes"], stream=s1.cuda_stream)
    eng.set_params(x0)
    for t in range(T):
        if t == 5:
            s2.wait_stream(s1)
            P.mtdao_set_stream(eng.h, s2.cuda_stream)
        P.mtdao_step(eng.h, gs[t].data_ptr(), P.F32, 1e-3, P.mtdao_sync_due(eng.h))
    s2.synchronize()
    got = gpu_states(eng, w["opt"])
    eng.close()
    for k in ref:
        assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k

    a = P.MTDAO(w["opt"], 4, w["shapes"], stream=s1.cuda_stream)
    b = P.MTDAO(w["opt"], 4, w["shapes"], stream=s2.cuda_stream)
    a.set_params(x0)
    b.set_params(x0)
    for t in range(T):                     # interleaved launches, two streams
        P.mtdao_step(a.h, gs[t].data_ptr(), P.F32, 1e-3, P.mtdao_sync_due(a.h))
        P.mtdao_step(b.h, gs[t].data_ptr(), P.F32, 1e-3, P.mtdao_sync_due(b.h))
    torch.cuda.synchronize()
    for eng in (a, b):
        got = gpu_states(eng, w["opt"])
        for k in ref:
            assert np.array_equal(got[k].view(np.uint32), ref[k].view(np.uint32)), k
        eng.close()


def test_binding_rejects_tensors_the_library_would_misread(P):
    """The library reads raw pointers, so the binding checks each tensor's
    shape, dtype, contiguity and device before passing it on."""
    w = workload_dict(RAGGED, 4)
    eng = P.MTDAO(w["opt"], 4, w["shapes"])
    n = eng.n_padded
    good = torch.zeros((4, n), device="cuda")
    eng.step(good, 1e-3)
    bad = [torch.zeros((4, n - 8), device="cuda"),                 # wrong shape
           torch.zeros((n, 4), device="cuda").t(),                 # transposed view: not contiguous
           torch.zeros((4, n), device="cuda", dtype=torch.float16),
           torch.zeros((4, n))]                                     # host memory for the device call
    for g in bad:
        with pytest.raises(ValueError):
            eng.step(g, 1e-3)
    with pytest.raises(ValueError):
        eng.step(good, 1e-3, dtype=P.BF16)                         # code contradicts the tensor
    with pytest.raises(ValueError):
        eng.step_host(good, 1e-3)                                  # device memory for the host call
    with pytest.raises(ValueError):
        eng.set_params(torch.zeros(n + 1, device="cuda"))
    with pytest.raises(ValueError):
        eng.run(torch.zeros((3, 4, n), device="cuda"), [1e-3] * 2)  # count does not match lrs
    assert eng.t == 1                                              # nothing ran
    eng.close()


@pytest.mark.parametrize("case", ["qhm_beta0_no_grad_term", "omega0", "sgdm_sum_omega1",
                                  "adopt_beta0", "max_replicas"])
def test_degenerate_hyperparameters(P, case):
    M, base, betas, om, kw = 4, "adam", (0.0, 0.999), (0.5, 0.5), {}
    if case == "omega0":
        betas, om = (0.9, 0.99), (0.0, 0.0)
    elif case == "sgdm_sum_omega1":
        base, betas, om = "sgdm", (0.5, 0.99), (0.3, 0.7)
    elif case == "adopt_beta0":
        base, betas, om, kw = "adopt", (0.0, 0.9), (0.5, 0.25), {"beta2": 0.9999, "lr": 2.0 ** -8}
    elif case == "max_replicas":
        M, betas, om = P.MAX_REPLICAS, (0.9,), (0.95,)
    shapes = [300, 5] if case == "max_replicas" else [3000, 17]
    w = workload_dict(shapes, M, base=base, betas=betas, omega=om, px=3, pu=2, pv=3, **kw)
    eng = gpu_run(P, w, 8)
    lay = W.layout(w["shapes"])
    ref = oracle_run(w["opt"], M, np.arange(lay["n_padded"]), 8, lay, w, SEED_G, SEED_I)
    compare(gpu_states(eng, w["opt"]), ref)
    eng.close()


def test_zero_learning_rate_leaves_parameters_bitwise(P):
    w = workload_dict(RAGGED, 4, betas=(0.9, 0.999), px=0, pu=3, pv=3)
    lay = W.layout(w["shapes"])
    x0 = G.init_params(w, lay, SEED_I, np.arange(lay["n_padded"]))
    eng = gpu_run(P, w, 6, lr=0.0, x0=x0)
    got = eng.state_view(0).cpu().numpy()
    assert np.array_equal(got.view(np.uint32), np.tile(x0, (4, 1)).view(np.uint32))
    eng.close()


def test_run_equals_step_by_step(P):
    """mtdao_run over a stack of gradient buffers (and with one reused
    buffer) gives the bits of the same steps issued one by one."""
    w = workload_dict(RAGGED, 4, betas=(0.9, 0.999), px=3, pu=2, pv=3)
    lay = W.layout(w["shapes"])
    idx = np.arange(lay["n_padded"])
    x0 = torch.from_numpy(G.init_params(w, lay, SEED_I, idx)).cuda()
    gs = torch.from_numpy(np.stack([host_grads(w, lay, SEED_G, t, idx) for t in range(7)])).cuda()
    lrs = [1e-3 * (1 + 0.1 * t) for t in range(7)]
    a, b, c, d = (P.MTDAO(w["opt"], 4, w["shapes"]) for _ in range(4))
    for e in (a, b, c, d):
        e.set_params(x0)
    for t in range(7):
        a.step(gs[t], lrs[t])
        c.step(gs[0], lrs[t])
    b.run(gs, lrs)
    d.run(gs[0], lrs)
    torch.cuda.synchronize()
    assert b.t == 7 and d.t == 7
    for s in range(a.n_states):
        assert torch.equal(a.state_view(s), b.state_view(s)), s
        assert torch.equal(c.state_view(s), d.state_view(s)), s
    for e in (a, b, c, d):
        e.close()
