"""Pins of the CPU oracle to things other than itself.

Each test checks the oracle against something the paper or the mathematics
fixes: closed forms under a constant gradient, the unrolled EMA and its
variance (section 2.1 and the appendix derivation), library routines
(torch.optim.Adam, numpy mean/norm), invariants of the worker average,
values the paper prints, and stated equivalences (Local Adam recovery,
section 2.3; model-sync vs momentum-sync equivalence for SGDM, section 3).
"""
import math
import os

import numpy as np
import pytest
import torch

from oracle.oracle import Oracle, adopt_clip_bound, comm_reduction, grad_norm, half_life, \
    half_life_periods

HERE = os.path.dirname(os.path.abspath(__file__))


def cfg(base="adam", betas=(0.9,), omega=None, beta2=0.999, eps=1e-8, bias=True,
        clip="none", rho=1.0, px=0, pu=0, pv=0, phase="alg1"):
    n = len(betas)
    if omega is None:
        omega = [0.95 / n] * n
    return {"base": base, "n_mom": n, "beta1": list(betas), "omega": list(omega),
            "beta2": beta2, "eps": eps, "bias_correction": bias, "clip_mode": clip,
            "clip_rho": rho, "period_x": px, "period_u": [pu] * n, "period_v": pv,
            "sync_phase": phase}


def rel(a, b):
    a, b = np.asarray(a), np.asarray(b)
    return float(np.max(np.abs(a - b) / np.maximum(np.abs(b), 1e-300)))


# ---------------------------------------------------------------- EMA pins

@pytest.mark.parametrize("base", ["adam", "sgdm"])
def test_ema_constant_gradient_closed_form(base):
    """u_j after t+1 steps from 0 with constant g is (1-beta_j^(t+1)) g, and
    v is (1-beta2^(t+1)) g^2 (section 2.1 unrolled EMA with g constant)."""
    betas = (0.5, 0.9, 0.999)
    c = cfg(base, betas, omega=(0.2, 0.3, 0.4))
    rng = np.random.default_rng(1)
    M, n = 2, 64
    g = rng.standard_normal((M, n)) * np.logspace(-4, 0, n)
    o = Oracle(c, M, n, x0=rng.standard_normal(n))
    for t in range(60):
        o.step(t, 1e-3, g)
        for j, b in enumerate(betas):
            assert rel(o.u[j], (1 - b ** (t + 1)) * g) < 1e-12
        if base == "adam":
            assert rel(o.v, (1 - 0.999 ** (t + 1)) * g * g) < 1e-12


def test_adopt_second_moment_constant_gradient():
    c = cfg("adopt", (0.9,), beta2=0.9999, bias=False)
    rng = np.random.default_rng(2)
    g = rng.standard_normal((1, 32))
    o = Oracle(c, 1, 32)
    for t in range(40):
        o.step(t, 1e-3, g)
        assert rel(o.v, (1 - 0.9999 ** (t + 1)) * g * g) < 1e-11


@pytest.mark.parametrize("beta", [0.5, 0.9, 0.999])
def test_ema_unrolled_form(beta):
    """u_{t+K} = beta^K u_t + (1-beta) sum_k beta^k g_{t+K-k} (section 2.1)."""
    c = cfg("sgdm", (beta,))
    rng = np.random.default_rng(3)
    n, K = 128, 37
    o = Oracle(c, 1, n)
    u_t = rng.standard_normal(n)
    o.u[0, 0] = u_t
    gs = rng.standard_normal((K, n))
    for s in range(K):
        o.step(100 + s, 0.01, gs[s:s + 1])
    expect = beta ** K * u_t
    for k in range(K):
        expect = expect + (1 - beta) * beta ** k * gs[K - 1 - k]
    assert np.max(np.abs(o.u[0, 0] - expect)) < 1e-13 * (1 + np.max(np.abs(expect)))


@pytest.mark.parametrize("beta", [0.9, 0.99])
def test_local_momentum_variance(beta):
    """Var(u_{t+K}) = (1-beta)/(1+beta) (1-beta^{2K}) sigma^2 for iid noise
    and a synced (constant) start (appendix, variance of local momentum)."""
    c = cfg("sgdm", (beta,))
    rng = np.random.default_rng(4)
    n, K, sigma = 1 << 18, 32, 0.7
    o = Oracle(c, 1, n)
    o.u[0, 0] = 0.25                       # synchronised start, same everywhere
    for s in range(K):
        o.step(s, 0.0, rng.standard_normal((1, n)) * sigma)
    emp = float(np.var(o.u[0, 0]))
    theory = (1 - beta) / (1 + beta) * (1 - beta ** (2 * K)) * sigma ** 2
    se = theory * math.sqrt(2.0 / n)
    assert abs(emp - theory) < 5 * se


def _golden():
    rows = {}
    with open(os.path.join(HERE, "golden", "paper_values.txt")) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            parts = line.split()
            kv = dict(p.split("=", 1) for p in parts[1:] if "=" in p and not p.startswith('"'))
            rows[parts[0]] = kv
    return rows


def test_paper_printed_decay_factor():
    """After K=32 steps with beta=0.9 the synced momentum keeps ~0.03 of its
    value (printed in section 2.1)."""
    row = _golden()["ema_decay_factor"]
    beta, K = float(row["beta"]), int(row["K"])
    o = Oracle(cfg("sgdm", (beta,)), 1, 1)
    o.u[0, 0, 0] = 1.0
    for s in range(K):
        o.step(s, 0.0, np.zeros((1, 1)))
    assert abs(o.u[0, 0, 0] - float(row["printed"])) <= float(row["tol"])


def test_paper_printed_half_life():
    """tau_0.5(0.9) ~ 6.6 steps (section 2.1): the EMA of a unit impulse with
    zero later gradients falls through 0.5 between steps 6 and 7, at 6.6 on a
    log scale."""
    row = _golden()["ema_half_life"]
    beta = float(row["beta"])
    o = Oracle(cfg("sgdm", (beta,)), 1, 1)
    o.u[0, 0, 0] = 1.0
    traj = [1.0]
    for s in range(10):
        o.step(s, 0.0, np.zeros((1, 1)))
        traj.append(float(o.u[0, 0, 0]))
    k = next(i for i, u in enumerate(traj) if u < 0.5)
    assert k == 7
    lo, hi = math.log(traj[k - 1]), math.log(traj[k])
    crossing = (k - 1) + (lo - math.log(0.5)) / (lo - hi)
    assert abs(crossing - float(row["printed"])) <= float(row["tol"])



HALF_LIFE_ROWS = ["halflife_desloc_adam", "halflife_desloc_adopt", "halflife_mtdao_adam",
                  "halflife_mtdao_adopt"]


@pytest.mark.parametrize("name", HALF_LIFE_ROWS)
def test_paper_printed_half_life_periods(name):
    """The wall-clock appendix's Half-Life configurations: K_u1 and K_v from
    beta_1, beta_2 and K_x = 32, as printed (exact)."""
    row = _golden()[name]
    base = "adopt" if float(row["beta2"]) == 0.9999 else "adam"
    c = cfg(base, (float(row["beta1"]),), beta2=float(row["beta2"]), bias=base == "adam")
    got = half_life_periods(c, int(row["K_x"]))
    assert got["period_x"] == int(row["K_x"])
    assert got["period_u"] == [int(row["K_u"])]
    assert got["period_v"] == int(row["K_v"])


@pytest.mark.parametrize("beta", [0.8, 0.9, 0.99, 0.999, 0.9999])
def test_half_life_matches_the_ema_impulse_response(beta):
    """tau_0.5 is where the EMA's memory of one value halves: the oracle's
    own EMA (an SGDM momentum fed zeros after a unit value) is above 1/2
    after floor(tau) steps and below it after ceil(tau) steps."""
    tau = half_life(beta)
    assert tau != math.floor(tau)
    o = Oracle(cfg("sgdm", (beta,)), 1, 1)
    o.u[0, 0, 0] = 1.0
    for s in range(math.ceil(tau)):
        if s == math.floor(tau):
            assert o.u[0, 0, 0] > 0.5
        o.step(s, 0.0, np.zeros((1, 1)))
    assert o.u[0, 0, 0] < 0.5
    assert half_life(0.0) == 0.0


@pytest.mark.parametrize("base,periods", [("adam", (8, (4, 16), 2)), ("adopt", (64, (16,), 16)),
                                          ("sgdm", (3, (5, 7, 2), 0)), ("adam", (0, (4,), 0)),
                                          ("adam", (1, (1, 1), 1))])
def test_comm_reduction_counts_the_averaged_vectors(base, periods):
    """The saving over DDP (one d-vector per step) equals T divided by the
    number of state vectors the schedule averages over T steps, T a common
    multiple of the periods (counted from the oracle's own sync rule)."""
    px, pu, pv = periods
    c = cfg(base, tuple([0.9] * len(pu)), bias=False)
    c.update(period_x=px, period_u=list(pu), period_v=pv)
    T = 1
    for k in (px, pv, *pu):
        if k > 0:
            T = T * k // math.gcd(T, k)
    T *= 3
    o = Oracle(c, 2, 1)
    vectors = sum(bin(o.due_before_step(t)).count("1") for t in range(1, T + 1))
    assert comm_reduction(c) == pytest.approx(T / vectors, rel=1e-14)
    if periods == (1, (1, 1), 1):
        assert comm_reduction(c) == pytest.approx(1.0 / 4)     # every state every step
    none = cfg(base, (0.9,), bias=False)
    assert comm_reduction(none) == math.inf

# ------------------------------------------------------------- Adam pins

def test_adam_constant_gradient_bias_corrected():
    """Constant g, bias correction on: every corrected momentum equals g and
    v-hat equals g^2, so Delta_t = g / (|g| + eps) for any N and omega."""
    c = cfg("adam", (0.5, 0.9, 0.999), omega=(0.2, 0.3, 0.4))
    rng = np.random.default_rng(5)
    M, n, T = 3, 50, 40
    g = rng.standard_normal((M, n)) * np.logspace(-5, 0, n)
    x0 = rng.standard_normal(n) * 0.02
    lrs = 1e-3 * (1 + rng.random(T))
    o = Oracle(c, M, n, x0=x0)
    for t in range(T):
        o.step(t, lrs[t], g)
    expect = x0[None, :] - lrs.sum() * g / (np.abs(g) + 1e-8)
    assert np.max(np.abs(o.x - expect)) < 1e-13


def test_adam_constant_gradient_no_bias_correction():
    """Literal Algorithm 1: Delta_t = [(1-sum w) + sum w_j (1-b_j^(t+1))] g /
    (|g| sqrt(1-b2^(t+1)) + eps); each omega_j pairs with its own beta_j."""
    betas, om = (0.5, 0.9, 0.999), (0.1, 0.25, 0.6)
    c = cfg("adam", betas, omega=om, bias=False, eps=1e-6)
    rng = np.random.default_rng(6)
    M, n, T = 2, 40, 30
    g = rng.standard_normal((M, n)) * np.logspace(-3, 0, n)
    x0 = rng.standard_normal(n)
    o = Oracle(c, M, n, x0=x0)
    x = np.broadcast_to(x0, (M, n)).copy()
    for t in range(T):
        o.step(t, 1e-2, g)
        w = (1 - sum(om)) + sum(o_ * (1 - b ** (t + 1)) for o_, b in zip(om, betas))
        x = x - 1e-2 * w * g / (np.abs(g) * math.sqrt(1 - 0.999 ** (t + 1)) + 1e-6)
    assert rel(o.x, x) < 1e-12


def _torch_adam_run(betas, eps, g_seq, x0):
    p = torch.nn.Parameter(torch.tensor(x0, dtype=torch.float64))
    opt = torch.optim.Adam([p], lr=1e-3, betas=betas, eps=eps, weight_decay=0.0,
                           foreach=False, fused=False)
    for t, g in enumerate(g_seq):
        opt.param_groups[0]["lr"] = 1e-3 * (1 + 0.01 * t)
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
    st = opt.state[p]
    return p.detach().numpy(), st["exp_avg"].numpy(), st["exp_avg_sq"].numpy()


@pytest.mark.parametrize("case", ["n1_omega1", "omega0", "qhm_beta0"])
def test_adam_reduces_to_torch_adam(case):
    """Reductions to the base optimizer: N=1, omega=1 is Adam; omega=0 (any
    N) is Adam with beta_1=0; beta_1=0 makes u = g (QHM special case)."""
    rng = np.random.default_rng(7)
    M, n, T = 2, 33, 25
    gs = rng.standard_normal((T, M, n)) * 1e-2
    x0 = rng.standard_normal(n) * 0.02
    if case == "n1_omega1":
        c, tb1 = cfg("adam", (0.9,), omega=(1.0,), beta2=0.99), 0.9
    elif case == "omega0":
        c, tb1 = cfg("adam", (0.9, 0.99), omega=(0.0, 0.0), beta2=0.99), 0.0
    else:
        c, tb1 = cfg("adam", (0.0,), omega=(0.6,), beta2=0.99), 0.0
    o = Oracle(c, M, n, x0=x0)
    for t in range(T):
        o.step(t, 1e-3 * (1 + 0.01 * t), gs[t])
    for m in range(M):
        xp, ea, eas = _torch_adam_run((tb1, 0.99), 1e-8, gs[:, m], x0)
        assert rel(o.x[m], xp) < 1e-12
        assert rel(o.v[m], eas) < 1e-12
        if case == "n1_omega1":
            assert rel(o.u[0, m], ea) < 1e-12
        if case == "qhm_beta0":
            assert rel(o.u[0, m], gs[-1, m]) < 1e-15


def test_local_adam_recovery():
    """N=1, omega=1 and equal periods recovers Local Adam (section 2.3): M
    Adam workers whose parameters and both moments are averaged every H
    steps."""
    rng = np.random.default_rng(8)
    M, n, T, H = 3, 17, 12, 4
    gs = rng.standard_normal((T, M, n)) * 1e-2
    x0 = rng.standard_normal(n) * 0.02
    c = cfg("adam", (0.9,), omega=(1.0,), beta2=0.99, px=H, pu=H, pv=H)
    o = Oracle(c, M, n, x0=x0)
    ps = [torch.nn.Parameter(torch.tensor(x0, dtype=torch.float64)) for _ in range(M)]
    opts = [torch.optim.Adam([p], lr=1e-3, betas=(0.9, 0.99), eps=1e-8, foreach=False)
            for p in ps]
    for t in range(T):
        o.step(t, 1e-3, gs[t])
        for m in range(M):
            ps[m].grad = torch.tensor(gs[t, m], dtype=torch.float64)
            opts[m].step()
        if (t + 1) % H == 0:
            with torch.no_grad():
                for key in ("exp_avg", "exp_avg_sq"):
                    mean = sum(opts[m].state[ps[m]][key] for m in range(M)) / M
                    for m in range(M):
                        opts[m].state[ps[m]][key].copy_(mean)
                mean = sum(p.detach() for p in ps) / M
                for p in ps:
                    p.copy_(mean)
    o.settle(T)
    for m in range(M):
        assert rel(o.x[m], ps[m].detach().numpy()) < 1e-12
        assert rel(o.u[0, m], opts[m].state[ps[m]]["exp_avg"].numpy()) < 1e-12
        assert rel(o.v[m], opts[m].state[ps[m]]["exp_avg_sq"].numpy()) < 1e-12


def test_global_norm_clip():
    """clip(g, rho): unchanged when ||g|| <= rho; otherwise g-hat =
    rho g/(||g||+1e-6).  Momenta use g-hat, v the raw gradient."""
    rng = np.random.default_rng(9)
    n = 200
    g_small = rng.standard_normal((1, n))
    g_small *= 0.5 / np.linalg.norm(g_small)
    c_clip = cfg("adam", (0.9, 0.99), clip="global_norm", rho=1.0)
    c_none = cfg("adam", (0.9, 0.99))
    a, b = Oracle(c_clip, 1, n), Oracle(c_none, 1, n)
    a.step(0, 1e-3, g_small)
    b.step(0, 1e-3, g_small)
    assert np.array_equal(a.x, b.x) and np.array_equal(a.u, b.u)

    g_big = g_small * 1e3
    a = Oracle(c_clip, 1, n)
    a.step(0, 1e-3, g_big)
    nrm = np.linalg.norm(g_big)
    g_hat = g_big / (nrm + 1e-6)
    assert abs(grad_norm(g_big) - nrm) < 1e-12 * nrm
    assert rel(a.u[0], (1 - 0.9) * g_hat) < 1e-12
    assert rel(a.u[1], (1 - 0.99) * g_hat) < 1e-12
    assert rel(a.v, (1 - 0.999) * g_big ** 2) < 1e-12


def test_sgdm_constant_gradient_closed_form():
    """Algorithm 3 under a constant gradient: u_j(t) = (1-beta_j^(t+1)) g, so
    Delta_t = [(1 - sum w) + sum w_j (1-beta_j^(t+1))] g, unnormalised."""
    betas, om = (0.5, 0.9, 0.99), (0.2, 0.3, 0.4)
    c = cfg("sgdm", betas, omega=om)
    rng = np.random.default_rng(15)
    M, n, T = 2, 30, 25
    g = rng.standard_normal((M, n))
    x0 = rng.standard_normal(n)
    o = Oracle(c, M, n, x0=x0)
    x = np.broadcast_to(x0, (M, n)).copy()
    for t in range(T):
        lr = 0.01 * (1 + 0.1 * t)
        o.step(t, lr, g)
        w = (1 - sum(om)) + sum(o_ * (1 - b ** (t + 1)) for o_, b in zip(om, betas))
        x = x - lr * w * g
    assert np.max(np.abs(o.x - x)) < 1e-13


# ------------------------------------------------------------ ADOPT pins

@pytest.mark.parametrize("clip", ["elementwise", "none"])
def test_adopt_constant_gradient_closed_form(clip):
    """Algorithm 2 under a constant gradient: v_t = (1-b2^(t+1)) g^2, the
    normalised gradient is g / (|g| sqrt(1-b2^(t+1)) + eps), clamped to
    +-(t+1)^(1/4); each u_j is the finite EMA sum of that known sequence."""
    betas, om = (0.9, 0.999), (0.3, 0.5)
    b2, eps = 0.9999, 1e-8
    c = cfg("adopt", betas, omega=om, beta2=b2, eps=eps, bias=False, clip=clip)
    rng = np.random.default_rng(10)
    M, n, T = 2, 24, 30
    g = rng.standard_normal((M, n)) * np.logspace(-4, 0, n)
    x0 = rng.standard_normal(n)
    lrs = 2.0 ** -8 * (1 + 0.05 * np.arange(T))
    o = Oracle(c, M, n, x0=x0)
    gt_hist = []
    x = np.broadcast_to(x0, (M, n)).copy()
    for t in range(T):
        o.step(t, lrs[t], g)
        gh = g / (np.abs(g) * math.sqrt(1 - b2 ** (t + 1)) + eps)
        if clip == "elementwise":
            ct = (t + 1) ** 0.25
            gh = np.clip(gh, -ct, ct)
        gt_hist.append(gh)
        us = [sum((1 - b) * b ** (t - k) * gt_hist[k] for k in range(t + 1)) for b in betas]
        delta = (1 - sum(om)) * gh + sum(w * u for w, u in zip(om, us))
        x = x - lrs[t] * delta
        for j in range(2):
            assert rel(o.u[j], us[j]) < 1e-12
    assert rel(o.x, x) < 1e-12
    if clip == "elementwise":
        assert abs(adopt_clip_bound(15) - 2.0) < 1e-15


@pytest.mark.parametrize("clip", ["elementwise", "none"])
def test_adopt_original_ordering_closed_form(clip):
    """adopt_prev_v: step 0 sets v = g_0^2 and moves nothing else; step t >= 1
    normalises with the previous v, v_{t-1} = b2^(t-1) g_0^2 + (1 - b2^(t-1)) g^2
    for a gradient g_0 then constant g, and clamps to +-t^(1/4) at the t-th
    update.  A small g_0 makes the clamp bind."""
    betas, om = (0.9, 0.99), (0.4, 0.5)
    b2, eps = 0.9999, 1e-8
    c = cfg("adopt", betas, omega=om, beta2=b2, eps=eps, bias=False, clip=clip)
    c["adopt_prev_v"] = True
    rng = np.random.default_rng(17)
    M, n, T = 2, 16, 20
    g = rng.standard_normal((M, n)) * np.logspace(-4, 1, n)
    g0 = 1e-3 * g
    x0 = rng.standard_normal(n)
    o = Oracle(c, M, n, x0=x0)
    o.step(0, 0.1, g0)
    assert np.array_equal(o.v, g0 * g0) and np.all(o.u == 0) and np.all(o.x == x0[None, :])
    x = np.broadcast_to(x0, (M, n)).copy()
    hist = []
    for t in range(1, T):
        o.step(t, 0.01, g)
        v_prev = b2 ** (t - 1) * g0 * g0 + (1 - b2 ** (t - 1)) * g * g
        gh = g / (np.sqrt(v_prev) + eps)
        if clip == "elementwise":
            gh = np.clip(gh, -t ** 0.25, t ** 0.25)
        hist.append(gh)
        us = [sum((1 - b) * b ** (len(hist) - 1 - k) * hist[k] for k in range(len(hist))) for b in betas]
        x = x - 0.01 * ((1 - sum(om)) * gh + sum(w * u for w, u in zip(om, us)))
        assert rel(o.v, b2 ** t * g0 * g0 + (1 - b2 ** t) * g * g) < 1e-12
    assert rel(o.x, x) < 1e-11
    if clip == "elementwise":
        assert np.max(np.abs(hist[0])) == 1.0          # the clamp bound at the first update


# ------------------------------------------------------------- sync pins

def test_sync_identity_on_identical_workers():
    rng = np.random.default_rng(11)
    for M in (1, 2, 3, 4, 7, 8):
        c = cfg("adam", (0.9, 0.99), px=1, pu=1, pv=1)
        o = Oracle(c, M, 40)
        base = rng.standard_normal((3 + 1, 40)).astype(np.float32).astype(np.float64)
        o.x[:] = base[0]
        o.u[0][:] = base[1]
        o.u[1][:] = base[2]
        o.v[:] = np.abs(base[3])
        before = o.states()
        o.sync(0b1111)
        after = o.states()
        for k in before:
            assert np.array_equal(before[k], after[k]), (M, k)


def test_sync_mean_brute_force_and_invariants():
    rng = np.random.default_rng(12)
    M, n = 5, 101
    c = cfg("adam", (0.9, 0.99))
    o = Oracle(c, M, n)
    o.x[:] = rng.standard_normal((M, n))
    o.u[0][:] = rng.standard_normal((M, n))
    o.u[1][:] = rng.standard_normal((M, n))
    o.v[:] = rng.random((M, n))
    before = o.states()
    o.sync(0b0101)                 # x and u2 only
    after = o.states()
    for k in ("x", "u2"):
        assert np.allclose(after[k], np.mean(before[k], axis=0)[None, :], rtol=1e-15, atol=0)
        assert np.allclose(after[k].sum(0), before[k].sum(0), rtol=1e-13, atol=1e-14)
    for k in ("u1", "v"):
        assert np.array_equal(after[k], before[k])
    again = o.states()
    o.sync(0b0101)
    for k, a in o.states().items():
        assert np.array_equal(a, again[k])      # idempotent


def test_sync_mean_of_non_finite_values():
    """The worker mean E_m[s] = sum_m s_m / M under IEEE arithmetic: a column
    that holds infinities of one sign averages to that infinity, both signs
    or a NaN give NaN, finite columns are the numpy mean.  (The GPU's
    compensated mean falls back to this plain sum where it would give NaN.)"""
    M, n = 4, 6
    c = cfg("adam", (0.9,))
    o = Oracle(c, M, n)
    vals = np.arange(M * n, dtype=np.float64).reshape(M, n) / 7.0
    vals[3, 0] = np.inf
    vals[1, 1] = -np.inf
    vals[0, 2], vals[3, 2] = np.inf, -np.inf
    vals[2, 3] = np.nan
    vals[:, 4] = -np.inf
    o.x[:] = vals
    o.sync(0b1)
    got = o.states()["x"]
    assert np.all(got == got[0:1]) or np.all(np.isnan(got) == np.isnan(got[0:1]))
    row = got[0]
    assert row[0] == np.inf and row[1] == -np.inf and np.isnan(row[2]) and np.isnan(row[3])
    assert row[4] == -np.inf and row[5] == pytest.approx(vals[:, 5].mean(), rel=1e-15)


@pytest.mark.parametrize("bad", [np.nan, np.inf, -np.inf])
def test_adopt_original_ordering_step0_with_non_finite_gradient(bad):
    """adopt_prev_v: step 0 only sets v = g_0^2, so a non-finite g_0 reaches
    v alone (inf^2 = inf, nan^2 = nan); u stays 0 and x stays x_0."""
    c = cfg("adopt", (0.9, 0.99), omega=(0.4, 0.5), beta2=0.9999, bias=False)
    c["adopt_prev_v"] = True
    M, n = 2, 8
    x0 = np.linspace(-1.0, 1.0, n)
    o = Oracle(c, M, n, x0=x0)
    g0 = np.full((M, n), 0.5)
    g0[1, 3] = bad
    o.step(0, 0.1, g0)
    assert np.all(o.u == 0) and np.all(o.x == x0[None, :])
    v = o.v
    assert (np.isnan(v[1, 3]) if np.isnan(bad) else v[1, 3] == np.inf)
    mask = np.ones((M, n), bool)
    mask[1, 3] = False
    assert np.all(v[mask] == 0.25)


def test_per_state_periods_counts():
    """H_x=64, H_u=H_v=16 over T=512 steps: x averaged 8 times, u and v 32."""
    c = cfg("adopt", (0.95, 0.999), beta2=0.9999, bias=False, px=64, pu=16, pv=16)
    o = Oracle(c, 2, 1)
    counts = np.zeros(4, int)
    for t in range(1, 513):
        mask = o.due_before_step(t)
        for s in range(4):
            counts[s] += (mask >> s) & 1
    assert counts.tolist() == [8, 32, 32, 32]
    lit = cfg("adopt", (0.95, 0.999), px=64, pu=16, pv=16, phase="alg2_literal", bias=False)
    ol = Oracle(lit, 2, 1)
    counts[:] = 0
    for t in range(512):
        mask = ol.due_after_step(t)
        for s in range(4):
            counts[s] += (mask >> s) & 1
    assert counts.tolist() == [8, 32, 32, 32]
    assert ol.due_after_step(0) == 0b1110 and ol.due_after_step(63) == 0b0001


def test_momentum_only_sync_leaves_parameters_apart():
    rng = np.random.default_rng(13)
    M, n = 4, 30
    c = cfg("adam", (0.9,), omega=(0.9,), px=64, pu=16, pv=16)
    o = Oracle(c, M, n, x0=rng.standard_normal(n))
    for t in range(16):
        o.step(t, 1e-3, rng.standard_normal((M, n)))
    o.settle(16)
    assert np.all(np.ptp(o.u[0], axis=0) == 0) and np.all(np.ptp(o.v, axis=0) == 0)
    assert np.all(np.ptp(o.x, axis=0) > 0)


def test_sgdm_model_sync_equals_momentum_sync():
    """Section 3: syncing only the model every step is equivalent to syncing
    only the momenta every step; both follow DDP-SGDM on the mean gradient
    for the worker-averaged iterate."""
    rng = np.random.default_rng(14)
    M, n, T = 4, 25, 20
    gs = rng.standard_normal((T, M, n))
    x0 = rng.standard_normal(n)
    om = (0.3, 0.6)
    res = []
    for px, pu in ((1, 0), (0, 1)):
        c = cfg("sgdm", (0.9, 0.99), omega=om, px=px, pu=pu)
        o = Oracle(c, M, n, x0=x0)
        for t in range(T):
            o.step(t, 0.05, gs[t])
        o.settle(T)
        res.append(o.x.mean(axis=0))
    ddp = Oracle(cfg("sgdm", (0.9, 0.99), omega=om), 1, n, x0=x0)
    for t in range(T):
        ddp.step(t, 0.05, gs[t].mean(axis=0, keepdims=True))
    assert np.max(np.abs(res[0] - res[1])) < 1e-12
    assert np.max(np.abs(res[0] - ddp.x[0])) < 1e-12


def test_invalid_pairings_rejected():
    with pytest.raises(ValueError):
        Oracle(cfg("adopt", (0.9,), clip="global_norm"), 1, 4).step(0, 1e-3, np.zeros((1, 4)))
    with pytest.raises(ValueError):
        Oracle(cfg("adam", (0.9,), clip="elementwise"), 1, 4).step(0, 1e-3, np.zeros((1, 4)))


# ----------------------------------------------------- diagnostics pins

def test_state_stats_against_numpy_and_closed_forms():
    """Section 4.1 metrics: cross-worker variance (1/M) sum ||s_m - s_bar||^2,
    norms and the dot products of each worker with the mean."""
    from oracle.oracle import state_stats
    rng = np.random.default_rng(16)
    M, n = 5, 333
    s = rng.standard_normal((M, n))
    out = state_stats(s)
    mean = s.mean(axis=0)
    assert abs(out[0] - s.var(axis=0).sum()) < 1e-12 * out[0]
    assert abs(out[1] - np.dot(mean, mean)) < 1e-12 * out[1]
    np.testing.assert_allclose(out[2:2 + M], np.linalg.norm(s, axis=1) ** 2, rtol=1e-13)
    np.testing.assert_allclose(out[2 + M:], s @ mean, rtol=1e-12)
    # M = 2: variance = ||a - b||^2 / 4
    two = state_stats(s[:2])
    assert abs(two[0] - np.sum((s[0] - s[1]) ** 2) / 4) < 1e-12 * two[0]
    # identical workers: no variance (up to the rounding of the fp64 mean),
    # every norm and dot equals ||s||^2
    same = state_stats(np.tile(s[0], (3, 1)))
    assert 0.0 <= same[0] <= 1e-28 * same[1]
    np.testing.assert_allclose(same[1:], np.dot(s[0], s[0]), rtol=1e-14)


def test_pseudo_grad_stats_against_numpy():
    """Section 4.1 / 5.4: pseudo-gradients Delta^m = x^m - a over a round,
    their mean, cosine similarity and the relative change of the model."""
    from oracle.oracle import pseudo_grad_stats
    rng = np.random.default_rng(18)
    M, n = 4, 257
    a = rng.standard_normal(n)
    x = a[None, :] + 0.1 * rng.standard_normal((M, n)) + 0.05
    out = pseudo_grad_stats(x, a)
    loc = x - a[None, :]
    glob = x.mean(axis=0) - a
    np.testing.assert_allclose(out[:M], np.sum(loc * loc, axis=1), rtol=1e-13)
    np.testing.assert_allclose(out[M:2 * M], loc @ glob, rtol=1e-12)
    assert abs(out[2 * M] - glob @ glob) < 1e-12 * out[2 * M]
    assert abs(out[2 * M + 1] - a @ a) < 1e-13 * out[2 * M + 1]
    # all workers moved identically: every cosine is 1, mean move = each move
    same = pseudo_grad_stats(np.tile(x[0], (3, 1)), a)
    np.testing.assert_allclose(same[3:6] / np.sqrt(same[:3] * same[6]), 1.0, rtol=1e-12)
