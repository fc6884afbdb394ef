"""Toy objectives with gradients computed from the workers' current
parameters (the paper's quadratic 1/2 lambda x^2 of Figure 2 and the noisy
Rosenbrock function with M = 256 workers of Figure 1), driven through the
library and, independently, through the oracle with the host version of the
same objective.  The paper prints no learning rate, period or starting point
for these figures, so the runs below use stated choices and check parity,
not the figures' qualitative outcome.

Gradient point: Algorithms 1-3 write the gradient of step t as the gradient
at the worker's parameters before that step's average; the library performs
an average at the end of the step that completes a period, so gradients read
from memory are taken at the averaged parameters (as in Local SGD).  The
oracle harness below evaluates at the same point (settle, then gradient).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle.oracle import Oracle
from parity_util import compare, state_names
from synth import generators as G
from synth import workloads as W

pytestmark = pytest.mark.gpu
SEED = 424242


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2510_05361_gb300 as P
    P.load()
    return P


def opt_of(base, beta, omega, K, beta2=0.999, bias=True):
    return {"base": base, "n_mom": 1, "beta1": [beta], "omega": [omega], "beta2": beta2,
            "eps": 1e-8, "bias_correction": bias and base == "adam", "clip_mode": "none",
            "period_x": K, "period_u": [K], "period_v": K, "sync_phase": "alg1"}


def gpu_toy(P, kind, opt, M, n_real, T, lr, sigma, x0, lam=None):
    from synth import device as D
    n = W.layout([n_real])["n_padded"]
    eng = P.MTDAO(opt, M, [n_real])
    x0p = np.zeros(n, np.float32)
    x0p[:n_real] = x0
    eng.set_params(torch.from_numpy(x0p).cuda())
    lam_t = None
    if lam is not None:
        lp = np.zeros(n, np.float32)
        lp[:n_real] = lam
        lam_t = torch.from_numpy(lp).cuda()
    g = torch.empty((M, n), dtype=torch.float32, device="cuda")
    xptr = eng.state_ptr(0, 0)
    for t in range(T):
        D.toy_grad(kind, xptr, g, M, n, n_real, SEED, t, sigma, lam_t)
        eng.step(g, lr, eng.sync_due())
    torch.cuda.synchronize()
    return eng


def oracle_toy(kind, opt, M, idx, T, lr, sigma, x0, lam=None):
    o = Oracle(opt, M, len(idx), x0=np.asarray(x0, np.float64)[idx])
    lam_s = None if lam is None else np.asarray(lam, np.float64)[idx]
    for t in range(T):
        o.settle(t)                                   # averages due before step t
        g = G.toy_grad(kind, o.x, SEED, t, sigma, lam_s, idx=idx)
        o.step(t, lr, g)
    o.settle(T)
    return o.states()


@pytest.mark.parametrize("omega", [0.95, 1.0])
def test_quadratic_toy_parity(P, omega):
    """1/2 lambda x^2 with lambda log-spaced over [0.1, 30], MT-DAO-SGDM (N=1,
    beta=0.999, omega=0.95) and its omega=1 form, 8 workers, period 16."""
    M, n_real, T, lr, sigma = 8, 4096, 128, 0.05, 0.5
    lam = np.logspace(-1, np.log10(30.0), n_real).astype(np.float32)
    x0 = np.ones(n_real, np.float32)
    opt = opt_of("sgdm", 0.999, omega, 16)
    eng = gpu_toy(P, "quadratic", opt, M, n_real, T, lr, sigma, x0, lam)
    got = {nm: eng.state_view(s).cpu().numpy()[:, :n_real] for s, nm in enumerate(state_names(opt))}
    eng.close()
    ref = oracle_toy("quadratic", opt, M, np.arange(n_real), T, lr, sigma, x0, lam)
    compare(got, ref)


@pytest.mark.parametrize("omega,beta", [(0.95, 0.9999), (1.0, 0.9999), (0.95, 0.999)])
def test_rosenbrock_toy_parity_256_workers(P, omega, beta):
    """Rosenbrock pairs from (-1.2, 1) with noise sigma = 2 on M = 256
    workers, MT-DAO-Adam (N=1) and Local Adam (omega=1), period 16; the
    oracle recomputes 16 of the 256 independent problems.

    Slow momenta only: near these iterates the gradient's Lipschitz constant
    is ~10^3 (dg_a/da = 1200 a^2 - 400 b + 2), so the fp32 rounding of x
    (~4e-7) becomes a ~4e-4 difference in the gradient itself, which a fast
    EMA (beta = 0.9) passes on to u almost unfiltered (measured: u within
    8e-5, x within 4e-7).  That is the objective's conditioning, not an
    optimizer error; beta >= 0.999 averages it away."""
    M, problems, T, lr, sigma = 256, 256, 150, 3e-3, 2.0
    n_real = 2 * problems
    x0 = np.tile(np.array([-1.2, 1.0], np.float32), problems)
    opt = opt_of("adam", beta, omega, 16)
    eng = gpu_toy(P, "rosenbrock", opt, M, n_real, T, lr, sigma, x0)
    rng = np.random.default_rng(5)
    ks = np.sort(rng.choice(problems, 16, replace=False))
    idx = np.stack([2 * ks, 2 * ks + 1], axis=1).ravel()
    idx_t = torch.from_numpy(idx).cuda()
    got = {nm: eng.state_view(s)[:, idx_t].cpu().numpy() for s, nm in enumerate(state_names(opt))}
    xm = eng.state_view(0)[:, :n_real].mean(0).cpu().numpy()
    eng.close()
    ref = oracle_toy("rosenbrock", opt, M, idx, T, lr, sigma, x0)
    compare(got, ref)
    dist = np.sqrt((xm[0::2] - 1) ** 2 + (xm[1::2] - 1) ** 2)
    print("rosenbrock omega=%g beta=%g: median distance to (1,1) after %d steps: %.4f"
          % (omega, beta, T, float(np.median(dist))))
