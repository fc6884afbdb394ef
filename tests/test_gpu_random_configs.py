"""Seeded random configurations, GPU against the oracle: base, number of
momenta, decay rates and weights (including beta_1 = 0, beta_2 = 0 and
weights that sum to 1), epsilon from 1e-12 to 1e-3, learning rates from 0
to 0.1, gradient scales from 1e-6 to 100, periods (including 0 = never),
both sync phases, clipping modes,
the ADOPT ordering flag, gradient dtype and kind, the replica count and a
ragged tensor list (with zero-size tensors) are drawn per case; every
element of every state is compared after T steps."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from parity_util import compare, host_grads, oracle_run
from synth import generators as G
from synth import workloads as W

pytestmark = pytest.mark.gpu
SEED_G, SEED_I = 777, 778


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2510_05361_gb300 as P
    P.load()
    return P


def draw(case, replica_counts=None):
    rng = np.random.default_rng(1000 + case)
    base = ["adam", "adopt", "sgdm"][case % 3]
    N = int(rng.integers(1, 5))
    betas = [float(rng.choice([0.0, 0.1, 0.5, 0.9, 0.95, 0.99, 0.999, 0.9999])) for _ in range(N)]
    if rng.random() < 0.25:
        omega = list(rng.dirichlet(np.ones(N)))                      # sum to 1: no gradient term
        omega = [float(o) * (1 - 1e-9) for o in omega]
    else:
        omega = [float(o) for o in rng.uniform(0, 1.0 / N, N)]
    periods = lambda: int(rng.choice([0, 1, 2, 3, 5, 8]))
    clip = "none"
    if base == "adopt" and rng.random() < 0.5:
        clip = "elementwise"
    if base != "adopt" and rng.random() < 0.3:
        clip = "global_norm"
    M = int(rng.choice([1, 2, 3, 4, 5, 6, 7, 8, 9, 12, 16, 32]))
    if replica_counts is not None:
        M = int(rng.choice(replica_counts))
    shapes = [int(rng.choice([0, 1, 7, 64, 333, 1000, 4099])) for _ in range(int(rng.integers(1, 6)))]
    if sum(shapes) == 0:
        shapes.append(513)
    opt = {"base": base, "n_mom": N, "beta1": betas, "omega": omega,
           "beta2": float(rng.choice([0.0, 0.5, 0.99, 0.999, 0.9999])),
           "eps": float(rng.choice([1e-12, 1e-8, 1e-6, 1e-3])),
           "bias_correction": base == "adam" and bool(rng.random() < 0.7), "clip_mode": clip,
           "clip_rho": float(rng.choice([0.5, 1.0, 50.0])), "period_x": periods(),
           "period_u": [periods() for _ in range(N)], "period_v": periods(),
           "sync_phase": "alg2_literal" if rng.random() < 0.3 else "alg1",
           "adopt_prev_v": base == "adopt" and bool(rng.random() < 0.4),
           "lr": float(rng.choice([0.0, 1e-4, 1e-3, 2.0 ** -8, 1e-2, 0.1]))}
    w = {"name": "random", "shapes": shapes, "M": M, "grad_kind": str(rng.choice(G.KINDS)),
         "grad_sigma": float(rng.choice([1e-6, 1e-3, 0.01, 1.0, 100.0])),
         "grad_dtype": "bf16" if rng.random() < 0.4 else "f32", "init_sigma": 0.02, "opt": opt}
    return w, int(rng.integers(3, 17))


def run_case(P, w, T):
    opt, M = w["opt"], w["M"]
    lay = W.layout(w["shapes"])
    n = lay["n_padded"]
    idx = np.arange(n)
    eng = P.MTDAO(opt, M, w["shapes"])
    eng.set_params(torch.from_numpy(G.init_params(w, lay, SEED_I, idx)).cuda())
    for t in range(T):
        g = torch.from_numpy(host_grads(w, lay, SEED_G, t, idx)).cuda()
        eng.step(g.to(torch.bfloat16) if w["grad_dtype"] == "bf16" else g, opt["lr"])
    torch.cuda.synchronize()
    names = ["x"] + ["u%d" % (j + 1) for j in range(opt["n_mom"])] + ([] if opt["base"] == "sgdm" else ["v"])
    got = {nm: eng.state_view(s).cpu().numpy() for s, nm in enumerate(names)}
    eng.close()
    compare(got, oracle_run(opt, M, idx, T, lay, w, SEED_G, SEED_I))


@pytest.mark.parametrize("case", range(96))
def test_random_configuration_parity(P, case):
    run_case(P, *draw(case))


@pytest.mark.parametrize("case", range(96, 120))
def test_random_configuration_parity_wide(P, case):
    """The same draws with replica counts on both sides of the block-staged
    fused step's layout switches (10, 24, 40, 64)."""
    run_case(P, *draw(case, replica_counts=[10, 24, 40, 64]))
