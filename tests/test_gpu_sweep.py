"""Parity on points of the flat-vector sweep workload (n = 2^20, M in
{1,2,4,8} and four points with 12 to 64 replicas, N in {1..4}, H in
{1,8,64}, including the base-optimizer
reduction point N=1, omega=1, H=1): T = 3H local steps (8 for H = 1) with
device-generated gradients, the oracle on a sample of elements."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from parity_util import compare, oracle_run, sample_indices, state_names
from synth import workloads as W

pytestmark = pytest.mark.gpu

POINTS = ([(M, N, 8) for M in (1, 2, 4, 8) for N in (1, 2, 3, 4)]
          + [(M, 1, 1) for M in (1, 2, 4, 8)]
          + [(4, 2, 64), (8, 4, 64), (2, 3, 1)]
          + [(12, 1, 8), (16, 3, 8), (32, 2, 8), (64, 4, 1)])   # the block-staged fused step


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2510_05361_gb300 as P
    P.load()
    return P


@pytest.mark.parametrize("M,N,H", POINTS)
def test_sweep_point_parity(P, M, N, H):
    w = W.sweep_point(20, M, N, H)
    if N == 1 and H == 1:
        assert w["opt"]["omega"] == [1.0]
    run_point(P, w, M, N, H)


@pytest.mark.parametrize("M,N,H,base", [(16, 2, 4, "adopt"), (24, 3, 4, "adam"), (40, 1, 2, "sgdm")])
def test_block_staged_fused_step_bf16_many_spans(P, M, N, H, base):
    """bf16 gradients through the block-staged fused step with 2^20 elements
    per replica: every persistent block walks many spans, each span's
    gradient tile copied 8 bytes at a time while the previous one is used."""
    w = W.sweep_point(20, M, N, H, base=base)
    w["grad_dtype"] = "bf16"
    run_point(P, w, M, N, H)


def run_point(P, w, M, N, H):
    from synth.device import DeviceInputs
    lay = W.layout(w["shapes"])
    opt, T = w["opt"], w["T"]
    eng = P.MTDAO(opt, M, w["shapes"])
    dev = DeviceInputs(w, lay, W.GRAD_SEED, W.INIT_SEED)
    eng.set_params(dev.init_params())
    g = None
    for t in range(T):
        g = dev.grads(t, out=g)
        eng.step(g, opt["lr"], eng.sync_due())
    torch.cuda.synchronize()
    idx = sample_indices(lay, 2048, seed=M * 100 + N * 10 + H)
    idx_t = torch.from_numpy(idx).cuda()
    got = {nm: eng.state_view(s)[:, idx_t].cpu().numpy() for s, nm in enumerate(state_names(opt))}
    eng.close()
    compare(got, oracle_run(opt, M, idx, T, lay, w, W.GRAD_SEED, W.INIT_SEED))
