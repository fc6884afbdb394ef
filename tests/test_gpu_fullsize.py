"""Parity at the workloads' full sizes, in the configuration the benchmark
times: the library runs every element of every replica for the workload's
full T steps with device-generated gradients; the oracle recomputes a sample
of elements (random positions plus each tensor's first and last 8 elements)
for all replicas over the same T steps from the host generator.  Without
norm clipping the elements are independent, so a sample is exact.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from parity_util import LAST_REPORT, compare, oracle_run, sample_indices, state_names
from synth import workloads as W

pytestmark = pytest.mark.gpu

SEED_G, SEED_I = W.GRAD_SEED, W.INIT_SEED


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2510_05361_gb300 as P
    P.load()
    return P


def device_bytes(w):
    lay = W.layout(w["shapes"])
    opt = w["opt"]
    states = 1 + opt["n_mom"] + (0 if opt["base"] == "sgdm" else 1)
    gb = 2 if w["grad_dtype"] == "bf16" else 4
    return w["M"] * lay["n_padded"] * (4 * states + gb)


@pytest.mark.parametrize("name,n_sample", [("tiny", 1 << 15), ("gpt2_small", 1 << 14),
                                           ("decoder_350m", 4096), ("decoder_1b", 1 << 14)])
def test_full_size_sampled_parity(P, name, n_sample):
    from synth.device import DeviceInputs
    w = W.get(name)
    lay = W.layout(w["shapes"])
    if device_bytes(w) + (8 << 30) > torch.cuda.mem_get_info()[0]:
        pytest.skip("not enough free device memory for %s" % name)
    opt, M, T = w["opt"], w["M"], w["T"]
    eng = P.MTDAO(opt, M, w["shapes"])
    dev = DeviceInputs(w, lay, SEED_G, SEED_I)
    eng.set_params(dev.init_params())
    g = None
    syncs = 0
    for t in range(T):
        g = dev.grads(t, out=g)
        mask = eng.sync_due()
        syncs += mask != 0
        eng.step(g, opt["lr"], mask)
    torch.cuda.synchronize()
    assert syncs > 0
    idx = sample_indices(lay, n_sample, seed=2)
    idx_t = torch.from_numpy(idx).cuda()
    got = {nm: eng.state_view(s)[:, idx_t].cpu().numpy() for s, nm in enumerate(state_names(opt))}
    del g
    eng.close()
    ref = oracle_run(opt, M, idx, T, lay, w, SEED_G, SEED_I)
    compare(got, ref)
    print(name, {k: "%.2e (raw %.2e)" % fr for k, fr in LAST_REPORT.items()})
