"""End-to-end use of the library as the optimizer of a small model: M = 4
workers train one MLP each on their own synthetic data shards (a fixed
teacher network plus noise), with the parameters living in the library's
arena (tensor views, no copies) and the gradients written in place into a
[M][n_padded] buffer.  Checks that the workers' loss falls well below its
starting value, that the parameters are bit-identical across workers after
every step that averages them, and that the padding stays zero.  The
optimizer arithmetic itself is checked against the oracle elsewhere; this
test covers the integration (layout, views, schedule, streams)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

SHAPES = [(64, 32), (64,), (8, 64), (8,)]          # W1, b1, W2, b2


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2510_05361_gb300 as P
    P.load()
    return P


def forward(params, x):
    w1, b1, w2, b2 = params
    return torch.tanh(x @ w1.T + b1) @ w2.T + b2


@pytest.mark.parametrize("base", ["adam", "adopt"])
def test_workers_train_a_small_model(P, base):
    M, T, batch = 4, 400, 128
    numels = [int(np.prod(s)) for s in SHAPES]
    opt = {"base": base, "n_mom": 2, "beta1": [0.9, 0.999], "omega": [0.475, 0.475],
           "beta2": 0.999 if base == "adam" else 0.9999, "eps": 1e-8,
           "bias_correction": base == "adam", "clip_mode": "none",
           "period_x": 16, "period_u": [8, 16], "period_v": 16, "sync_phase": "alg1"}
    lr = 3e-3 if base == "adam" else 2.0 ** -8
    eng = P.MTDAO(opt, M, numels)
    gen = torch.Generator(device="cpu").manual_seed(7)
    x0 = torch.zeros(eng.n_padded)
    for v, shp in zip(eng.tensor_views(x0, SHAPES), SHAPES):
        v.copy_(torch.randn(shp, generator=gen) * (0.5 / np.sqrt(shp[-1])))
    eng.set_params(x0.cuda())
    teacher = [torch.randn(s, generator=gen).cuda() * (1.0 / np.sqrt(s[-1])) for s in SHAPES]

    grads = torch.zeros((M, eng.n_padded), device="cuda")
    gviews = [eng.tensor_views(grads[m], SHAPES) for m in range(M)]
    xs = eng.state_view(0)
    pviews = [eng.tensor_views(xs[m], SHAPES) for m in range(M)]
    inside = torch.zeros(eng.n_padded, dtype=torch.bool, device="cuda")
    for off, k in zip(eng.offsets, numels):
        inside[off:off + k] = True

    data_gen = [torch.Generator(device="cuda").manual_seed(100 + m) for m in range(M)]
    probe = torch.randn((1024, 32), device="cuda", generator=torch.Generator(device="cuda").manual_seed(1))
    target = forward(teacher, probe)

    def probe_loss(m):
        with torch.no_grad():
            return float(torch.mean((forward(pviews[m], probe) - target) ** 2))

    start = [probe_loss(m) for m in range(M)]
    for t in range(T):
        for m in range(M):
            xb = torch.randn((batch, 32), device="cuda", generator=data_gen[m])
            yb = forward(teacher, xb) + 0.05 * torch.randn((batch, 8), device="cuda", generator=data_gen[m])
            params = [p.detach().requires_grad_() for p in pviews[m]]   # share the arena's memory
            loss = torch.mean((forward(params, xb) - yb) ** 2)
            for gv, g in zip(gviews[m], torch.autograd.grad(loss, params)):
                gv.copy_(g)
        mask = eng.step(grads, lr)
        if mask & 1:
            torch.cuda.synchronize()
            assert torch.equal(xs[1:], xs[:1].expand(M - 1, -1)), t       # bit-identical workers
    torch.cuda.synchronize()
    assert int((xs[:, ~inside] != 0).sum()) == 0                          # padding untouched
    end = [probe_loss(m) for m in range(M)]
    assert all(e < 0.1 * s for s, e in zip(start, end)), (start, end)
    eng.close()
