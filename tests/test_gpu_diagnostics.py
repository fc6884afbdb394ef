"""Sync with diagnostics (mtdao_sync_stats) against the oracle's definitions
of the paper's cross-worker metrics (section 4.1), and bit-equality of the
averaged states with the plain sync."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle.oracle import state_stats
from parity_util import workload_dict

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2510_05361_gb300 as P
    P.load()
    return P


def _fill(eng, rng, spread):
    vals = {}
    for s in range(eng.n_states):
        common = rng.standard_normal(eng.n_padded).astype(np.float32)
        arr = (common[None, :] + spread * rng.standard_normal((eng.M, eng.n_padded))).astype(np.float32)
        if s == eng.n_states - 1:
            arr = np.abs(arr)
        eng.state_view(s).copy_(torch.from_numpy(arr).cuda())
        vals[s] = arr
    return vals


@pytest.mark.parametrize("M", [1, 2, 3, 4, 8, 9, 16, 32, 33, 37, 64, 65, 100, 256, 300, 1024])
def test_sync_stats_match_oracle_and_plain_sync(P, M):
    """M <= 8: one pass with the replicas in registers; 9 <= M <= 64: one
    pass with a span of all replicas staged in shared memory (four-column
    means up to 32); M > 64: two passes through a scratch mean.  All match the oracle's definitions and
    leave the states bit-identical to the plain average."""
    shapes = [70001, 999, 4096] if M <= 37 else [7001, 99, 1024]
    w = workload_dict(shapes, M, betas=(0.9, 0.99))
    a = P.MTDAO(w["opt"], M, shapes)
    b = P.MTDAO(w["opt"], M, shapes)
    rng = np.random.default_rng(M)
    vals = _fill(a, rng, spread=0.05)
    for s, arr in vals.items():
        b.state_view(s).copy_(torch.from_numpy(arr).cuda())
    mask = 0b1101                                 # x, u2, v
    stats = a.sync_stats(mask).cpu().numpy()
    b.sync(mask)
    again = P.MTDAO(w["opt"], M, shapes)
    for s, arr in vals.items():
        again.state_view(s).copy_(torch.from_numpy(arr).cuda())
    stats2 = again.sync_stats(mask).cpu().numpy()
    torch.cuda.synchronize()
    assert np.array_equal(stats, stats2)          # fixed-order sums
    sel = [s for s in range(a.n_states) if (mask >> s) & 1]
    assert stats.shape == (len(sel), 2 + 2 * M)
    for row, s in zip(stats, sel):
        ref = state_stats(vals[s].astype(np.float64))
        err = np.abs(row - ref) / np.maximum(np.abs(ref), 1e-30)
        assert np.all(err[1:] <= 1e-5), (s, err)
        if M > 1:
            assert err[0] <= 1e-5, (s, err[0])
        else:
            assert row[0] == 0.0
    for s in range(a.n_states):
        ga = a.state_view(s).cpu().numpy()
        gb = b.state_view(s).cpu().numpy()
        assert np.array_equal(ga.view(np.uint32), gb.view(np.uint32)), s
    for e in (a, b, again):
        e.close()


@pytest.mark.parametrize("M", [4, 12, 40])
def test_one_pass_diagnostics_over_many_spans(P, M):
    """Large lists: the one-pass diagnostics for 9 <= M <= 64 run a
    persistent grid whose blocks take many spans each (2^21 elements), the
    next span's copy in flight while the current one is summed; for M = 4
    the sync diagnostics run 264 tile blocks per state, so the finalize adds
    runs of block rows per thread, and the pseudo-gradient pass runs its
    whole persistent grid.  Sums match the oracle's definitions, the averaged
    states equal the plain average bit for bit."""
    from oracle.oracle import pseudo_grad_stats
    shapes = [1 << 25, 1 << 20] if M <= 8 else [1 << 21]
    w = workload_dict(shapes, M, betas=(0.9, 0.99))
    a = P.MTDAO(w["opt"], M, shapes)
    b = P.MTDAO(w["opt"], M, shapes)
    rng = np.random.default_rng(100 + M)
    vals = _fill(a, rng, spread=0.05)
    for s, arr in vals.items():
        b.state_view(s).copy_(torch.from_numpy(arr).cuda())
    mask = 0b111
    stats = a.sync_stats(mask).cpu().numpy()
    b.sync(mask)
    torch.cuda.synchronize()
    for row, s in zip(stats, range(3)):
        ref = state_stats(vals[s].astype(np.float64))
        err = np.abs(row - ref) / np.maximum(np.abs(ref), 1e-30)
        assert np.all(err <= 1e-5), (s, err)
    for s in range(3):
        assert np.array_equal(a.state_view(s).cpu().numpy().view(np.uint32),
                              b.state_view(s).cpu().numpy().view(np.uint32)), s
    # pseudo-gradients of x against an anchor (its current value), after moving x
    a.track_anchor(0b1)
    anchor = a.state_view(0)[0].cpu().numpy().astype(np.float64)
    moved = (a.state_view(0) + 0.01 * torch.randn((M, a.n_padded), device="cuda",
                                                   generator=torch.Generator(device="cuda").manual_seed(M)))
    a.state_view(0).copy_(moved)
    got = a.pseudo_grad_stats(0).cpu().numpy()
    cur = a.state_view(0).cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(got, pseudo_grad_stats(cur, anchor), rtol=1e-5)
    a.close()
    b.close()


def test_sync_stats_cosine_and_variance_during_training(P):
    """After a few local steps from a common start, the cosine between each
    worker's momentum and the mean momentum is in (0, 1] and the variance
    vanishes after the momenta are averaged."""
    M = 4
    w = workload_dict([50000], M, betas=(0.9,), px=0, pu=0, pv=0)
    eng = P.MTDAO(w["opt"], M, w["shapes"])
    eng.set_params(torch.zeros(eng.n_padded, device="cuda"))
    gen = torch.Generator(device="cuda").manual_seed(3)
    common = torch.randn(eng.n_padded, device="cuda", generator=gen)
    for t in range(8):
        g = common[None, :] + 0.5 * torch.randn((M, eng.n_padded), device="cuda", generator=gen)
        eng.step(g.contiguous(), 1e-3, 0)
    st = eng.sync_stats(0b10).cpu().numpy()[0]     # u1
    cos = st[2 + M:] / np.sqrt(st[2:2 + M] * st[1])
    assert np.all(cos > 0.5) and np.all(cos <= 1.0 + 1e-6)
    assert st[0] > 0
    st2 = eng.sync_stats(0b10).cpu().numpy()[0]
    assert st2[0] <= 1e-10 * st2[1]
    eng.close()


def test_sync_stats_rejects_bad_masks(P):
    out = torch.zeros(64, dtype=torch.float64, device="cuda")
    w = workload_dict([1024], 2, betas=(0.9,))
    eng = P.MTDAO(w["opt"], 2, w["shapes"])
    with pytest.raises(P.MTDAOError):
        P.mtdao_sync_stats(eng.h, 1 << 7, out.data_ptr())
    eng.close()


@pytest.mark.parametrize("M", [2, 4, 8, 9, 16, 32, 33, 37, 64, 65, 256, 300, 1024])
def test_pseudo_grad_stats_against_oracle(P, M):
    """Anchor = parameters at the last average; mid-round diagnostics of the
    pseudo-gradients match the oracle's definitions on the same values."""
    from oracle.oracle import pseudo_grad_stats
    w = workload_dict([40000, 123], M, betas=(0.9, 0.999), px=8, pu=4, pv=8)
    eng = P.MTDAO(w["opt"], M, w["shapes"])
    eng.set_params(torch.randn(eng.n_padded, device="cuda") * 0.02)
    eng.track_anchor(0b011)                           # x and u1
    gen = torch.Generator(device="cuda").manual_seed(M)
    common = torch.randn(eng.n_padded, device="cuda", generator=gen)

    def step():
        g = common[None, :] + torch.randn((M, eng.n_padded), device="cuda", generator=gen)
        eng.step(g.contiguous(), 1e-3)

    for _ in range(8):
        step()                                        # x and u1 averaged at the end of step 8
    at_sync = eng.pseudo_grad_stats(0).cpu().numpy()
    assert np.all(at_sync[:M] == 0) and at_sync[2 * M] == 0 and at_sync[2 * M + 1] > 0
    anchors = {s: eng.state_view(s)[0].cpu().numpy().astype(np.float64) for s in (0, 1)}
    for _ in range(3):
        step()                                        # steps 9-11: no average due
    for s in (0, 1):
        got = eng.pseudo_grad_stats(s).cpu().numpy()
        cur = eng.state_view(s).cpu().numpy().astype(np.float64)
        np.testing.assert_allclose(got, pseudo_grad_stats(cur, anchors[s]), rtol=1e-5)
        cos = got[M:2 * M] / np.sqrt(got[:M] * got[2 * M])
        assert np.all(cos > 0.3) and np.all(cos <= 1.0 + 1e-6)
    step()                                            # step 12 averages u1: new u1 anchor
    assert np.all(eng.pseudo_grad_stats(1).cpu().numpy()[:M] == 0)
    with pytest.raises(P.MTDAOError):
        eng.pseudo_grad_stats(2)                      # u2 has no anchor
    eng.close()


def test_pseudo_grad_stats_needs_an_anchor(P):
    w = workload_dict([1024], 2, betas=(0.9,))
    eng = P.MTDAO(w["opt"], 2, w["shapes"])
    out = torch.zeros(8, dtype=torch.float64, device="cuda")
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_pseudo_grad_stats(eng.h, 0, out.data_ptr())
    assert e.value.code == P.ERR_STATE
    eng.track_anchor(0b1)
    eng.track_anchor(0)
    with pytest.raises(P.MTDAOError):
        P.mtdao_pseudo_grad_stats(eng.h, 0, out.data_ptr())
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_track_anchor(eng.h, 1 << 5)
    assert e.value.code == P.ERR_INVALID
    eng.close()
