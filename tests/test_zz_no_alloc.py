"""mtdao_grad_sqnorm_static: the per-replica gradient sum of squares for
callers that cannot allocate device memory (their memory is reserved by
another allocator, an allocation would synchronise a latency-critical loop,
or they hold no handle because creating one allocates).

The entry point keeps its partial sums in a fixed static device array.  This
test calls it through the C ABI twice in a row on different inputs (different
M, dtype and size, so the second call runs over slots the first one left
behind) and checks each result against the handle-based mtdao_grad_sqnorm:
both run the same grid in the same order, so the results must be equal bit
for bit; both are also checked against an fp64 sum of squares with the
tolerance the other norm tests use (1e-6 relative).  It also checks that a
repeated call leaves the device's free memory unchanged and that sizes
beyond the limits and a misaligned output are rejected.  Kept in a file that
pytest collects last.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from parity_util import host_grads, workload_dict
from synth import workloads as W

pytestmark = pytest.mark.gpu

TOL = 1e-6


def _grads(shapes, M, gdt, sigma, seed):
    w = workload_dict(shapes, M, sigma=sigma, gdt=gdt)
    lay = W.layout(shapes)
    g = host_grads(w, lay, seed, 0, np.arange(lay["n_padded"]))
    t = torch.from_numpy(g).cuda()
    if gdt == "bf16":
        t = t.to(torch.bfloat16)
    return w, lay["n_padded"], g, t


def test_static_scratch_norm_matches_handle_version():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2510_05361_gb300 as P
    P.load()
    stream = torch.cuda.current_stream().cuda_stream
    cases = [([70000, 3, 1000], 3, "f32", 0.5, 11),
             ([12288, 5], 8, "bf16", 2.0, 12)]
    for shapes, M, gdt, sigma, seed in cases:
        w, n, g_host, g = _grads(shapes, M, gdt, sigma, seed)
        dt = P.BF16 if gdt == "bf16" else P.F32
        eng = P.MTDAO(w["opt"], M, shapes)
        ref = torch.zeros(M, dtype=torch.float64, device="cuda")
        P.mtdao_grad_sqnorm(eng.h, g.data_ptr(), dt, ref.data_ptr())
        out = torch.full((M,), float("nan"), dtype=torch.float64, device="cuda")
        P.mtdao_grad_sqnorm_static(g.data_ptr(), dt, M, n, out.data_ptr(), stream)
        torch.cuda.synchronize()
        got, want = out.cpu().numpy(), ref.cpu().numpy()
        assert np.array_equal(got.view(np.uint64), want.view(np.uint64)), (got, want)
        exact = np.sum(g_host.astype(np.float64) ** 2, axis=1)
        assert np.all(np.abs(got - exact) <= TOL * exact)

        free_before = torch.cuda.mem_get_info()[0]
        P.mtdao_grad_sqnorm_static(g.data_ptr(), dt, M, n, out.data_ptr(), stream)
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free_before
        assert np.array_equal(out.cpu().numpy(), got)
        eng.close()

    w, n, _, g = _grads([1024], 2, "f32", 1.0, 13)
    out = torch.zeros(8, dtype=torch.float64, device="cuda")
    for M, npad in ((P.MAX_REPLICAS + 1, n), (0, n), (2, 100)):
        with pytest.raises(P.MTDAOError) as e:
            P.mtdao_grad_sqnorm_static(g.data_ptr(), P.F32, M, npad, out.data_ptr(), stream)
        assert e.value.code == P.ERR_INVALID
        assert P.mtdao_last_error(None)
    # an output that is not 8-byte aligned is refused before any launch
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_grad_sqnorm_static(g.data_ptr(), P.F32, 2, n, out.data_ptr() + 4, stream)
    assert e.value.code == P.ERR_ALIGN
    torch.cuda.synchronize()
