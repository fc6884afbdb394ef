"""The C ABI used from C: tests/c/abi_program.c is compiled as strict C99
against include/mtdao.h alone (no CUDA headers, no C++) and linked against
libmtdao.so.  Its host-only results must equal the Python binding's; on a
GPU, its run through the host-gradient entry point must reproduce the
binding's device-path run bit for bit."""
import os
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c", "abi_program.c")


@pytest.fixture(scope="module")
def P():
    from paper_2510_05361_gb300 import build
    build.build()
    import paper_2510_05361_gb300 as P
    P.load()
    return P


@pytest.fixture(scope="module")
def program(P, tmp_path_factory):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    libdir = os.path.dirname(P.LIB_PATH)
    exe = str(tmp_path_factory.mktemp("abi") / "abi_program")
    subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic",
                    "-I", os.path.join(ROOT, "include"), SRC, "-o", exe,
                    "-L", libdir, "-lmtdao", "-Wl,-rpath," + libdir], check=True)
    return exe


def test_c_program_host_calls_match_the_binding(P, program):
    out = subprocess.run([program, "host"], capture_output=True, text=True, check=True).stdout
    got = dict(line.split(" ", 1) for line in out.strip().splitlines())
    assert int(got["version"]) == P.mtdao_version()
    cfg = P.mtdao_config_default(0, 2)
    assert int(got["num_states"]) == P.mtdao_num_states(cfg)
    offs, npad = P.mtdao_plan_layout([1000, 7, 4096])
    assert [int(v) for v in got["layout"].split()] == offs + [npad]
    cfg.period_x, cfg.period_u[0], cfg.period_u[1], cfg.period_v = 6, 2, 3, 4
    assert [int(v) for v in got["masks"].split()] == [P.mtdao_due_mask(cfg, t) for t in range(12)]
    assert float(got["half_life"]) == P.mtdao_half_life(0.999)
    P.mtdao_config_half_life_periods(cfg, 32)
    assert [int(v) for v in got["half_life_periods"].split()] == [cfg.period_x, cfg.period_u[0],
                                                                   cfg.period_u[1], cfg.period_v]
    assert float(got["comm_reduction"]) == P.mtdao_comm_reduction(cfg)
    assert int(got["invalid"]) == P.ERR_INVALID


@pytest.mark.gpu
def test_c_program_run_matches_the_binding(P, program, tmp_path):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from parity_util import host_grads
    from synth import generators as G
    from synth import workloads as W
    shapes, M, T = [1000, 7, 4096, 333], 4, 9
    w = {"grad_kind": "normal", "grad_sigma": 0.01, "grad_dtype": "f32", "init_sigma": 0.02,
         "shapes": shapes, "M": M}
    lay = W.layout(shapes)
    n = lay["n_padded"]
    idx = np.arange(n)
    x0 = G.init_params(w, lay, 11, idx).astype(np.float32)
    grads = np.stack([host_grads(w, lay, 12, t, idx) for t in range(T)]).astype(np.float32)
    (tmp_path / "spec.txt").write_text("%d %d %d %s\n" % (M, T, len(shapes), " ".join(map(str, shapes))))
    x0.tofile(tmp_path / "x0.bin")
    grads.tofile(tmp_path / "grads.bin")
    r = subprocess.run([program, "run", str(tmp_path)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == "steps %d" % T

    cfg = P.mtdao_config_default(0, 2)
    opt = {"base": "adam", "n_mom": 2, "beta1": [cfg.beta1[0], cfg.beta1[1]],
           "omega": [cfg.omega[0], cfg.omega[1]], "beta2": cfg.beta2, "eps": cfg.eps,
           "bias_correction": True, "clip_mode": "none", "period_x": 4, "period_u": [4, 4],
           "period_v": 4, "sync_phase": "alg1"}
    eng = P.MTDAO(opt, M, shapes)
    eng.set_params(torch.from_numpy(x0).cuda())
    for t in range(T):
        eng.step(torch.from_numpy(grads[t]).cuda(), 1e-3)
    torch.cuda.synchronize()
    ref = np.stack([eng.state_view(s).cpu().numpy() for s in range(eng.n_states)])
    eng.close()
    got = np.fromfile(tmp_path / "states.bin", dtype=np.float32).reshape(ref.shape)
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))
