"""CPU checks of the C ABI: the library builds/loads, exports every function
that include/mtdao.h declares, and its host-only logic (validation, layout,
sync schedule) is right.  No GPU work is launched."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle.oracle import Oracle
from synth import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mtdao.h")


@pytest.fixture(scope="module")
def P():
    from paper_2510_05361_gb300 import build
    build.build()
    import paper_2510_05361_gb300 as P
    P.load()
    return P


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mtdao_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("mtdao_create", "mtdao_step", "mtdao_sync", "mtdao_destroy"):
        assert required in names


def test_library_exports_every_declared_symbol(P):
    lib = ctypes.CDLL(P.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing
    assert P.mtdao_version() == 2


def test_layout_matches_the_published_convention(P):
    for shapes in ([1], [7, 9, 1024], W.WORKLOADS["gpt2_small"]["shapes"],
                   W.WORKLOADS["decoder_1b"]["shapes"]):
        offs, npad = P.mtdao_plan_layout(shapes)
        lay = W.layout(shapes)
        assert offs == lay["offsets"] and npad == lay["n_padded"]
        assert npad % 256 == 0 and all(o % 8 == 0 for o in offs)
    assert W.layout(W.WORKLOADS["decoder_1b"]["shapes"])["n_padded"] == 1311086592


def _opt(base="adam", betas=(0.9, 0.999), **kw):
    n = len(betas)
    opt = {"base": base, "n_mom": n, "beta1": list(betas), "omega": [0.95 / n] * n,
           "beta2": 0.999, "eps": 1e-8, "bias_correction": base == "adam", "clip_mode": "none",
           "period_x": 64, "period_u": [16] * n, "period_v": 16, "sync_phase": "alg1"}
    opt.update(kw)
    return opt


@pytest.mark.parametrize("phase", ["alg1", "alg2_literal"])
@pytest.mark.parametrize("base", ["adam", "adopt", "sgdm"])
def test_sync_schedule_matches_the_oracle(P, base, phase):
    opt = _opt(base, (0.9, 0.99, 0.5), period_x=12, period_u=[3, 0, 8], period_v=5,
               sync_phase=phase, bias_correction=(base == "adam"))
    cfg = P.make_config(opt)
    o = Oracle(opt, 2, 1)
    for t in range(200):
        lib_mask = P.mtdao_due_mask(cfg, t)
        ora_mask = o.due_before_step(t + 1) if phase == "alg1" else o.due_after_step(t)
        assert lib_mask == ora_mask, (t, lib_mask, ora_mask)


def test_paper_period_counts(P):
    """Per-state periods H_x=64, H_u=H_v=16 over T=512 (the ~350M workload):
    x averaged 8 times, each momentum and v 32 times."""
    cfg = P.make_config(W.WORKLOADS["decoder_350m"]["opt"])
    counts = np.zeros(4, int)
    for t in range(512):
        m = P.mtdao_due_mask(cfg, t)
        counts += [(m >> s) & 1 for s in range(4)]
    assert counts.tolist() == [8, 32, 32, 32]


@pytest.mark.parametrize("bad", [
    {"beta1": [1.0, 0.9]}, {"beta1": [-0.1, 0.9]}, {"omega": [0.6, 0.6]}, {"omega": [1.2, 0.0]},
    {"beta2": 1.0}, {"eps": 0.0}, {"period_x": -1}, {"period_u": [4, -2]},
    {"clip_mode": "elementwise"}, {"n_mom": 5, "beta1": [0.9] * 5, "omega": [0.1] * 5,
                                   "period_u": [1] * 5},
    {"base": "adopt", "bias_correction": True}, {"base": "adopt", "clip_mode": "global_norm",
                                                 "bias_correction": False},
    {"clip_mode": "global_norm", "clip_rho": 0.0}, {"beta1": [float("nan"), 0.9]},
    {"adopt_prev_v": True},
])
def test_invalid_configurations_are_rejected(P, bad):
    opt = _opt()
    opt.update(bad)
    try:
        cfg = P.make_config(opt)
    except (IndexError, KeyError):
        return                                   # not even representable in the C struct
    with pytest.raises(P.MTDAOError) as e:
        P.mtdao_config_validate(cfg, 4)
    assert e.value.code == P.ERR_INVALID
    assert P.mtdao_last_error(None)


def test_valid_configurations(P):
    for name, w in W.WORKLOADS.items():
        P.mtdao_config_validate(P.make_config(w["opt"]), w["M"])
    for base in (0, 1, 2):
        for n in (1, 2, 3, 4):
            P.mtdao_config_validate(P.mtdao_config_default(base, n), 8)
    with pytest.raises(P.MTDAOError):
        P.mtdao_config_validate(P.make_config(_opt()), 0)
    with pytest.raises(P.MTDAOError):
        P.mtdao_config_validate(P.make_config(_opt()), P.MAX_REPLICAS + 1)


def test_null_handle_is_safe(P):
    P.lib.mtdao_destroy(None)
    assert P.lib.mtdao_get_step(None) == -1
    assert P.lib.mtdao_sync(None, 1) == P.ERR_INVALID


@pytest.mark.parametrize("base,betas,beta2,kx", [
    ("adam", (0.95,), 0.99, 32), ("adopt", (0.95,), 0.9999, 32), ("adam", (0.999,), 0.999, 32),
    ("adopt", (0.999,), 0.9999, 32), ("adam", (0.9, 0.999, 0.5), 0.999, 16),
    ("sgdm", (0.99, 0.0), 0.999, 8), ("adopt", (0.9, 0.99), 0.9999, 0), ("adam", (0.9999,), 0.9, 1000),
])
def test_half_life_helpers_match_the_oracle(P, base, betas, beta2, kx):
    """mtdao_half_life / mtdao_config_half_life_periods / mtdao_comm_reduction
    against the oracle's own versions (which the pin suite ties to the
    periods printed in the wall-clock appendix and to the sync count)."""
    from oracle.oracle import comm_reduction, half_life, half_life_periods
    for b in (*betas, beta2):
        assert P.mtdao_half_life(b) == pytest.approx(half_life(b), rel=1e-15)
    opt = _opt(base, betas, beta2=beta2, bias_correction=(base == "adam"))
    cfg = P.mtdao_config_half_life_periods(P.make_config(opt), kx)
    ref = half_life_periods(opt, kx)
    assert cfg.period_x == ref["period_x"] == kx
    assert [cfg.period_u[j] for j in range(len(betas))] == ref["period_u"]
    if base != "sgdm":
        assert cfg.period_v == ref["period_v"]
    P.mtdao_config_validate(cfg, 4)
    assert P.mtdao_comm_reduction(cfg) == pytest.approx(comm_reduction(ref), rel=1e-15)


def test_half_life_helpers_reject_bad_arguments(P):
    for beta in (1.0, -0.1, float("nan"), 2.0):
        with pytest.raises(P.MTDAOError) as e:
            P.mtdao_half_life(beta)
        assert e.value.code == P.ERR_INVALID
    cfg = P.make_config(_opt())
    before = (cfg.period_x, cfg.period_u[0], cfg.period_v)
    with pytest.raises(P.MTDAOError):
        P.mtdao_config_half_life_periods(cfg, -1)
    cfg.beta2 = 1.0
    with pytest.raises(P.MTDAOError):
        P.mtdao_config_half_life_periods(cfg, 32)
    assert (cfg.period_x, cfg.period_u[0], cfg.period_v) == before      # unchanged on error
    cfg = P.make_config(_opt(period_x=0, period_u=[0, 0], period_v=0))
    assert P.mtdao_comm_reduction(cfg) == float("inf")
    cfg.period_v = -3
    with pytest.raises(P.MTDAOError):
        P.mtdao_comm_reduction(cfg)


def test_binding_gradient_dtype_code(P):
    """The binding derives the library's dtype code from the gradient
    tensor and refuses an explicit code that contradicts it (the kernel
    would read the buffer as the other type)."""
    import torch
    code = P.MTDAO._grad_code
    assert code(torch.zeros(3), None) == P.F32
    assert code(torch.zeros(3, dtype=torch.bfloat16), None) == P.BF16
    assert code(torch.zeros(3, dtype=torch.bfloat16), P.BF16) == P.BF16
    assert code(0x1000, None) == P.F32              # a raw pointer: as given, F32 by default
    assert code(0x1000, P.BF16) == P.BF16
    with pytest.raises(ValueError):
        code(torch.zeros(3), P.BF16)
    with pytest.raises(ValueError):
        code(torch.zeros(3, dtype=torch.bfloat16), P.F32)


def test_static_norm_checks_arguments_before_touching_a_device(P):
    """mtdao_grad_sqnorm_static rejects NULL, misaligned or out-of-range
    arguments before it makes any CUDA call (the pointers below are never
    dereferenced), with the code the header states."""
    g, out = 0x10000, 0x20000          # 16-byte aligned stand-ins, never read
    cases = [((0, P.F32, 2, 256, out), P.ERR_INVALID),
             ((g, P.F32, 2, 256, 0), P.ERR_INVALID),
             ((g + 8, P.F32, 2, 256, out), P.ERR_ALIGN),
             ((g, P.F32, 2, 256, out + 4), P.ERR_ALIGN),
             ((g, 7, 2, 256, out), P.ERR_INVALID),
             ((g, P.F32, 0, 256, out), P.ERR_INVALID),
             ((g, P.F32, P.MAX_REPLICAS + 1, 256, out), P.ERR_INVALID),
             ((g, P.BF16, 2, 100, out), P.ERR_INVALID),
             ((g, P.BF16, 2, 0, out), P.ERR_INVALID)]
    for args, code in cases:
        with pytest.raises(P.MTDAOError) as e:
            P.mtdao_grad_sqnorm_static(*args, 0)
        assert e.value.code == code, (args, e.value)
        assert P.mtdao_last_error(None)
